// Decode read: one query per (b, h) against a cache of T keys and values, the
// read of Sec. 2.3 (Eq. "fem-free-energy-main", softmax prior of App. C) for a
// query that sees every cached key -- the last row of a causal read whose
// query was appended at position T - 1:
//
//   s_i = q . k_i / sqrt(d),   o_j = (1/beta_j) log sum_i softmax(s)_i exp(beta_j v_ij),
//   lse = LSE_i s_i,   beta_j = 0 meaning the prior mean.
//
// HBM-bound (K and V read once).  A CTA takes kDecChunk keys of one (b, h),
// brought to shared memory by bulk copies; small CTAs keep many copies in
// flight per SM (a CTA can also stream a longer range through a two-stage
// ring, which measured slower: its chunks' copies wait on its own compute).  Per chunk, with m = max s_i and P_i = exp(s_i - m):
//   L   = sum_i P_i
//   c_j = max_i v_ij
//   A_j = sum_i P_i exp(beta_j (v_ij - c_j))
//   W_j = sum_i P_i expm1(beta_j (v_ij - c_j)) / beta_j      (v_ij - c_j at beta 0)
// Chunks, and then the CTAs' ranges, are combined by bringing both sides to
// the common maxima m*, c_j*: factor exp(m - m*) on every term,
// r = exp(beta (c - c*)) on A, and W <- r W + expm1(beta (c - c*))/beta L
// (the joint rescale of two running shifts).  The read is
//   o = c + log1p(beta W / L) / beta   when beta W / L > -1/2,
//   o = c + log(A / L) / beta          otherwise,   o = c + W / L at beta = 0.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

constexpr int kDecChunk = 64;  // keys per chunk: K and V rows take 2 x 64 x d x 2 bytes per stage
constexpr int kDecMergeGroup = 16;  // chunk partials folded by one CTA of the first merge level

template <int D>
struct DecPart {
  static constexpr int kFloats = 2 + 3 * D;  // m, L, c[D], A[D], W[D]
};

__device__ __forceinline__ float dec_expm1_over_beta(float b, float x) {
  // expm1(b x) / b, continuous at b = 0
  return b != 0.f ? expm1f(b * x) / b : x;
}

// (m, L, c, A, W) <- the combination of itself and (mc, Lc, cc, Ac, Wc), both
// brought to the common maxima (one channel; m and L shared by the channels).
__device__ __forceinline__ void dec_fold(float b, float m, float mc, float L, float Lc, float &c, float cc, float &A,
                                         float Ac, float &W, float Wc) {
  const float mn = fmaxf(m, mc), cn = fmaxf(c, cc);
  const float fr = expf(m - mn), fc = expf(mc - mn);
  const float rr = expf(b * (c - cn)), rc = expf(b * (cc - cn));
  const float er = dec_expm1_over_beta(b, c - cn), ec = dec_expm1_over_beta(b, cc - cn);
  W = fr * fmaf(rr, W, er * L) + fc * fmaf(rc, Wc, ec * Lc);
  A = fr * rr * A + fc * rc * Ac;
  c = cn;
}

template <int D>
__device__ __forceinline__ void dec_issue(const __nv_bfloat16 *k, const __nv_bfloat16 *v, size_t row0, int rows,
                                          uint32_t dst, uint32_t bar) {
  const uint32_t bytes = static_cast<uint32_t>(rows * D * 2);
  mbar_arrive_expect_tx(bar, 2 * bytes);
  bulk_load(dst, k + row0 * D, bytes, bar);
  bulk_load(dst + kDecChunk * D * 2, v + row0 * D, bytes, bar);
}

template <int D>
__global__ void __launch_bounds__(128) decode_chunk_kernel(const __nv_bfloat16 *__restrict__ q,
                                                            const __nv_bfloat16 *__restrict__ k,
                                                            const __nv_bfloat16 *__restrict__ v,
                                                            const float *__restrict__ beta, int H, int T,
                                                            int keys_per_cta, float *__restrict__ part,
                                                            unsigned *__restrict__ err) {
  extern __shared__ __align__(16) uint8_t dec_smem[];  // 2 stages of K rows [C][D] then V rows [C][D], bf16
  constexpr int kStage = 2 * kDecChunk * D * 2;
  __shared__ __align__(8) uint64_t s_bar[2];
  __shared__ float s_p[128];  // one entry per thread (kDecChunk <= 128)
  __shared__ float s_q[D];
  __shared__ float s_red[4];
  constexpr int kPairs = D / 2, kGroups = 128 / kPairs, kKeysPer = kDecChunk / kGroups;
  __shared__ float2 s_c[kGroups][kPairs], s_A[kGroups][kPairs], s_W[kGroups][kPairs];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = blockIdx.x, bh = blockIdx.y, h = bh % H;
  const int key0 = g * keys_per_cta, key1 = min(T, key0 + keys_per_cta);
  const int n_ch = (key1 - key0 + kDecChunk - 1) / kDecChunk;
  const size_t base_row = static_cast<size_t>(bh) * T;
  if (tid == 0) {
    mbar_init(smem_u32(&s_bar[0]), 1);
    mbar_init(smem_u32(&s_bar[1]), 1);
    fence_mbar_init();
    for (int c = 0; c < 2 && c < n_ch; ++c)
      dec_issue<D>(k, v, base_row + key0 + c * kDecChunk, min(kDecChunk, key1 - key0 - c * kDecChunk),
                   smem_u32(dec_smem) + c * kStage, smem_u32(&s_bar[c]));
  }
  for (int j = tid; j < D; j += 128) s_q[j] = __bfloat162float(q[static_cast<size_t>(bh) * D + j]);
  // running state: m, L in every thread; c, A, W of pair pj in the group-0 threads
  const int pj = tid % kPairs, kg = tid / kPairs;
  const float2 b2 = *reinterpret_cast<const float2 *>(beta + h * D + 2 * pj);
  const float2 bl2 = make_float2(b2.x * kLog2e, b2.y * kLog2e);
  const float2 inv_b = make_float2(b2.x > 0.f ? 1.f / b2.x : 0.f, b2.y > 0.f ? 1.f / b2.y : 0.f);
  float m_run = -INFINITY, L_run = 0.f;
  float2 c_run = make_float2(0.f, 0.f), A_run = make_float2(0.f, 0.f), W_run = make_float2(0.f, 0.f);
  constexpr int kPer = D / 32;
  const float scale = rsqrtf(static_cast<float>(D));
  __syncthreads();

  for (int ch = 0; ch < n_ch; ++ch) {
    const int st = ch & 1, rows = min(kDecChunk, key1 - key0 - ch * kDecChunk);
    if (!mbar_wait(smem_u32(&s_bar[st]), (ch >> 1) & 1, err, kErrWaitTma)) return;
    const __nv_bfloat16 *sK = reinterpret_cast<const __nv_bfloat16 *>(dec_smem + st * kStage);
    const __nv_bfloat16 *sV = sK + kDecChunk * D;
    // scores: warp w takes keys w, w + 4, ...; lane l the D/32 channels from D/32 l
    for (int i = warp; i < rows; i += 4) {
      const __nv_bfloat16 *kr = sK + i * D + lane * kPer;
      float dot = 0.f;
#pragma unroll
      for (int u = 0; u < kPer; ++u) dot = fmaf(s_q[lane * kPer + u], __bfloat162float(kr[u]), dot);
#pragma unroll
      for (int off = 16; off; off >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, off);
      if (lane == 0) s_p[i] = dot * scale;
    }
    __syncthreads();
    // chunk maximum m, then P_i = exp(s_i - m) and L = sum P_i
    const float sv = tid < rows ? s_p[tid] : -INFINITY;
    float mx = sv;
#pragma unroll
    for (int off = 16; off; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    if (lane == 0) s_red[warp] = mx;
    __syncthreads();
    const float m = fmaxf(fmaxf(s_red[0], s_red[1]), fmaxf(s_red[2], s_red[3]));
    const float p = tid < rows ? expf(sv - m) : 0.f;
    float ls = p;
#pragma unroll
    for (int off = 16; off; off >>= 1) ls += __shfl_xor_sync(0xffffffffu, ls, off);
    __syncthreads();  // every thread has read s_red and its s_p entry
    s_p[tid] = p;
    if (lane == 0) s_red[warp] = ls;
    // per channel pair over the keys of this thread's group: the chunk maximum
    // c_j first (exact in bf16), then A and W, each value pair one bf16x2 load
    const int i0 = kg * kKeysPer, i1 = min(rows, i0 + kKeysPer);
    const __nv_bfloat162 *sV2 = reinterpret_cast<const __nv_bfloat162 *>(sV) + pj;
    __nv_bfloat162 cm = __floats2bfloat162_rn(-INFINITY, -INFINITY);
    for (int i = i0; i < i1; ++i) cm = __hmax2(cm, sV2[i * kPairs]);
    s_c[kg][pj] = __bfloat1622float2(cm);
    __syncthreads();
    const float L = (s_red[0] + s_red[1]) + (s_red[2] + s_red[3]);
    float2 c2 = s_c[0][pj];
#pragma unroll
    for (int q2 = 1; q2 < kGroups; ++q2) c2 = make_float2(fmaxf(c2.x, s_c[q2][pj].x), fmaxf(c2.y, s_c[q2][pj].y));
    const float2 negc2 = make_float2(-c2.x, -c2.y);
    float2 A = make_float2(0.f, 0.f), W = make_float2(0.f, 0.f);
    for (int i = i0; i < i1; ++i) {
      const float2 x = __fadd2_rn(__bfloat1622float2(sV2[i * kPairs]), negc2);  // <= 0
      const float2 P = make_float2(s_p[i], s_p[i]);
      const float2 t = __fmul2_rn(bl2, x);
      const float2 e = make_float2(ex2_approx(t.x), ex2_approx(t.y));
      // expm1(b x)/b: a Taylor series of expm1(y)/y for |y| < 1/2 (truncation
      // below 4e-6 relative), (e^y - 1)/b beyond; x itself at b = 0
      const float2 y = __fmul2_rn(b2, x);
      float2 poly = __ffma2_rn(y, make_float2(1.f / 720.f, 1.f / 720.f), make_float2(1.f / 120.f, 1.f / 120.f));
      poly = __ffma2_rn(y, poly, make_float2(1.f / 24.f, 1.f / 24.f));
      poly = __ffma2_rn(y, poly, make_float2(1.f / 6.f, 1.f / 6.f));
      poly = __ffma2_rn(y, poly, make_float2(0.5f, 0.5f));
      poly = __ffma2_rn(y, poly, make_float2(1.f, 1.f));
      const float2 lin = __fmul2_rn(x, poly);
      const float2 big = __fmul2_rn(__fadd2_rn(e, make_float2(-1.f, -1.f)), inv_b);
      const float2 em1 = make_float2(fabsf(y.x) < 0.5f ? lin.x : big.x, fabsf(y.y) < 0.5f ? lin.y : big.y);
      A = __ffma2_rn(P, e, A);
      W = __ffma2_rn(P, em1, W);
    }
    s_A[kg][pj] = A;
    s_W[kg][pj] = W;
    __syncthreads();  // the stage is read: refill it two chunks ahead
    if (tid == 0 && ch + 2 < n_ch)
      dec_issue<D>(k, v, base_row + key0 + (ch + 2) * kDecChunk, min(kDecChunk, key1 - key0 - (ch + 2) * kDecChunk),
                   smem_u32(dec_smem) + st * kStage, smem_u32(&s_bar[st]));
    if (kg == 0) {
#pragma unroll
      for (int q2 = 1; q2 < kGroups; ++q2) {
        A = __fadd2_rn(A, s_A[q2][pj]);
        W = __fadd2_rn(W, s_W[q2][pj]);
      }
      if (ch == 0) {
        c_run = c2;
        A_run = A;
        W_run = W;
      } else {
        dec_fold(b2.x, m_run, m, L_run, L, c_run.x, c2.x, A_run.x, A.x, W_run.x, W.x);
        dec_fold(b2.y, m_run, m, L_run, L, c_run.y, c2.y, A_run.y, A.y, W_run.y, W.y);
      }
    }
    if (ch == 0) {
      m_run = m;
      L_run = L;
    } else {
      const float mn = fmaxf(m_run, m);
      L_run = L_run * expf(m_run - mn) + L * expf(m - mn);
      m_run = mn;
    }
    __syncthreads();  // s_red, s_c, s_A, s_W are reused by the next chunk
  }
  float *pp = part + (static_cast<size_t>(bh) * gridDim.x + g) * DecPart<D>::kFloats;
  if (tid == 0) {
    pp[0] = m_run;
    pp[1] = L_run;
  }
  if (kg == 0) {
    *reinterpret_cast<float2 *>(pp + 2 + 2 * pj) = c_run;
    *reinterpret_cast<float2 *>(pp + 2 + D + 2 * pj) = A_run;
    *reinterpret_cast<float2 *>(pp + 2 + 2 * D + 2 * pj) = W_run;
  }
}

// Partials of a head combined in order, in two levels: CTA (grp, bh) of the
// first level folds partials grp*G .. grp*G + G - 1 into one partial; the
// second level folds those and writes the read.
template <int D>
__global__ void __launch_bounds__(D) decode_merge_kernel(const float *__restrict__ part, int n_parts,
                                                          const float *__restrict__ beta, int H,
                                                          float *__restrict__ part_out, float *__restrict__ out,
                                                          float *__restrict__ lse) {
  const int grp = blockIdx.x, bh = blockIdx.y, h = bh % H, j = threadIdx.x;
  const int p0 = grp * kDecMergeGroup, p1 = out ? n_parts : min(n_parts, p0 + kDecMergeGroup);
  const float *pb = part + static_cast<size_t>(bh) * n_parts * DecPart<D>::kFloats;
  const float b = beta[h * D + j];
  const float *pf = pb + static_cast<size_t>(out ? 0 : p0) * DecPart<D>::kFloats;
  float m = pf[0], L = pf[1], c = pf[2 + j], A = pf[2 + D + j], W = pf[2 + 2 * D + j];
  for (int k = (out ? 0 : p0) + 1; k < p1; ++k) {
    const float *pc = pb + static_cast<size_t>(k) * DecPart<D>::kFloats;
    const float mc = pc[0], Lc = pc[1];
    dec_fold(b, m, mc, L, Lc, c, pc[2 + j], A, pc[2 + D + j], W, pc[2 + 2 * D + j]);
    const float mn = fmaxf(m, mc);
    L = L * expf(m - mn) + Lc * expf(mc - mn);
    m = mn;
  }
  if (!out) {
    float *po = part_out + (static_cast<size_t>(bh) * gridDim.x + grp) * DecPart<D>::kFloats;
    if (j == 0) {
      po[0] = m;
      po[1] = L;
    }
    po[2 + j] = c;
    po[2 + D + j] = A;
    po[2 + 2 * D + j] = W;
    return;
  }
  float o;
  if (b == 0.f) {
    o = c + W / L;
  } else {
    const float z = b * W / L;
    o = z > -0.5f ? c + log1pf(z) / b : c + logf(A / L) / b;
  }
  out[static_cast<size_t>(bh) * D + j] = o;
  if (lse && j == 0) lse[bh] = m + logf(L);
}

// Key range per CTA: one chunk.
static int dec_keys_per_cta(int, int, int) { return kDecChunk; }

size_t decode_workspace_bytes(int BH, int T, int d, int num_sms) {
  const int per = dec_keys_per_cta(BH, T, num_sms);
  const size_t n_parts = (static_cast<size_t>(T) + per - 1) / per;
  const size_t n_groups = (n_parts + kDecMergeGroup - 1) / kDecMergeGroup;
  return static_cast<size_t>(BH) * (n_parts + n_groups) * (2 + 3 * static_cast<size_t>(d)) * sizeof(float);
}

template <int D>
static cudaError_t launch_decode_d(const __nv_bfloat16 *q, const __nv_bfloat16 *k, const __nv_bfloat16 *v,
                                   const float *beta, float *out, float *lse, int BH, int H, int T, float *part,
                                   int num_sms, unsigned *err, cudaStream_t stream) {
  const int per = dec_keys_per_cta(BH, T, num_sms);
  const int n_parts = (T + per - 1) / per;
  const int n_groups = (n_parts + kDecMergeGroup - 1) / kDecMergeGroup;
  // one stage suffices when every CTA reads a single chunk
  const size_t smem = (per > kDecChunk ? 2 : 1) * 2 * static_cast<size_t>(kDecChunk) * D * 2;
  cudaError_t e =
      cudaFuncSetAttribute(decode_chunk_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  decode_chunk_kernel<D><<<dim3(n_parts, BH), 128, smem, stream>>>(q, k, v, beta, H, T, per, part, err);
  if (n_groups > 1) {
    float *part2 = part + static_cast<size_t>(BH) * n_parts * DecPart<D>::kFloats;
    decode_merge_kernel<D><<<dim3(n_groups, BH), D, 0, stream>>>(part, n_parts, beta, H, part2, nullptr, nullptr);
    decode_merge_kernel<D><<<dim3(1, BH), D, 0, stream>>>(part2, n_groups, beta, H, nullptr, out, lse);
  } else {
    decode_merge_kernel<D><<<dim3(1, BH), D, 0, stream>>>(part, n_parts, beta, H, nullptr, out, lse);
  }
  return cudaGetLastError();
}

cudaError_t launch_decode(const void *q, const void *k, const void *v, const float *beta, float *out, float *lse,
                          int BH, int H, int T, int d, float *part, int num_sms, unsigned *err, cudaStream_t stream) {
  const __nv_bfloat16 *qb = static_cast<const __nv_bfloat16 *>(q), *kb = static_cast<const __nv_bfloat16 *>(k),
                      *vb = static_cast<const __nv_bfloat16 *>(v);
  if (d == 64) return launch_decode_d<64>(qb, kb, vb, beta, out, lse, BH, H, T, part, num_sms, err, stream);
  if (d == 128) return launch_decode_d<128>(qb, kb, vb, beta, out, lse, BH, H, T, part, num_sms, err, stream);
  return cudaErrorInvalidValue;
}

}  // namespace fem
