// Decode read: one query per (b, h) against a cache of T keys and values, the
// read of Sec. 2.3 (Eq. "fem-free-energy-main", softmax prior of App. C) for a
// query that sees every cached key -- the last row of a causal read whose
// query was appended at position T - 1:
//
//   s_i = q . k_i / sqrt(d),   o_j = (1/beta_j) log sum_i softmax(s)_i exp(beta_j v_ij),
//   lse = LSE_i s_i,   beta_j = 0 meaning the prior mean.
//
// HBM-bound (K and V read once).  A CTA takes kDecChunk keys of one (b, h):
// K by TMA in the 128-byte-swizzled layout (so the threads that each take one
// key's half row read shared memory without bank conflicts), V by a bulk
// copy; small CTAs keep many copies in flight per SM.  Per chunk, with
// m = max s_i and P_i = exp(s_i - m):
//   L   = sum_i P_i
//   c_j = max_i v_ij
//   A_j = sum_i P_i exp(beta_j (v_ij - c_j))
//   W_j = sum_i P_i expm1(beta_j (v_ij - c_j)) / beta_j      (v_ij - c_j at beta 0)
// A second kernel combines a head's chunk partials (in kDecMergeGroups groups,
// then the groups) by bringing both sides to the common maxima m*, c_j*:
// factor exp(m - m*) on every term,
// r = exp(beta (c - c*)) on A, and W <- r W + expm1(beta (c - c*))/beta L
// (the joint rescale of two running shifts).  The read is
//   o = c + log1p(beta W / L) / beta   when beta W / L > -1/2,
//   o = c + log(A / L) / beta          otherwise,   o = c + W / L at beta = 0.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

constexpr int kDecChunk = kDecodeKeysPerCta;  // keys per CTA: K and V rows take 2 x 64 x d x 2 bytes of shared memory
constexpr int kDecThreads = 2 * kDecChunk;  // two threads per key for the scores

template <int D>
struct DecPart {
  static constexpr int kFloats = 2 + 3 * D;  // m, L, c[D], A[D], W[D]
};

// e = exp(b x) and em1b = expm1(b x) / b for x <= 0 (em1b = x at b = 0): the
// Taylor series of expm1(y)/y for |y| < 1/2 (truncation below 4e-6
// relative), (e - 1) / b beyond.
__device__ __forceinline__ void dec_exp_pair(float b, float inv_b, float x, float &e, float &em1b) {
  const float y = b * x;
  e = ex2_approx(y * kLog2e);
  if (fabsf(y) < 0.5f) {
    float poly = fmaf(y, 1.f / 720.f, 1.f / 120.f);
    poly = fmaf(y, poly, 1.f / 24.f);
    poly = fmaf(y, poly, 1.f / 6.f);
    poly = fmaf(y, poly, 0.5f);
    poly = fmaf(y, poly, 1.f);
    em1b = x * poly;
  } else {
    em1b = (e - 1.f) * inv_b;
  }
}

// (m, L, c, A, W) <- the combination of itself and (mc, Lc, cc, Ac, Wc), both
// brought to the common maxima max(m, mc), max(c, cc) (one channel; m and L
// shared by the channels): the side with the smaller maximum takes the
// factor exp(m - m*), the side with the smaller shift r = exp(b (c - c*)) on
// A and W <- r W + expm1(b (c - c*))/b L.
__device__ __forceinline__ void dec_fold(float b, float inv_b, float &m, float mc, float &L, float Lc, float &c,
                                         float cc, float &A, float Ac, float &W, float Wc) {
  const float dm = mc - m;
  const float em = ex2_approx(-fabsf(dm) * kLog2e);
  const float fr = dm > 0.f ? em : 1.f, fc = dm > 0.f ? 1.f : em;
  const float dc = cc - c;
  float r, er;
  dec_exp_pair(b, inv_b, -fabsf(dc), r, er);
  const float rr = dc > 0.f ? r : 1.f, rc = dc > 0.f ? 1.f : r;
  const float err = dc > 0.f ? er : 0.f, erc = dc > 0.f ? 0.f : er;
  W = fr * fmaf(rr, W, err * L) + fc * fmaf(rc, Wc, erc * Lc);
  A = fr * rr * A + fc * rc * Ac;
  L = fr * L + fc * Lc;
  m = fmaxf(m, mc);
  c = fmaxf(c, cc);
}

// Folds the partials k0 .. k1-1 of a head (layout DecPart) for channel j into
// r = {m, L, c_j, A_j, W_j}, loading up to eight partials at once ahead of
// their folds (one round of memory latency per eight).
template <int D>
__device__ __forceinline__ void dec_fold_range(const float *pb, int k0, int k1, int j, float b, float inv_b,
                                               float (&r)[5]) {
  constexpr int F = DecPart<D>::kFloats, kAhead = 8;
  bool first = true;
  float m = 0.f, L = 0.f, c = 0.f, A = 0.f, W = 0.f;
  for (int k = k0; k < k1; k += kAhead) {
    float mc[kAhead], Lc[kAhead], cc[kAhead], Ac[kAhead], Wc[kAhead];
#pragma unroll
    for (int u = 0; u < kAhead; ++u) {
      if (k + u < k1) {
        const float *pc = pb + static_cast<size_t>(k + u) * F;
        mc[u] = pc[0];
        Lc[u] = pc[1];
        cc[u] = pc[2 + j];
        Ac[u] = pc[2 + D + j];
        Wc[u] = pc[2 + 2 * D + j];
      }
    }
#pragma unroll
    for (int u = 0; u < kAhead; ++u) {
      if (k + u < k1) {
        if (first) {
          m = mc[u], L = Lc[u], c = cc[u], A = Ac[u], W = Wc[u];
          first = false;
        } else {
          dec_fold(b, inv_b, m, mc[u], L, Lc[u], c, cc[u], A, Ac[u], W, Wc[u]);
        }
      }
    }
  }
  r[0] = m;
  r[1] = L;
  r[2] = c;
  r[3] = A;
  r[4] = W;
}

// Per (key, channel pair) the kernel needs exp(beta x) and expm1(beta x)/beta
// with x = v - c <= 0.  For beta >= kDecFastBeta the latter is (e - 1)/beta
// from the same e: its absolute error (that of e, about 2^-22) divided by beta
// stays below 2^-16.  Smaller beta (and beta = 0) take the Taylor series.
constexpr float kDecFastBeta = 1.f / 64.f;

template <int D>
__global__ void __launch_bounds__(kDecThreads) decode_chunk_kernel(const __grid_constant__ CUtensorMap tmap_k,
                                                            const __nv_bfloat16 *__restrict__ q,
                                                            const __nv_bfloat16 *__restrict__ v,
                                                            const float *__restrict__ beta, int H, int T,
                                                            float *__restrict__ part, int *__restrict__ count,
                                                            unsigned *__restrict__ err) {
  // K rows by TMA as D/64 boxes of [kDecChunk rows x 64 channels] with the
  // 128-byte swizzle (1024-byte aligned), then V rows [kDecChunk][D] by a bulk copy
  extern __shared__ uint8_t dec_raw[];
  uint8_t *dec_smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(dec_raw) + 1023) & ~uintptr_t(1023));
  constexpr uint32_t kBoxBytes = kDecChunk * 128, kKBytes = (D / 64) * kBoxBytes;
  __shared__ __align__(8) uint64_t s_bar;
  __shared__ float s_dot[2][kDecChunk];
  __shared__ __align__(16) float s_p[kDecChunk];
  constexpr int kWarps = kDecThreads / 32;
  __shared__ float s_red[kWarps];
  constexpr int kPairs = D / 2, kGroups = kDecThreads / kPairs, kKeysPer = kDecChunk / kGroups;
  __shared__ float2 s_c[kGroups][kPairs], s_A[kGroups][kPairs], s_W[kGroups][kPairs];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = blockIdx.x, bh = blockIdx.y, h = bh % H;
  const int key0 = g * kDecChunk, rows = min(kDecChunk, T - key0);
  const uint32_t sk = smem_u32(dec_smem), bar = smem_u32(&s_bar);
  if (tid == 0) {
    if (g == 0) count[bh] = 0;  // the merge kernel's arrival counter of this head
    mbar_init(bar, 1);
    fence_mbar_init();
    mbar_arrive_expect_tx(bar, kKBytes + static_cast<uint32_t>(rows * D * 2));
    for (int bx = 0; bx < D / 64; ++bx) tma_load_3d(sk + bx * kBoxBytes, &tmap_k, bar, bx * 64, key0, bh);
    bulk_load(sk + kKBytes, v + (static_cast<size_t>(bh) * T + key0) * D, static_cast<uint32_t>(rows * D * 2), bar);
  }
  // scores: thread (hf, i) takes key i = tid % kDecChunk and channels
  // [hf D/2, hf D/2 + D/2); its half of q stays in registers as pairs
  const int ki = tid % kDecChunk, hf = tid / kDecChunk;
  constexpr int kChunks = D / 16;  // 16-byte chunks (8 channels) per half row
  float2 qr[D / 4];
  {
    const __nv_bfloat162 *q2 = reinterpret_cast<const __nv_bfloat162 *>(q + static_cast<size_t>(bh) * D + hf * (D / 2));
#pragma unroll
    for (int u = 0; u < D / 4; ++u) qr[u] = __bfloat1622float2(q2[u]);
  }
  const int pj = tid % kPairs, kg = tid / kPairs;
  const float2 b2 = *reinterpret_cast<const float2 *>(beta + h * D + 2 * pj);
  __syncthreads();
  if (!mbar_wait(bar, 0, err, kErrWaitTma)) return;
  {
    float2 dot2 = make_float2(0.f, 0.f);
#pragma unroll
    for (int u = 0; u < kChunks; ++u) {
      const int gc = hf * kChunks + u;  // logical 16-byte chunk of the row
      const uint4 raw = *reinterpret_cast<const uint4 *>(dec_smem + (gc >> 3) * kBoxBytes + ki * 128 +
                                                         (((gc & 7) ^ (ki & 7)) << 4));
      const __nv_bfloat162 *kk = reinterpret_cast<const __nv_bfloat162 *>(&raw);
#pragma unroll
      for (int e = 0; e < 4; ++e) dot2 = __ffma2_rn(__bfloat1622float2(kk[e]), qr[4 * u + e], dot2);
    }
    s_dot[hf][ki] = dot2.x + dot2.y;
  }
  __syncthreads();
  // chunk maximum m over the valid keys, then P_i = exp(s_i - m) and L = sum P_i
  const float scale = rsqrtf(static_cast<float>(D));
  const float sv = tid < rows ? (s_dot[0][tid] + s_dot[1][tid]) * scale : -INFINITY;
  float mx = sv;
#pragma unroll
  for (int off = 16; off; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  if (lane == 0) s_red[warp] = mx;
  __syncthreads();
  float m = s_red[0];
#pragma unroll
  for (int w = 1; w < kWarps; ++w) m = fmaxf(m, s_red[w]);
  const float p = tid < rows ? expf(sv - m) : 0.f;
  float ls = p;
#pragma unroll
  for (int off = 16; off; off >>= 1) ls += __shfl_xor_sync(0xffffffffu, ls, off);
  __syncthreads();  // every thread has read s_red
  if (tid < kDecChunk) s_p[tid] = p;
  if (lane == 0) s_red[warp] = ls;
  // per channel pair over the keys of this thread's group: the chunk maximum
  // c_j first (exact in bf16), then A and W, each value pair one bf16x2 load
  const int i0 = kg * kKeysPer;
  const __nv_bfloat162 *sV2 = reinterpret_cast<const __nv_bfloat162 *>(dec_smem + kKBytes) + pj;
  __nv_bfloat162 cm = __floats2bfloat162_rn(-INFINITY, -INFINITY);
#pragma unroll 8
  for (int i = i0; i < i0 + kKeysPer; ++i)
    if (i < rows) cm = __hmax2(cm, sV2[i * kPairs]);
  s_c[kg][pj] = __bfloat1622float2(cm);
  __syncthreads();
  float L = 0.f;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) L += s_red[w];
  float2 c2 = s_c[0][pj];
#pragma unroll
  for (int q2 = 1; q2 < kGroups; ++q2) c2 = make_float2(fmaxf(c2.x, s_c[q2][pj].x), fmaxf(c2.y, s_c[q2][pj].y));
  const float2 negc2 = make_float2(-c2.x, -c2.y);
  const float2 bl2 = make_float2(b2.x * kLog2e, b2.y * kLog2e);
  const int i1 = min(rows, i0 + kKeysPer);
  float2 A = make_float2(0.f, 0.f), W = make_float2(0.f, 0.f);
  if (b2.x >= kDecFastBeta && b2.y >= kDecFastBeta) {
    // W = sum_i P_i (e_i - 1) / beta, the division once at the end
#pragma unroll 8
    for (int i = i0; i < i1; ++i) {
      const float2 x = __fadd2_rn(__bfloat1622float2(sV2[i * kPairs]), negc2);  // <= 0
      const float2 t = __fmul2_rn(bl2, x);
      const float2 e = make_float2(ex2_approx(t.x), ex2_approx(t.y));
      const float2 P = make_float2(s_p[i], s_p[i]);
      A = __ffma2_rn(P, e, A);
      W = __ffma2_rn(P, __fadd2_rn(e, make_float2(-1.f, -1.f)), W);
    }
    W = __fmul2_rn(W, make_float2(1.f / b2.x, 1.f / b2.y));
  } else {
    const float2 inv_b = make_float2(b2.x > 0.f ? 1.f / b2.x : 0.f, b2.y > 0.f ? 1.f / b2.y : 0.f);
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
  }
  s_A[kg][pj] = A;
  s_W[kg][pj] = W;
  __syncthreads();
  float *pp = part + (static_cast<size_t>(bh) * gridDim.x + g) * DecPart<D>::kFloats;
  if (tid == 0) {
    pp[0] = m;
    pp[1] = L;
  }
  if (kg == 0) {
#pragma unroll
    for (int q2 = 1; q2 < kGroups; ++q2) {
      A = __fadd2_rn(A, s_A[q2][pj]);
      W = __fadd2_rn(W, s_W[q2][pj]);
    }
    *reinterpret_cast<float2 *>(pp + 2 + 2 * pj) = c2;
    *reinterpret_cast<float2 *>(pp + 2 + D + 2 * pj) = A;
    *reinterpret_cast<float2 *>(pp + 2 + 2 * D + 2 * pj) = W;
  }
}

// Partials of a head combined by kDecMergeGroups blocks of D threads: block
// (grp, bh) folds its share of the chunk partials for channel j = thread in
// order into a group partial; the last of a head's blocks to finish (an
// arrival counter, which the chunk kernel's first block of the head zeroes)
// folds the group partials and writes the read.
constexpr int kDecMergeGroups = 8;

template <int D>
__global__ void __launch_bounds__(D) decode_merge_kernel(const float *__restrict__ part, int n_parts,
                                                         float *__restrict__ gpart, int *__restrict__ count,
                                                         const float *__restrict__ beta, int H,
                                                         float *__restrict__ out, float *__restrict__ lse) {
  constexpr int G = kDecMergeGroups, F = DecPart<D>::kFloats;
  const int grp = blockIdx.x, bh = blockIdx.y, h = bh % H, j = threadIdx.x;
  const float b = beta[h * D + j], inv_b = b > 0.f ? 1.f / b : 0.f;
  const int n_groups = min(G, n_parts);
  if (grp >= n_groups) return;
  // launched as a programmatic dependent of the chunk kernel: its partials
  // are complete and visible once this wait returns
  asm volatile("griddepcontrol.wait;" ::: "memory");
  float r[5];
  dec_fold_range<D>(part + static_cast<size_t>(bh) * n_parts * F, grp * n_parts / n_groups,
                    (grp + 1) * n_parts / n_groups, j, b, inv_b, r);
  float *po = gpart + (static_cast<size_t>(bh) * G + grp) * F;
  if (j == 0) {
    po[0] = r[0];
    po[1] = r[1];
  }
  po[2 + j] = r[2];
  po[2 + D + j] = r[3];
  po[2 + 2 * D + j] = r[4];
  __shared__ int s_last;
  __threadfence();
  __syncthreads();
  if (j == 0) s_last = atomicAdd(&count[bh], 1) == n_groups - 1;
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  dec_fold_range<D>(gpart + static_cast<size_t>(bh) * G * F, 0, n_groups, j, b, inv_b, r);
  const float m = r[0], L = r[1], c = r[2], A = r[3], W = r[4];
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

// Workspace: chunk partials [BH][n_parts], group partials [BH][kDecMergeGroups]
// (DecPart floats each), then one arrival counter per head.
static size_t dec_count_offset(int BH, int T, int d) {
  const size_t n_parts = (static_cast<size_t>(T) + kDecChunk - 1) / kDecChunk;
  return static_cast<size_t>(BH) * (n_parts + kDecMergeGroups) * (2 + 3 * static_cast<size_t>(d)) * sizeof(float);
}

size_t decode_workspace_bytes(int BH, int T, int d, int) {
  return dec_count_offset(BH, T, d) + static_cast<size_t>(BH) * sizeof(int);
}

template <int D>
static cudaError_t launch_decode_d(const CUtensorMap &tk, const __nv_bfloat16 *q, const __nv_bfloat16 *v,
                                   const float *beta, float *out, float *lse, int BH, int H, int T, float *part,
                                   unsigned *err, cudaStream_t stream) {
  const int n_parts = (T + kDecChunk - 1) / kDecChunk;
  const size_t smem = 1024 + 2 * static_cast<size_t>(kDecChunk) * D * 2;
  cudaError_t e =
      cudaFuncSetAttribute(decode_chunk_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  float *gpart = part + static_cast<size_t>(BH) * n_parts * DecPart<D>::kFloats;
  int *count = reinterpret_cast<int *>(reinterpret_cast<uint8_t *>(part) + dec_count_offset(BH, T, D));
  decode_chunk_kernel<D><<<dim3(n_parts, BH), kDecThreads, smem, stream>>>(tk, q, v, beta, H, T, part, count, err);
  // the merge launches while the chunk kernel drains and waits for it on the device
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kDecMergeGroups, BH);
  cfg.blockDim = dim3(D);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, decode_merge_kernel<D>, static_cast<const float *>(part), n_parts, gpart, count, beta,
                         H, out, lse);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t launch_decode(const CUtensorMap &tk, const void *q, const void *v, const float *beta, float *out,
                          float *lse, int BH, int H, int T, int d, float *part, unsigned *err, cudaStream_t stream) {
  const __nv_bfloat16 *qb = static_cast<const __nv_bfloat16 *>(q), *vb = static_cast<const __nv_bfloat16 *>(v);
  if (d == 64) return launch_decode_d<64>(tk, qb, vb, beta, out, lse, BH, H, T, part, err, stream);
  if (d == 128) return launch_decode_d<128>(tk, qb, vb, beta, out, lse, BH, H, T, part, err, stream);
  return cudaErrorInvalidValue;
}

}  // namespace fem
