// The FEM read on CUDA cores, exact to fp32 rounding: fp32 inputs of any head
// dimension up to 256, and bf16 inputs of head dimension 16 or 32 (too narrow
// for the tensor-core read's 64-channel tiles to pay; here every product and
// sum is fp32).
//
// One warp per output row t, four consecutive rows of one (b, h) per block;
// lane l owns channels l, l+32, ...  The block stages the keys' K and V rows
// in shared memory, a tile of fem_simt_tile(d) keys at a time (as fp32), so the
// walk below reads them with shared-memory latency.  For every key
// i in the support the warp forms s_{t,i} = q_t . k_i / sqrt(d) (lane-partial
// dot product, butterfly sum) and folds key i into
//   L   = sum_i P_i,                          P_i = exp(s_i - m)
//   A_j = sum_i P_i exp(beta_j (v_ij - c_j))
//   W_j = sum_i P_i expm1(beta_j (v_ij - c_j)) / beta_j   (v_ij - c_j at beta 0)
// with a running row maximum m and an exact running per-channel maximum c_j
// of the visible values (the per-channel stabilisation of App. E, per row).
// When m grows by dm, L, A and W scale by exp(-dm); when c_j grows to c',
// with r = exp(beta (c - c')), A <- r A and W <- r W + expm1(beta (c - c'))/beta L
// (the joint rescale of the two running shifts).  The read is then
//   o = c + log1p(beta W / L) / beta   when beta W / L > -1/2 (no cancellation),
//   o = c + log(A / L) / beta          otherwise,
//   o = c + W / L                      at beta = 0 (the prior mean),
// which is (1/beta) log sum_i p_t(i) exp(beta v_ij) (Sec. 2.3).
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

constexpr int kSimtMaxPerLane = 8;  // d <= 256

// rows up to which a row gets a block of its own (its keys split over the warps)
constexpr long long kSimtSplitRows = 2048;

// keys per staged tile: K and V of a tile take 32 KB at most (8 KB at d = 16)
inline __host__ __device__ int fem_simt_tile(int d) {
  const int kt = 4096 / d;
  return kt > 64 ? 64 : (kt < 8 ? 8 : kt);
}

__device__ __forceinline__ float expm1_over_beta(float b, float x) {
  // expm1(b x) / b, continuous at b = 0
  return b != 0.f ? expm1f(b * x) / b : x;
}

__device__ __forceinline__ float ld_in(const float *p) { return *p; }
__device__ __forceinline__ float ld_in(const __nv_bfloat16 *p) { return __bfloat162float(*p); }

// PER: channel slots per lane, d <= 32 PER (the unrolled per-slot code costs
// issue slots even where a slot is empty).  SPLIT (few rows): one row per
// block, each warp folding a quarter of every staged tile's keys from an empty
// state, the four states merged at the end (each scaled to the common row
// maximum, each channel's moved to the larger shift as when a key raises it),
// so that a row's dependent chain is a quarter as long.
template <typename In, int PER, bool SPLIT>
__global__ void __launch_bounds__(128) fem_simt_kernel(const In *__restrict__ q, const In *__restrict__ k,
                                                        const In *__restrict__ v, const float *__restrict__ beta,
                                                        float *__restrict__ out, float *__restrict__ lse, int H,
                                                        int T, int d, int causal) {
  extern __shared__ float simt_smem[];  // [tile][d] K, then [tile][d] V
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int bpr = SPLIT ? T : (T + 3) / 4;  // blocks per (b, h)
  const long long bh = blockIdx.x / bpr;
  const int t0 = static_cast<int>(blockIdx.x % bpr) * (SPLIT ? 1 : 4), t = SPLIT ? t0 : t0 + warp;
  const bool valid = t < T;
  const long long row = bh * T + t;
  const int h = static_cast<int>(bh % H);
  const int n = !valid ? 0 : (causal ? t + 1 : T);                // keys this row sees
  const int n_blk = SPLIT ? n : (causal ? min(T, t0 + 4) : T);    // keys any row of the block sees
  const int per = (d + 31) / 32;  // <= PER
  const int tile = fem_simt_tile(d);
  const float inv_sqrt_d = rsqrtf(static_cast<float>(d));
  const In *kb = k + bh * T * d;
  const In *vb = v + bh * T * d;
  float *sk = simt_smem, *sv = simt_smem + tile * d;

  float qv[PER], bj[PER], c[PER], A[PER], W[PER];
#pragma unroll
  for (int u = 0; u < PER; ++u) {
    const int j = lane + 32 * u;
    const bool ok = valid && u < per && j < d;
    qv[u] = ok ? ld_in(q + row * d + j) : 0.f;
    bj[u] = ok ? beta[h * d + j] : 0.f;
    c[u] = -INFINITY;
    A[u] = 0.f;
    W[u] = 0.f;
  }
  float m = -INFINITY, L = 0.f;

  for (int i0 = 0; i0 < n_blk; i0 += tile) {
    const int nt = min(tile, n_blk - i0);
    __syncthreads();  // the previous tile is consumed
    for (int e = tid; e < nt * d; e += 128) {
      sk[e] = ld_in(kb + static_cast<long long>(i0) * d + e);
      sv[e] = ld_in(vb + static_cast<long long>(i0) * d + e);
    }
    __syncthreads();
    const int n_here = min(nt, n - i0);  // this row's keys in the tile
    // SPLIT: this warp's quarter of them
    const int quarter = (n_here + 3) / 4;
    const int ii0 = SPLIT ? min(n_here, warp * quarter) : 0, ii1 = SPLIT ? min(n_here, ii0 + quarter) : n_here;
    for (int ii = ii0; ii < ii1; ++ii) {
      const float *kr = sk + ii * d;
      float part = 0.f;
#pragma unroll
      for (int u = 0; u < PER; ++u) {
        const int j = lane + 32 * u;
        if (u < per && j < d) part = fmaf(qv[u], kr[j], part);
      }
#pragma unroll
      for (int off = 16; off; off >>= 1) part += __shfl_xor_sync(0xffffffffu, part, off);
      const float s = part * inv_sqrt_d;
      if (s > m) {
        const float alpha = expf(m - s);  // 0 when m = -inf
        L *= alpha;
#pragma unroll
        for (int u = 0; u < PER; ++u) {
          A[u] *= alpha;
          W[u] *= alpha;
        }
        m = s;
      }
      const float p = expf(s - m);
      const float *vr = sv + ii * d;
#pragma unroll
      for (int u = 0; u < PER; ++u) {
        const int j = lane + 32 * u;
        if (!(u < per && j < d)) continue;
        const float x = vr[j];
        const float b = bj[u];
        if (x > c[u]) {
          if (c[u] != -INFINITY) {
            const float r = expf(b * (c[u] - x));
            W[u] = r * W[u] + expm1_over_beta(b, c[u] - x) * L;
            A[u] *= r;
          }
          c[u] = x;
        }
        A[u] += p * expf(b * (x - c[u]));
        W[u] += p * expm1_over_beta(b, x - c[u]);
      }
      L += p;
    }
  }
  if (SPLIT) {
    // warps 1..3 leave their states in shared memory (m, L, then c, A, W per channel); warp 0
    // folds them into its own in key order
    __syncthreads();  // the last tile is consumed
    float *st = simt_smem + (warp - 1) * (2 + 3 * d);
    if (warp > 0) {
      if (lane == 0) {
        st[0] = m;
        st[1] = L;
      }
#pragma unroll
      for (int u = 0; u < PER; ++u) {
        const int j = lane + 32 * u;
        if (!(u < per && j < d)) continue;
        st[2 + j] = c[u];
        st[2 + d + j] = A[u];
        st[2 + 2 * d + j] = W[u];
      }
    }
    __syncthreads();
    if (warp > 0) return;
    for (int w = 1; w < 4; ++w) {
      const float *sw = simt_smem + (w - 1) * (2 + 3 * d);
      const float m2 = sw[0], L2 = sw[1];
      if (m2 == -INFINITY) continue;  // a warp that saw no key
      if (m == -INFINITY) {           // this one saw none: take the other state
        m = m2;
        L = L2;
#pragma unroll
        for (int u = 0; u < PER; ++u) {
          const int j = lane + 32 * u;
          if (!(u < per && j < d)) continue;
          c[u] = sw[2 + j];
          A[u] = sw[2 + d + j];
          W[u] = sw[2 + 2 * d + j];
        }
        continue;
      }
      const float mn = fmaxf(m, m2), a1 = expf(m - mn), a2 = expf(m2 - mn);
      const float L1 = L * a1, Ls = L2 * a2;
#pragma unroll
      for (int u = 0; u < PER; ++u) {
        const int j = lane + 32 * u;
        if (!(u < per && j < d)) continue;
        const float b = bj[u], c2 = sw[2 + j];
        float A1 = A[u] * a1, W1 = W[u] * a1, A2 = sw[2 + d + j] * a2, W2 = sw[2 + 2 * d + j] * a2;
        if (c2 > c[u]) {
          const float r = expf(b * (c[u] - c2));
          W1 = r * W1 + expm1_over_beta(b, c[u] - c2) * L1;
          A1 *= r;
          c[u] = c2;
        } else if (c2 < c[u]) {
          const float r = expf(b * (c2 - c[u]));
          W2 = r * W2 + expm1_over_beta(b, c2 - c[u]) * Ls;
          A2 *= r;
        }
        A[u] = A1 + A2;
        W[u] = W1 + W2;
      }
      L = L1 + Ls;
      m = mn;
    }
  }
  if (!valid) return;

#pragma unroll
  for (int u = 0; u < PER; ++u) {
    const int j = lane + 32 * u;
    if (!(u < per && j < d)) continue;
    const float b = bj[u];
    float o;
    if (b == 0.f) {
      o = c[u] + W[u] / L;
    } else {
      const float z = b * W[u] / L;
      o = z > -0.5f ? c[u] + log1pf(z) / b : c[u] + logf(A[u] / L) / b;
    }
    out[row * d + j] = o;
  }
  if (lse && lane == 0) lse[row] = m + logf(L);
}

template <typename In>
static cudaError_t launch_simt(const In *q, const In *k, const In *v, const float *beta, float *out, float *lse, int B,
                               int H, int T, int d, int causal, cudaStream_t stream) {
  if (d > 32 * kSimtMaxPerLane) return cudaErrorInvalidValue;
  // few rows: a block per row, its keys split over the four warps (the merge area of three
  // states fits in the staging space: 3 (2 + 3 d) <= 2 tile d floats)
  const long long rows = static_cast<long long>(B) * H * T;
  const bool split = rows <= kSimtSplitRows;
  const unsigned blocks = static_cast<unsigned>(split ? rows : static_cast<long long>(B) * H * ((T + 3) / 4));
  const size_t smem = 2 * static_cast<size_t>(fem_simt_tile(d)) * d * sizeof(float);
  const int per = (d + 31) / 32;
#define FEM_SIMT_LAUNCH(P)                                                                                          \
  (split ? fem_simt_kernel<In, P, true><<<blocks, 128, smem, stream>>>(q, k, v, beta, out, lse, H, T, d, causal)     \
         : fem_simt_kernel<In, P, false><<<blocks, 128, smem, stream>>>(q, k, v, beta, out, lse, H, T, d, causal))
  if (per == 1)
    FEM_SIMT_LAUNCH(1);
  else if (per == 2)
    FEM_SIMT_LAUNCH(2);
  else if (per <= 4)
    FEM_SIMT_LAUNCH(4);
  else
    FEM_SIMT_LAUNCH(8);
#undef FEM_SIMT_LAUNCH
  return cudaGetLastError();
}

cudaError_t launch_f32(const float *q, const float *k, const float *v, const float *beta, float *out, float *lse,
                       int B, int H, int T, int d, int causal, cudaStream_t stream) {
  return launch_simt<float>(q, k, v, beta, out, lse, B, H, T, d, causal, stream);
}

cudaError_t launch_simt_bf16(const void *q, const void *k, const void *v, const float *beta, float *out, float *lse,
                             int B, int H, int T, int d, int causal, cudaStream_t stream) {
  return launch_simt<__nv_bfloat16>(static_cast<const __nv_bfloat16 *>(q), static_cast<const __nv_bfloat16 *>(k),
                                    static_cast<const __nv_bfloat16 *>(v), beta, out, lse, B, H, T, d, causal, stream);
}

}  // namespace fem
