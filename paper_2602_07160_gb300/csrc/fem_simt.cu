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
// issue slots even where a slot is empty)
template <typename In, int PER>
__global__ void __launch_bounds__(128) fem_simt_kernel(const In *__restrict__ q, const In *__restrict__ k,
                                                        const In *__restrict__ v, const float *__restrict__ beta,
                                                        float *__restrict__ out, float *__restrict__ lse, int H,
                                                        int T, int d, int causal) {
  extern __shared__ float simt_smem[];  // [tile][d] K, then [tile][d] V
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int bpr = (T + 3) / 4;  // blocks per (b, h)
  const long long bh = blockIdx.x / bpr;
  const int t0 = static_cast<int>(blockIdx.x % bpr) * 4, t = t0 + warp;
  const bool valid = t < T;
  const long long row = bh * T + t;
  const int h = static_cast<int>(bh % H);
  const int n = !valid ? 0 : (causal ? t + 1 : T);  // keys this row sees
  const int n_blk = causal ? min(T, t0 + 4) : T;    // keys any row of the block sees
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
    for (int ii = 0; ii < n_here; ++ii) {
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
  const unsigned blocks = static_cast<unsigned>(static_cast<long long>(B) * H * ((T + 3) / 4));
  const size_t smem = 2 * static_cast<size_t>(fem_simt_tile(d)) * d * sizeof(float);
  const int per = (d + 31) / 32;
  if (per == 1)
    fem_simt_kernel<In, 1><<<blocks, 128, smem, stream>>>(q, k, v, beta, out, lse, H, T, d, causal);
  else if (per == 2)
    fem_simt_kernel<In, 2><<<blocks, 128, smem, stream>>>(q, k, v, beta, out, lse, H, T, d, causal);
  else if (per <= 4)
    fem_simt_kernel<In, 4><<<blocks, 128, smem, stream>>>(q, k, v, beta, out, lse, H, T, d, causal);
  else
    fem_simt_kernel<In, 8><<<blocks, 128, smem, stream>>>(q, k, v, beta, out, lse, H, T, d, causal);
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
