// Backward of the read for fp32 inputs on CUDA cores, from the saved out and
// lse (flash-attention-style recomputation of the scores).  With
// p_{t,i} = exp(s_{t,i} - lse_t) and x = beta_j (v_{i,j} - o_{t,j}), the
// posterior is q_{t,i,j} = p_{t,i} exp(x) (since beta_j o_{t,j} + lse_t is its
// log-normaliser), and the derivatives of the read are
//
//   dF_{t,j}/dv_{i,j} = q_{t,i,j}                      (Prop. "app-geom")
//   dF_{t,j}/ds_{t,i} = (q - p)/beta = p expm1(x)/beta  (Prop. "app-bounds" (iv))
//   dF_{t,j}/dbeta_j  = KL(q || p)/beta^2 = sum_i p phi(x)/beta^2,
//                       phi(x) = 1 + (x - 1) e^x        (Eq. "app-beta-deriv")
//
// (sum_i p_i e^x = 1 turns KL = beta (E_q v - o) into the cancellation-free
// sum of p phi(x) >= 0; at beta = 0 they become v - o and (v - o)^2 / 2).
// Two passes, each a warp per group of consecutive rows: rows (dq and dbeta,
// with dS_{t,i} = sum_j dout_{t,j} dF_{t,j}/ds_{t,i}), then keys (dk and dv,
// summing over the rows that see the key).
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

// For y = v - o, x = b y and the log prior weight lp2 = (s - lse) log2 e, the
// p-weighted terms q = p e^x, p expm1(x)/b and p phi(x)/b^2, formed without
// e^x alone (which can overflow where p is tiny) and continuous at b = 0.
// The exponentials go to the special-function unit in base 2 (relative error
// about 2^-22); expm1(x)/b for |x| < 1/2 is y times the Taylor series of
// expm1(x)/x (truncation below 4e-6 relative); inv_b and inv_b2 are 1/b and
// 1/b^2 (0 at b = 0, where only the series branches are taken).
__device__ __forceinline__ void bwd_terms(float b, float inv_b, float inv_b2, float y, float lp2, float &qv,
                                          float &ds, float &dbt) {
  const float x = b * y, p = ex2_approx(lp2);
  qv = ex2_approx(fmaf(x, kLog2e, lp2));
  if (fabsf(x) < 0.5f) {
    float poly = fmaf(x, 1.f / 720.f, 1.f / 120.f);
    poly = fmaf(x, poly, 1.f / 24.f);
    poly = fmaf(x, poly, 1.f / 6.f);
    poly = fmaf(x, poly, 0.5f);
    poly = fmaf(x, poly, 1.f);
    ds = p * y * poly;
  } else {
    ds = (qv - p) * inv_b;
  }
  if (fabsf(x) < 0.1f) {
    // phi(x) = x^2/2 + x^3/3 + x^4/8 + x^5/30 + x^6/144 + ..., divided by b^2
    dbt = p * y * y * fmaf(x, fmaf(x, fmaf(x, fmaf(x, 1.f / 144.f, 1.f / 30.f), 0.125f), 1.f / 3.f), 0.5f);
  } else {
    dbt = fmaf(x - 1.f, qv, p) * inv_b2;  // p phi(x) = p + (x - 1) q
  }
}

// MODE 0: a warp per R consecutive query rows t -> dq_t and the rows' dbeta terms.
// MODE 1: a warp per R consecutive key rows i  -> dk_i and dv_i.
// Lane l holds channels l + 32 u (u < PER); the R rows share every load of
// the other side's row and their butterfly sums interleave.
template <int MODE, int R, int PER>
__global__ void __launch_bounds__(128) fem_bwd_kernel(const float *__restrict__ q, const float *__restrict__ k,
                                                       const float *__restrict__ v, const float *__restrict__ beta,
                                                       const float *__restrict__ out, const float *__restrict__ lse,
                                                       const float *__restrict__ dout, float *__restrict__ da,
                                                       float *__restrict__ db, float *__restrict__ dbeta, int H,
                                                       int T, int d, int causal, long long n_groups) {
  const int lane = threadIdx.x & 31;
  const long long grp = static_cast<long long>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (grp >= n_groups) return;
  const int gpb = (T + R - 1) / R;  // row groups per (b, h)
  const long long bh = grp / gpb;
  const int r0 = static_cast<int>(grp % gpb) * R;
  const int nr = min(R, T - r0);  // rows of this group
  const int h = static_cast<int>(bh % H);
  const float inv_sqrt_d = rsqrtf(static_cast<float>(d));
  const size_t base = static_cast<size_t>(bh) * T * d;
  float bj[PER], ib[PER];
  float own[R][PER], own2[R][PER], own3[R][PER], acc1[R][PER], acc2[R][PER], lse_r[R];
#pragma unroll
  for (int u = 0; u < PER; ++u) {
    const int j = lane + 32 * u;
    bj[u] = j < d ? beta[h * d + j] : 0.f;
    ib[u] = bj[u] != 0.f ? 1.f / bj[u] : 0.f;
  }
#pragma unroll
  for (int w = 0; w < R; ++w) {
    const int r = min(r0 + w, T - 1);  // rows past T repeat the last one; their results are not stored
    lse_r[w] = MODE == 0 ? lse[bh * T + r] : 0.f;
#pragma unroll
    for (int u = 0; u < PER; ++u) {
      const int j = lane + 32 * u;
      const bool ok = j < d;
      // MODE 0: own = q_t, own2 = o_t, own3 = dout_t;  MODE 1: own = k_i, own2 = v_i
      own[w][u] = ok ? (MODE == 0 ? q : k)[base + static_cast<size_t>(r) * d + j] : 0.f;
      own2[w][u] = ok ? (MODE == 0 ? out : v)[base + static_cast<size_t>(r) * d + j] : 0.f;
      own3[w][u] = ok && MODE == 0 ? dout[base + static_cast<size_t>(r) * d + j] : 0.f;
      acc1[w][u] = 0.f;
      acc2[w][u] = 0.f;
    }
  }
  // the other side of the score: keys 0 .. (causal ? last row : T-1) for rows,
  // rows (causal ? first key : 0) .. T-1 for keys
  const int lo = MODE == 0 ? 0 : (causal ? r0 : 0);
  const int hi = MODE == 0 ? (causal ? r0 + nr : T) : T;
  for (int o = lo; o < hi; ++o) {
    const size_t ob = base + static_cast<size_t>(o) * d;
    float oth[PER], oth2[PER], oth3[PER];
#pragma unroll
    for (int u = 0; u < PER; ++u) {
      const int j = lane + 32 * u;
      const bool ok = j < d;
      oth[u] = ok ? (MODE == 0 ? k : q)[ob + j] : 0.f;
      oth2[u] = ok ? (MODE == 0 ? v : out)[ob + j] : 0.f;
      oth3[u] = ok && MODE == 1 ? dout[ob + j] : 0.f;
    }
    const float lse_o = MODE == 1 ? lse[bh * T + o] : 0.f;
    float part[R];
#pragma unroll
    for (int w = 0; w < R; ++w) {
      part[w] = 0.f;
#pragma unroll
      for (int u = 0; u < PER; ++u) part[w] = fmaf(own[w][u], oth[u], part[w]);
    }
#pragma unroll
    for (int off = 16; off; off >>= 1)
#pragma unroll
      for (int w = 0; w < R; ++w) part[w] += __shfl_xor_sync(0xffffffffu, part[w], off);
    float dS[R];
#pragma unroll
    for (int w = 0; w < R; ++w) {
      // the pair (query row, key) is visible: key <= row when causal
      const int rw = r0 + w;
      const bool vis = !causal || (MODE == 0 ? o <= rw : rw <= o);
      const float lp2 = vis ? (part[w] * inv_sqrt_d - (MODE == 0 ? lse_r[w] : lse_o)) * kLog2e : -INFINITY;
      dS[w] = 0.f;
#pragma unroll
      for (int u = 0; u < PER; ++u) {
        // y = v_{i,j} - o_{t,j} with (i, t) = (o, row) for rows and (row, o) for keys
        const float y = MODE == 0 ? oth2[u] - own2[w][u] : own2[w][u] - oth2[u];
        const float g = MODE == 0 ? own3[w][u] : oth3[u];
        float qv, ds, dbt;
        bwd_terms(bj[u], ib[u], ib[u] * ib[u], y, lp2, qv, ds, dbt);
        dS[w] = fmaf(g, ds, dS[w]);
        if (MODE == 0) acc2[w][u] = fmaf(g, dbt, acc2[w][u]);  // dbeta terms of this row
        else acc2[w][u] = fmaf(g, qv, acc2[w][u]);             // dv_i: sum_t dout_{t,j} q_{t,i,j}
      }
    }
#pragma unroll
    for (int off = 16; off; off >>= 1)
#pragma unroll
      for (int w = 0; w < R; ++w) dS[w] += __shfl_xor_sync(0xffffffffu, dS[w], off);
#pragma unroll
    for (int w = 0; w < R; ++w)
#pragma unroll
      for (int u = 0; u < PER; ++u) acc1[w][u] = fmaf(dS[w], oth[u], acc1[w][u]);
  }
#pragma unroll
  for (int w = 0; w < R; ++w) {
    if (w >= nr) break;
    const int r = r0 + w;
#pragma unroll
    for (int u = 0; u < PER; ++u) {
      const int j = lane + 32 * u;
      if (j >= d) continue;
      da[base + static_cast<size_t>(r) * d + j] = acc1[w][u] * inv_sqrt_d;
      if (MODE == 0) atomicAdd(&dbeta[h * d + j], acc2[w][u]);
      else db[base + static_cast<size_t>(r) * d + j] = acc2[w][u];
    }
  }
}

template <int R, int PER>
static cudaError_t launch_bwd_rp(const float *q, const float *k, const float *v, const float *beta, const float *out,
                                 const float *lse, const float *dout, float *dq, float *dk, float *dv, float *dbeta,
                                 int B, int H, int T, int d, int causal, cudaStream_t stream) {
  const long long n_groups = static_cast<long long>(B) * H * ((T + R - 1) / R);
  const unsigned blocks = static_cast<unsigned>((n_groups + 3) / 4);
  fem_bwd_kernel<0, R, PER><<<blocks, 128, 0, stream>>>(q, k, v, beta, out, lse, dout, dq, nullptr, dbeta, H, T, d,
                                                        causal, n_groups);
  fem_bwd_kernel<1, R, PER><<<blocks, 128, 0, stream>>>(q, k, v, beta, out, lse, dout, dk, dv, nullptr, H, T, d,
                                                        causal, n_groups);
  return cudaGetLastError();
}

cudaError_t launch_bwd_f32(const float *q, const float *k, const float *v, const float *beta, const float *out,
                           const float *lse, const float *dout, float *dq, float *dk, float *dv, float *dbeta, int B,
                           int H, int T, int d, int causal, cudaStream_t stream) {
  cudaError_t e = cudaMemsetAsync(dbeta, 0, static_cast<size_t>(H) * d * sizeof(float), stream);
  if (e != cudaSuccess) return e;
  // rows per warp: four while a lane holds at most two channels, fewer beyond
  if (d <= 32) return launch_bwd_rp<4, 1>(q, k, v, beta, out, lse, dout, dq, dk, dv, dbeta, B, H, T, d, causal, stream);
  if (d <= 64) return launch_bwd_rp<4, 2>(q, k, v, beta, out, lse, dout, dq, dk, dv, dbeta, B, H, T, d, causal, stream);
  if (d <= 128) return launch_bwd_rp<2, 4>(q, k, v, beta, out, lse, dout, dq, dk, dv, dbeta, B, H, T, d, causal, stream);
  if (d <= 256) return launch_bwd_rp<1, 8>(q, k, v, beta, out, lse, dout, dq, dk, dv, dbeta, B, H, T, d, causal, stream);
  return cudaErrorInvalidValue;
}

}  // namespace fem
