// FEM read over a gated-linear-attention prior (App. "Gated Linear Attention
// (GLA) Prior"): with nonnegative features qf, kf (the caller's
// ReLU(RoPE(.)) + eps) and per-step log-decays g_t <= 0,
//
//   s_t(i) = K_{t,i} <qf_t, kf_i>  (i <= t),  K_{t,i} = exp(g_{i+1} + ... + g_t),
//   p_t = s_t / Z_t,   o_{t,j} = (1/beta_j) log sum_i p_t(i) exp(beta_j v_{i,j}).
//
// The associative form (Eq. "gla-assoc") turns every channel into a linear-
// attention state: o_{t,j} = (1/beta_j) log(<qf_t, S_{t,j}> / <qf_t, S_t>)
// with S_{t,j} = sum_{i<=t} K_{t,i} kf_i exp(beta_j v_{i,j}), and the
// normaliser Z_t = <qf_t, S_t>, S_t = sum_i K_{t,i} kf_i, is the same state for
// a constant channel (the paper's "constant 1 channel").  A channel's state is
// kept as exp(lam) S^ with the log-scale lam_t = max(lam_{t-1} + g_t,
// beta v_{t,j}) -- the log of its largest term, which decays with the prior --
// so neither exp(beta v) nor the decay under- or overflows (the per-channel
// stabilisation of App. E); the normaliser's scale stays 0.  At beta_j = 0 the
// state carries v itself and o is the ratio (the prior mean).
//
// One block per (b, h).  Four lanes share a channel, each keeping a quarter
// of its m-float state in registers (a warp holds 7 channels and the constant
// channel), so the per-step chains are short and a head has several warps.
// The block stages qf, kf, exp(g), g and v for kGlaSteps steps in shared
// memory and writes the steps' outputs from there.  A recurrent O(T) scan in
// fp32 on CUDA cores.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

constexpr int kGlaSteps = 16;
constexpr int kGlaParts = 4;                          // lanes per channel
constexpr int kGlaChPerWarp = 32 / kGlaParts - 1;     // real channels per warp (the 8th is the normaliser)
constexpr int kGlaMaxD = 155;
constexpr int kGlaMaxWarps = (kGlaMaxD + kGlaChPerWarp - 1) / kGlaChPerWarp;

template <int M>
__global__ void __launch_bounds__(32 * kGlaMaxWarps) gla_kernel(const float *__restrict__ qf,
                                                                const float *__restrict__ kf,
                                                                const float *__restrict__ v,
                                                                const float *__restrict__ logdecay,
                                                                const float *__restrict__ beta,
                                                                float *__restrict__ out, float *__restrict__ logz,
                                                                int H, int T, int d) {
  constexpr int MP = M / kGlaParts;  // state floats per lane
  __shared__ __align__(16) float s_q[kGlaSteps][M];
  __shared__ __align__(16) float s_k[kGlaSteps][M];
  __shared__ float s_v[kGlaSteps][kGlaMaxD];
  __shared__ float s_o[kGlaSteps][kGlaMaxD];
  __shared__ float s_a[kGlaSteps], s_g[kGlaSteps], s_lz[kGlaSteps];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int bh = blockIdx.x, h = bh % H;
  const int cw = lane / kGlaParts, part = lane % kGlaParts;
  const bool norm = cw == kGlaChPerWarp;
  const int j = warp * kGlaChPerWarp + cw;            // this lane's channel
  const bool real = !norm && j < d;
  const float b = real ? beta[h * d + j] : 0.f;
  const bool lin = b == 0.f;                          // the state carries v itself
  const size_t row0 = static_cast<size_t>(bh) * T;
  float S[MP];
#pragma unroll
  for (int i = 0; i < MP; ++i) S[i] = 0.f;
  float lam = -INFINITY;  // log-scale of a beta > 0 channel's state
  for (int t0 = 0; t0 < T; t0 += kGlaSteps) {
    const int n = min(kGlaSteps, T - t0);
    for (int e = tid; e < n * M; e += blockDim.x) {
      s_q[e / M][e % M] = qf[(row0 + t0) * M + e];
      s_k[e / M][e % M] = kf[(row0 + t0) * M + e];
    }
    for (int e = tid; e < n * d; e += blockDim.x) s_v[e / d][e % d] = v[(row0 + t0) * d + e];
    for (int e = tid; e < n; e += blockDim.x) {
      const float g = logdecay[row0 + t0 + e];
      s_g[e] = g;
      s_a[e] = expf(g);
    }
    __syncthreads();
    for (int u = 0; u < n; ++u) {
      const float x = real ? s_v[u][j] : 0.f;
      float E, a;
      if (!real) {
        E = 1.f;
        a = s_a[u];
      } else if (lin) {
        E = x;
        a = s_a[u];
      } else {
        const float le = b * x, lo = lam + s_g[u];
        const float ln = fmaxf(lo, le);
        a = expf(lo - ln);  // 0 on the first step
        E = expf(le - ln);
        lam = ln;
      }
      const float4 *k4 = reinterpret_cast<const float4 *>(&s_k[u][part * MP]);
      const float4 *q4 = reinterpret_cast<const float4 *>(&s_q[u][part * MP]);
      float n0 = 0.f, n1 = 0.f;
#pragma unroll
      for (int i4 = 0; i4 < MP / 4; ++i4) {
        const float4 kk = k4[i4], qq = q4[i4];
        S[4 * i4] = fmaf(a, S[4 * i4], E * kk.x);
        S[4 * i4 + 1] = fmaf(a, S[4 * i4 + 1], E * kk.y);
        S[4 * i4 + 2] = fmaf(a, S[4 * i4 + 2], E * kk.z);
        S[4 * i4 + 3] = fmaf(a, S[4 * i4 + 3], E * kk.w);
        n0 = fmaf(qq.x, S[4 * i4], n0);
        n1 = fmaf(qq.y, S[4 * i4 + 1], n1);
        n0 = fmaf(qq.z, S[4 * i4 + 2], n0);
        n1 = fmaf(qq.w, S[4 * i4 + 3], n1);
      }
      float num = n0 + n1;
#pragma unroll
      for (int off = 1; off < kGlaParts; off <<= 1) num += __shfl_xor_sync(0xffffffffu, num, off);
      const float den = __shfl_sync(0xffffffffu, num, kGlaChPerWarp * kGlaParts);  // Z_t, the constant channel
      if (real && part == 0) s_o[u][j] = lin ? num / den : (lam + (logf(num) - logf(den))) / b;
      if (warp == 0 && lane == kGlaChPerWarp * kGlaParts) s_lz[u] = logf(den);
    }
    __syncthreads();  // the steps' outputs are in shared memory; the staged inputs are consumed
    for (int e = tid; e < n * d; e += blockDim.x) out[(row0 + t0) * d + e] = s_o[e / d][e % d];
    if (logz)
      for (int e = tid; e < n; e += blockDim.x) logz[row0 + t0 + e] = s_lz[e];
  }
}

cudaError_t launch_gla(const float *qf, const float *kf, const float *v, const float *logdecay, const float *beta,
                       float *out, float *logz, int BH, int H, int T, int m, int d, cudaStream_t stream) {
  if (d > kGlaMaxD) return cudaErrorInvalidValue;
  const int warps = (d + kGlaChPerWarp - 1) / kGlaChPerWarp;
  const dim3 grid(BH), block(32 * warps);
  switch (m) {
    case 16: gla_kernel<16><<<grid, block, 0, stream>>>(qf, kf, v, logdecay, beta, out, logz, H, T, d); break;
    case 32: gla_kernel<32><<<grid, block, 0, stream>>>(qf, kf, v, logdecay, beta, out, logz, H, T, d); break;
    case 64: gla_kernel<64><<<grid, block, 0, stream>>>(qf, kf, v, logdecay, beta, out, logz, H, T, d); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace fem
