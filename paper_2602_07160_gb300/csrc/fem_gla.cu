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
// The scan is linear in the state, so the time axis is split into segments
// (three passes): each segment's end state from a zero start, in parallel;
// the segments' start states by a short sequential combine over segments,
// start(p+1) = exp(Phi_p) start(p) + local_end(p) with Phi_p the segment's
// summed log-decay (log-scaled like the states); then every segment again
// from its start state, writing the outputs.  Within a segment four lanes
// share a channel, each keeping a quarter of its m-float state in registers
// (a warp holds 7 channels and the constant channel), and the block stages
// qf, kf, g and v for kGlaSteps steps in shared memory, in two buffers filled
// by asynchronous copies one stage ahead.  fp32 on CUDA cores.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

constexpr int kGlaSteps = 16;
constexpr int kGlaParts = 4;                          // lanes per channel
constexpr int kGlaChPerWarp = 32 / kGlaParts - 1;     // real channels per warp (the 8th is the normaliser)
constexpr int kGlaMaxD = 155;
constexpr int kGlaMaxWarps = (kGlaMaxD + kGlaChPerWarp - 1) / kGlaChPerWarp;

__device__ __forceinline__ void cp_async4(float *dst, const float *src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// Per-lane role within a block of one (b, h).
struct GlaLane {
  int warp, lane, part, j;
  bool real, lin;
  float b;
};

__device__ __forceinline__ GlaLane gla_lane(const float *beta, int h, int d) {
  GlaLane L;
  L.warp = threadIdx.x >> 5;
  L.lane = threadIdx.x & 31;
  const int cw = L.lane / kGlaParts;
  L.part = L.lane % kGlaParts;
  L.j = L.warp * kGlaChPerWarp + cw;
  L.real = cw != kGlaChPerWarp && L.j < d;
  L.b = L.real ? beta[h * d + L.j] : 0.f;
  L.lin = L.b == 0.f;
  return L;
}

// MODE 0: the segment's end state from a zero start, and its summed log-decay.
// MODE 1: the segment from its start state, writing out and log Z.
template <int M, int MODE>
__global__ void __launch_bounds__(32 * kGlaMaxWarps) gla_seg_kernel(
    const float *__restrict__ qf, const float *__restrict__ kf, const float *__restrict__ v,
    const float *__restrict__ logdecay, const float *__restrict__ beta, float *__restrict__ out,
    float *__restrict__ logz, int H, int T, int d, int seg_len, float *__restrict__ state, float *__restrict__ phi) {
  constexpr int MP = M / kGlaParts;  // state floats per lane
  // the staged inputs in two buffers: the next stage's copies land while this one runs
  __shared__ __align__(16) float s_q[2][kGlaSteps][M];
  __shared__ __align__(16) float s_k[2][kGlaSteps][M];
  __shared__ float s_v[2][kGlaSteps][kGlaMaxD];
  __shared__ float s_g[2][kGlaSteps];
  __shared__ float s_o[kGlaSteps][kGlaMaxD];
  __shared__ float s_a[kGlaSteps], s_lz[kGlaSteps];
  const int tid = threadIdx.x, p = blockIdx.x, n_seg = gridDim.x, bh = blockIdx.y, h = bh % H;
  const GlaLane L = gla_lane(beta, h, d);
  const size_t row0 = static_cast<size_t>(bh) * T;
  const int t_begin = p * seg_len, t_end = min(T, t_begin + seg_len);
  float *st = state + ((static_cast<size_t>(bh) * n_seg + p) * blockDim.x + tid) * (MP + 1);
  float S[MP];
  float lam = -INFINITY;  // log-scale of a beta > 0 channel's state
  if (MODE == 0) {
#pragma unroll
    for (int i = 0; i < MP; ++i) S[i] = 0.f;
  } else {
#pragma unroll
    for (int i = 0; i < MP; ++i) S[i] = st[i];
    lam = st[MP];
  }
  float phi_acc = 0.f;
  // a stage's inputs by asynchronous 4-byte copies (any d), one commit group per stage
  auto stage = [&](int ts, int buf) {
    const int ns = min(kGlaSteps, t_end - ts);
    for (int e = tid; e < ns * M; e += blockDim.x) {
      cp_async4(&s_q[buf][e / M][e % M], qf + (row0 + ts) * M + e);
      cp_async4(&s_k[buf][e / M][e % M], kf + (row0 + ts) * M + e);
    }
    for (int e = tid; e < ns * d; e += blockDim.x) cp_async4(&s_v[buf][e / d][e % d], v + (row0 + ts) * d + e);
    for (int e = tid; e < ns; e += blockDim.x) cp_async4(&s_g[buf][e], logdecay + row0 + ts + e);
    cp_async_commit();
  };
  if (t_begin < t_end) stage(t_begin, 0);
  int buf = 0;
  for (int t0 = t_begin; t0 < t_end; t0 += kGlaSteps, buf ^= 1) {
    const int n = min(kGlaSteps, t_end - t0);
    // this stage's copies have landed, and every thread is done with the
    // previous stage (whose buffer the next prefetch overwrites)
    cp_async_wait_all();
    __syncthreads();
    if (t0 + kGlaSteps < t_end) stage(t0 + kGlaSteps, buf ^ 1);
    for (int e = tid; e < n; e += blockDim.x) s_a[e] = expf(s_g[buf][e]);
    __syncthreads();
    for (int u = 0; u < n; ++u) {
      const float x = L.real ? s_v[buf][u][L.j] : 0.f;
      float E, a;
      if (!L.real) {
        E = 1.f;
        a = s_a[u];
      } else if (L.lin) {
        E = x;
        a = s_a[u];
      } else {
        const float le = L.b * x, lo = lam + s_g[buf][u];
        const float ln = fmaxf(lo, le);
        a = expf(lo - ln);  // 0 on the first step of a zero state
        E = expf(le - ln);
        lam = ln;
      }
      if (MODE == 0) phi_acc += s_g[buf][u];
      const float4 *k4 = reinterpret_cast<const float4 *>(&s_k[buf][u][L.part * MP]);
      const float4 *q4 = reinterpret_cast<const float4 *>(&s_q[buf][u][L.part * MP]);
      float n0 = 0.f, n1 = 0.f;
#pragma unroll
      for (int i4 = 0; i4 < MP / 4; ++i4) {
        const float4 kk = k4[i4];
        S[4 * i4] = fmaf(a, S[4 * i4], E * kk.x);
        S[4 * i4 + 1] = fmaf(a, S[4 * i4 + 1], E * kk.y);
        S[4 * i4 + 2] = fmaf(a, S[4 * i4 + 2], E * kk.z);
        S[4 * i4 + 3] = fmaf(a, S[4 * i4 + 3], E * kk.w);
        if (MODE == 1) {
          const float4 qq = q4[i4];
          n0 = fmaf(qq.x, S[4 * i4], n0);
          n1 = fmaf(qq.y, S[4 * i4 + 1], n1);
          n0 = fmaf(qq.z, S[4 * i4 + 2], n0);
          n1 = fmaf(qq.w, S[4 * i4 + 3], n1);
        }
      }
      if (MODE == 1) {
        float num = n0 + n1;
#pragma unroll
        for (int off = 1; off < kGlaParts; off <<= 1) num += __shfl_xor_sync(0xffffffffu, num, off);
        const float den = __shfl_sync(0xffffffffu, num, kGlaChPerWarp * kGlaParts);  // Z_t, the constant channel
        if (L.real && L.part == 0) s_o[u][L.j] = L.lin ? num / den : (lam + (logf(num) - logf(den))) / L.b;
        if (L.warp == 0 && L.lane == kGlaChPerWarp * kGlaParts) s_lz[u] = logf(den);
      }
    }
    if (MODE == 1) {
      __syncthreads();  // the steps' outputs are in shared memory
      for (int e = tid; e < n * d; e += blockDim.x) out[(row0 + t0) * d + e] = s_o[e / d][e % d];
      if (logz)
        for (int e = tid; e < n; e += blockDim.x) logz[row0 + t0 + e] = s_lz[e];
    }
  }
  if (MODE == 0) {
#pragma unroll
    for (int i = 0; i < MP; ++i) st[i] = S[i];
    st[MP] = lam;
    if (tid == 0) phi[static_cast<size_t>(bh) * n_seg + p] = phi_acc;
  }
}

// Start states in place of the local end states: start(0) = 0 and
// start(p+1) = exp(Phi_p) start(p) + local_end(p), log-scaled for beta > 0.
template <int M>
__global__ void __launch_bounds__(32 * kGlaMaxWarps) gla_combine_kernel(const float *__restrict__ beta, int H, int d,
                                                                        int n_seg, float *__restrict__ state,
                                                                        const float *__restrict__ phi) {
  constexpr int MP = M / kGlaParts;
  const int tid = threadIdx.x, bh = blockIdx.x, h = bh % H;
  const GlaLane L = gla_lane(beta, h, d);
  const bool scaled = L.real && !L.lin;
  float R[MP];
#pragma unroll
  for (int i = 0; i < MP; ++i) R[i] = 0.f;
  float rl = -INFINITY;
  for (int p = 0; p < n_seg; ++p) {
    float *st = state + ((static_cast<size_t>(bh) * n_seg + p) * blockDim.x + tid) * (MP + 1);
    float loc[MP];
#pragma unroll
    for (int i = 0; i < MP; ++i) loc[i] = st[i];
    const float ll = st[MP];
#pragma unroll
    for (int i = 0; i < MP; ++i) st[i] = R[i];
    st[MP] = rl;
    const float f = phi[static_cast<size_t>(bh) * n_seg + p];
    if (scaled) {
      const float lo = rl + f, ln = fmaxf(lo, ll);
      if (ln == -INFINITY) continue;  // both still empty
      const float fr = expf(lo - ln), fl = expf(ll - ln);
#pragma unroll
      for (int i = 0; i < MP; ++i) R[i] = fmaf(fr, R[i], fl * loc[i]);
      rl = ln;
    } else {
      const float fr = expf(f);
#pragma unroll
      for (int i = 0; i < MP; ++i) R[i] = fmaf(fr, R[i], loc[i]);
    }
  }
}

// Resident blocks per SM of the output pass (the heavier of the two passes).
static int gla_blocks_per_sm(int m, int threads) {
  int n = 0;
  cudaError_t e = cudaErrorInvalidValue;
  if (m == 16) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, gla_seg_kernel<16, 1>, threads, 0);
  if (m == 32) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, gla_seg_kernel<32, 1>, threads, 0);
  if (m == 64) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, gla_seg_kernel<64, 1>, threads, 0);
  return e == cudaSuccess && n > 0 ? n : 1;
}

size_t gla_workspace_bytes(int BH, int T, int m, int d, int num_sms, int *seg_len_out, int *n_seg_out) {
  const int warps = (d + kGlaChPerWarp - 1) / kGlaChPerWarp;
  // Segments of at least 64 steps.  A pass takes about (waves of resident
  // blocks) x (segment length) steps of time, so the count minimises that
  // product: whole waves of the grid, not a fraction of a last one.
  const long long cap = static_cast<long long>(gla_blocks_per_sm(m, 32 * warps)) * num_sms;
  const int max_seg = max(1, (T + 63) / 64);
  int n_seg0 = 1;
  long long best = -1;
  for (int ns = 1; ns <= max_seg; ++ns) {
    const long long waves = (static_cast<long long>(BH) * ns + cap - 1) / cap;
    const long long cost = waves * ((T + ns - 1) / ns);
    if (best < 0 || cost < best) {
      best = cost;
      n_seg0 = ns;
    }
    if (waves > 4) break;
  }
  const int seg_len = (T + n_seg0 - 1) / n_seg0;
  const int n_seg = (T + seg_len - 1) / seg_len;
  if (seg_len_out) *seg_len_out = seg_len;
  if (n_seg_out) *n_seg_out = n_seg;
  const size_t per_lane = static_cast<size_t>(m / kGlaParts + 1);
  return (static_cast<size_t>(BH) * n_seg * 32 * warps * per_lane + static_cast<size_t>(BH) * n_seg) * sizeof(float);
}

template <int M>
static cudaError_t launch_gla_m(const float *qf, const float *kf, const float *v, const float *logdecay,
                                const float *beta, float *out, float *logz, int BH, int H, int T, int d, void *ws,
                                int num_sms, cudaStream_t stream) {
  int seg_len = 0, n_seg = 0;
  const int warps = (d + kGlaChPerWarp - 1) / kGlaChPerWarp;
  const size_t bytes = gla_workspace_bytes(BH, T, M, d, num_sms, &seg_len, &n_seg);
  float *state = static_cast<float *>(ws);
  float *phi = state + (bytes / sizeof(float) - static_cast<size_t>(BH) * n_seg);
  const dim3 grid(n_seg, BH), block(32 * warps);
  gla_seg_kernel<M, 0><<<grid, block, 0, stream>>>(qf, kf, v, logdecay, beta, out, logz, H, T, d, seg_len, state, phi);
  gla_combine_kernel<M><<<BH, block, 0, stream>>>(beta, H, d, n_seg, state, phi);
  gla_seg_kernel<M, 1><<<grid, block, 0, stream>>>(qf, kf, v, logdecay, beta, out, logz, H, T, d, seg_len, state, phi);
  return cudaGetLastError();
}

cudaError_t launch_gla(const float *qf, const float *kf, const float *v, const float *logdecay, const float *beta,
                       float *out, float *logz, int BH, int H, int T, int m, int d, void *ws, int num_sms,
                       cudaStream_t stream) {
  if (d > kGlaMaxD) return cudaErrorInvalidValue;
  switch (m) {
    case 16: return launch_gla_m<16>(qf, kf, v, logdecay, beta, out, logz, BH, H, T, d, ws, num_sms, stream);
    case 32: return launch_gla_m<32>(qf, kf, v, logdecay, beta, out, logz, BH, H, T, d, ws, num_sms, stream);
    case 64: return launch_gla_m<64>(qf, kf, v, logdecay, beta, out, logz, BH, H, T, d, ws, num_sms, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace fem
