// Time-decay conditioner convolution (App. "Low-rank Convolution: Time-Decay
// Conditioner (TDC)", Eq. "tdc-conv"): for decay rates s_t >= 0 and inputs u_t
// (per channel of the hidden width H_c),
//
//   h_t = sum_{i<=t} exp(-(s_{i+1} + ... + s_t)) u_i,
//
// a causal separable convolution whose kernel is rank one in time
// (Prop. "tdc-lowrank"), i.e. the first-order recurrence h_t = exp(-s_t) h_{t-1} + u_t.
// HBM-bound (12 bytes per element); the time axis is split into segments:
// segment end states from zero in parallel, a combine over segments
// (start(p+1) = exp(-S_p) start(p) + local_end(p), S_p the segment's summed
// rate), then every segment from its start state writing h.  Thread = channel,
// so every load and store is coalesced over the channels of a step; short
// segments and sixteen steps' loads in flight per thread keep more bytes in
// flight.  The combine is a scan of the affine maps x -> exp(-S_p) x +
// local_end(p): a warp per (b, channel), each lane composing its run of
// segments (eight segments' loads at a time), then a shuffle scan over the
// lanes.  (A single pass with a decoupled look-back over segments measured
// slower: 44 us against 27 us for the three kernels at B4 T8192 Hc64, its
// look-back walking one dependent load at a time.)
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

constexpr int kTdcSeg = 32;  // steps per segment

// MODE 0: local end state and summed rate of a segment; MODE 1: h from the start state.
template <int MODE>
__global__ void tdc_seg_kernel(const float *__restrict__ s, const float *__restrict__ u, float *__restrict__ h, int T,
                               int Hc, float *__restrict__ state, float *__restrict__ rate) {
  const int p = blockIdx.x, n_seg = gridDim.x, b = blockIdx.y;
  const int t0 = p * kTdcSeg, t1 = min(T, t0 + kTdcSeg);
  for (int c = threadIdx.x; c < Hc; c += blockDim.x) {
    const size_t sidx = (static_cast<size_t>(b) * n_seg + p) * Hc + c;
    float acc = MODE == 0 ? 0.f : state[sidx], sum = 0.f;
    // the loads do not depend on the recurrence: sixteen steps' loads in flight
#pragma unroll 16
    for (int t = t0; t < t1; ++t) {
      const size_t e = (static_cast<size_t>(b) * T + t) * Hc + c;
      const float st = s[e];
      acc = fmaf(ex2_approx(-st * kLog2e), acc, u[e]);
      if (MODE == 0) sum += st;
      else h[e] = acc;
    }
    if (MODE == 0) {
      state[sidx] = acc;
      rate[sidx] = sum;
    }
  }
}

__global__ void tdc_combine_kernel(int B, int n_seg, int Hc, float *__restrict__ state, const float *__restrict__ rate) {
  const int wid = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (wid >= B * Hc) return;
  const int b = wid / Hc, c = wid % Hc;
  const int per = (n_seg + 31) / 32, p0 = min(n_seg, lane * per), p1 = min(n_seg, p0 + per);
  float *st = state + static_cast<size_t>(b) * n_seg * Hc + c;
  const float *rt = rate + static_cast<size_t>(b) * n_seg * Hc + c;
  // this lane's segments composed: x -> A x + Bc, eight segments' loads at a time
  constexpr int G = 8;
  float A = 1.f, Bc = 0.f;
  for (int g0 = p0; g0 < p1; g0 += G) {
    float a[G], loc[G];
#pragma unroll
    for (int u = 0; u < G; ++u) {
      const size_t i = static_cast<size_t>(min(g0 + u, p1 - 1)) * Hc;
      a[u] = rt[i];
      loc[u] = st[i];
    }
#pragma unroll
    for (int u = 0; u < G; ++u) {
      if (g0 + u < p1) {
        const float e = expf(-a[u]);
        Bc = fmaf(e, Bc, loc[u]);
        A *= e;
      }
    }
  }
  // inclusive scan over the lanes: lane l's map after lanes 0 .. l-1's
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float Ap = __shfl_up_sync(0xffffffffu, A, off), Bp = __shfl_up_sync(0xffffffffu, Bc, off);
    if (lane >= off) {
      Bc = fmaf(A, Bp, Bc);
      A *= Ap;
    }
  }
  // start of this lane's first segment: the lanes before it applied to zero
  float run = __shfl_up_sync(0xffffffffu, Bc, 1);
  if (lane == 0) run = 0.f;
  for (int g0 = p0; g0 < p1; g0 += G) {
    float a[G], loc[G];
#pragma unroll
    for (int u = 0; u < G; ++u) {
      const size_t i = static_cast<size_t>(min(g0 + u, p1 - 1)) * Hc;
      a[u] = rt[i];
      loc[u] = st[i];
    }
#pragma unroll
    for (int u = 0; u < G; ++u) {
      if (g0 + u < p1) {
        st[static_cast<size_t>(g0 + u) * Hc] = run;
        run = fmaf(expf(-a[u]), run, loc[u]);
      }
    }
  }
}

size_t tdc_workspace_bytes(int B, int T, int Hc) {
  const size_t n_seg = (static_cast<size_t>(T) + kTdcSeg - 1) / kTdcSeg;
  return 2 * static_cast<size_t>(B) * n_seg * Hc * sizeof(float);
}

cudaError_t launch_tdc(const float *s, const float *u, float *h, int B, int T, int Hc, void *ws, cudaStream_t stream) {
  const int n_seg = (T + kTdcSeg - 1) / kTdcSeg;
  float *state = static_cast<float *>(ws);
  float *rate = state + static_cast<size_t>(B) * n_seg * Hc;
  const int threads = min(256, ((Hc + 31) / 32) * 32);
  const dim3 grid(n_seg, B);
  tdc_seg_kernel<0><<<grid, threads, 0, stream>>>(s, u, h, T, Hc, state, rate);
  tdc_combine_kernel<<<(B * Hc + 7) / 8, 256, 0, stream>>>(B, n_seg, Hc, state, rate);
  tdc_seg_kernel<1><<<grid, threads, 0, stream>>>(s, u, h, T, Hc, state, rate);
  return cudaGetLastError();
}

}  // namespace fem
