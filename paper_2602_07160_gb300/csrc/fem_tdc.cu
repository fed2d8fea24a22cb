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
// so every load and store is coalesced over the channels of a step.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

constexpr int kTdcSeg = 64;  // steps per segment

// MODE 0: local end state and summed rate of a segment; MODE 1: h from the start state.
template <int MODE>
__global__ void tdc_seg_kernel(const float *__restrict__ s, const float *__restrict__ u, float *__restrict__ h, int T,
                               int Hc, float *__restrict__ state, float *__restrict__ rate) {
  const int p = blockIdx.x, n_seg = gridDim.x, b = blockIdx.y;
  const int t0 = p * kTdcSeg, t1 = min(T, t0 + kTdcSeg);
  for (int c = threadIdx.x; c < Hc; c += blockDim.x) {
    const size_t sidx = (static_cast<size_t>(b) * n_seg + p) * Hc + c;
    float acc = MODE == 0 ? 0.f : state[sidx], sum = 0.f;
    // the loads do not depend on the recurrence: eight steps' loads in flight
#pragma unroll 8
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

__global__ void tdc_combine_kernel(int n_seg, int Hc, float *__restrict__ state, const float *__restrict__ rate) {
  const int b = blockIdx.x;
  for (int c = threadIdx.x; c < Hc; c += blockDim.x) {
    float run = 0.f;
    for (int p = 0; p < n_seg; ++p) {
      const size_t sidx = (static_cast<size_t>(b) * n_seg + p) * Hc + c;
      const float loc = state[sidx];
      state[sidx] = run;
      run = fmaf(expf(-rate[sidx]), run, loc);
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
  tdc_combine_kernel<<<B, threads, 0, stream>>>(n_seg, Hc, state, rate);
  tdc_seg_kernel<1><<<grid, threads, 0, stream>>>(s, u, h, T, Hc, state, rate);
  return cudaGetLastError();
}

}  // namespace fem
