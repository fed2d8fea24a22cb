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
#include <cooperative_groups.h>

#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {
namespace cg = cooperative_groups;

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

// ---------------------------------------------------------------------------
// One-launch form for T <= kTdcClusterMaxT: a cluster of n CTAs per (b, 32
// channels), n = 1, 2, 4 or 8 so that a thread has about kTdcSubLen steps, CTA r
// taking the r-th n-th of the time axis, warp w of a CTA the w-th of its 32
// sub-segments, lane = channel (each warp load is one 128-byte step of 32
// channels).  (1) every thread's sub-segment map x -> exp(-S) x + a from zero
// (S its summed rate); (2) warp c scans channel c's 32 maps in order, lane =
// sub-segment, with shuffles (the exclusive prefixes back in shared memory),
// the cluster barrier publishes the CTA's total maps, and warp 0 loads the
// totals of the CTAs before it from their shared memory and composes them into
// the CTA's start state; (3) every thread runs its sub-segment again from its
// start state and writes h.  The second read of s and u finds them in L2.  No
// workspace and one launch instead of three; the maps compose like the combine
// kernel's.
// ---------------------------------------------------------------------------
constexpr int kTdcCtas = 8;           // CTAs per cluster at most (portable cluster size)
constexpr int kTdcSubs = 32;          // sub-segments (warps) per CTA
constexpr int kTdcSubLen = 32;        // steps per sub-segment the cluster size aims at
constexpr int kTdcClusterMaxT = 16384;

__global__ void __launch_bounds__(32 * kTdcSubs, 1)
    tdc_cluster_kernel(const float *__restrict__ s, const float *__restrict__ u, float *__restrict__ h, int T, int Hc,
                       int len_sub) {
  __shared__ float s_S[kTdcSubs][33], s_a[kTdcSubs][33];  // [sub-segment][channel]: maps, then their exclusive prefixes
  __shared__ float s_tot[2][32];                           // the CTA's total map (S, a) per channel
  __shared__ float s_start[32];                            // the state before the CTA's first step
  cg::cluster_group cluster = cg::this_cluster();
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int rank = static_cast<int>(cluster.block_rank());  // the block's part of the time axis
  const int c = static_cast<int>(blockIdx.y) * 32 + lane, b = static_cast<int>(blockIdx.z);
  const bool valid = c < Hc;
  const int t0 = min(T, (rank * kTdcSubs + w) * len_sub), t1 = min(T, t0 + len_sub);
  const size_t base = static_cast<size_t>(b) * T * Hc + c;

  // (1) the sub-segment's map from a zero state; the loads do not depend on the recurrence
  float acc = 0.f, S = 0.f;
  if (valid) {
#pragma unroll 16
    for (int t = t0; t < t1; ++t) {
      const size_t e = base + static_cast<size_t>(t) * Hc;
      const float st = s[e];
      acc = fmaf(ex2_approx(-st * kLog2e), acc, u[e]);
      S += st;
    }
  }
  s_S[w][lane] = S;
  s_a[w][lane] = acc;
  __syncthreads();
  // (2) warp w scans channel w's maps over the sub-segments (lane = sub-segment): an
  // earlier map (Sp, ap) followed by a later one (S, a) is (Sp + S, exp(-S) ap + a)
  {
    float SS = s_S[lane][w], A = s_a[lane][w];
#pragma unroll
    for (int off = 1; off < kTdcSubs; off <<= 1) {
      const float Sp = __shfl_up_sync(0xffffffffu, SS, off), ap = __shfl_up_sync(0xffffffffu, A, off);
      if (lane >= off) {
        A = fmaf(ex2_approx(-SS * kLog2e), ap, A);
        SS += Sp;
      }
    }
    float exS = __shfl_up_sync(0xffffffffu, SS, 1), exA = __shfl_up_sync(0xffffffffu, A, 1);
    if (lane == 0) exS = exA = 0.f;
    s_S[lane][w] = exS;
    s_a[lane][w] = exA;
    if (lane == kTdcSubs - 1) {
      s_tot[0][w] = SS;
      s_tot[1][w] = A;
    }
  }
  cluster.sync();  // every CTA's total maps are in its shared memory
  if (w == 0) {
    float tS[kTdcCtas], tA[kTdcCtas];  // the totals of the CTAs before this one, loaded together
#pragma unroll
    for (int q = 0; q < kTdcCtas; ++q) {
      if (q < rank) {
        const float *tot = cluster.map_shared_rank(&s_tot[0][0], q);
        tS[q] = tot[lane];
        tA[q] = tot[32 + lane];
      }
    }
    float x = 0.f;  // h before step 0 is zero
#pragma unroll
    for (int q = 0; q < kTdcCtas; ++q)
      if (q < rank) x = fmaf(ex2_approx(-tS[q] * kLog2e), x, tA[q]);
    s_start[lane] = x;
  }
  cluster.sync();  // the remote reads are done (no CTA leaves while another reads it); start states ready
  // (3) the sub-segment again from its start state, writing h
  acc = fmaf(ex2_approx(-s_S[w][lane] * kLog2e), s_start[lane], s_a[w][lane]);
  if (valid) {
#pragma unroll 16
    for (int t = t0; t < t1; ++t) {
      const size_t e = base + static_cast<size_t>(t) * Hc;
      acc = fmaf(ex2_approx(-s[e] * kLog2e), acc, u[e]);
      h[e] = acc;
    }
  }
}

bool tdc_one_launch(int B, int T, int Hc) { return T <= kTdcClusterMaxT && (Hc + 31) / 32 <= 65535 && B <= 65535; }

size_t tdc_workspace_bytes(int B, int T, int Hc) {
  if (tdc_one_launch(B, T, Hc)) return 0;
  const size_t n_seg = (static_cast<size_t>(T) + kTdcSeg - 1) / kTdcSeg;
  return 2 * static_cast<size_t>(B) * n_seg * Hc * sizeof(float);
}

cudaError_t launch_tdc(const float *s, const float *u, float *h, int B, int T, int Hc, void *ws, cudaStream_t stream) {
  if (tdc_one_launch(B, T, Hc)) {
    int n = 1;  // CTAs per cluster: the smallest power of two giving sub-segments of at most kTdcSubLen steps
    while (n < kTdcCtas && n * kTdcSubs * kTdcSubLen < T) n *= 2;
    const int len_sub = (T + n * kTdcSubs - 1) / (n * kTdcSubs);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(n, (Hc + 31) / 32, B);
    cfg.blockDim = dim3(32 * kTdcSubs);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = n;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, tdc_cluster_kernel, s, u, h, T, Hc, len_sub);
  }
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
