// Value-statistics pre-pass of the FEM read (one read of V).
//
// For every (b, h) and channel j it produces
//   * ChanInfo: the channel's bank mode and the linear bank's anchor, from the
//     minimum, maximum and mean of v_.j over the valid keys;
//   * cpre[b,h,kt,j]: the running maximum of v_.j over key tiles 0..kt.  The
//     main kernel raises the shifted bank's per-channel shift c_j along this
//     schedule, so masked keys (beyond the last row a tile serves, or >= T)
//     never enter c_j.  This is the per-channel LSE stabilisation of App. E
//     ("Numerical stability"), made online;
//   * causal only: the rows of each diagonal tile whose visible maximum lies
//     so far below that tile's shift that the fp16 bank cannot represent them
//     (beta_j * (cpre - visible max) > kHazardTilt).  They are appended to a
//     list that the exact fix-up kernel recomputes.
//
// Block = 32 channels x 8 key groups of 16 keys; grid = (B*H, ceil(d/32)).
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

__global__ void __launch_bounds__(256) value_stats_kernel(const __nv_bfloat16 *__restrict__ v,
                                                           const float *__restrict__ beta, int H, int T, int d,
                                                           int causal, ChanInfo *__restrict__ chan,
                                                           float *__restrict__ cpre,
                                                           FixupEntry *__restrict__ fixups,
                                                           int *__restrict__ fixup_count) {
  constexpr int kGroups = 8, kPer = kBlockK / kGroups;  // 16 keys per thread per tile
  __shared__ float s_max[kGroups][32];
  __shared__ float s_min[kGroups][32];
  __shared__ float s_sum[kGroups][32];
  __shared__ int s_first[kGroups][32];
  __shared__ int s_hz[32];

  const int x = threadIdx.x, y = threadIdx.y;
  const int bh = blockIdx.x, g = blockIdx.y;
  const int h = bh % H;
  const int ch = g * 32 + x;
  const bool ch_ok = ch < d;
  const float b = ch_ok ? beta[h * d + ch] : 0.f;
  const __nv_bfloat16 *vb = v + static_cast<size_t>(bh) * T * d;
  const int n_kt = (T + kBlockK - 1) / kBlockK;

  float run_c = -INFINITY;  // running max over tiles (all threads keep it)
  float gmax = -INFINITY, gmin = INFINITY, gsum = 0.f;

  for (int kt = 0; kt < n_kt; ++kt) {
    const int k0 = kt * kBlockK + y * kPer;
    float vals[kPer];
    float lmax = -INFINITY, lmin = INFINITY, lsum = 0.f;
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      const int key = k0 + i;
      float val = -INFINITY;
      if (ch_ok && key < T) {
        val = __bfloat162float(vb[static_cast<size_t>(key) * d + ch]);
        lmin = fminf(lmin, val);
        lsum += val;
      }
      vals[i] = val;
      lmax = fmaxf(lmax, val);
    }
    s_max[y][x] = lmax;
    s_min[y][x] = lmin;
    s_sum[y][x] = lsum;
    __syncthreads();
    float tmax = -INFINITY, tmin = INFINITY;
#pragma unroll
    for (int yy = 0; yy < kGroups; ++yy) {
      tmax = fmaxf(tmax, s_max[yy][x]);
      tmin = fminf(tmin, s_min[yy][x]);
      gsum += s_sum[yy][x];
    }
    const float c_old = run_c;
    run_c = fmaxf(run_c, tmax);
    gmax = fmaxf(gmax, tmax);
    gmin = fminf(gmin, tmin);
    if (y == 0 && ch_ok) cpre[(static_cast<size_t>(bh) * n_kt + kt) * d + ch] = run_c;

    if (causal) {
      // Exclusive prefix maximum before this thread's 16 keys, then the first
      // key at which the visible maximum comes within kHazardTilt/beta of the
      // tile's shift.  Rows of the tile before that key are hazardous.
      float run = c_old;
      for (int yy = 0; yy < y; ++yy) run = fmaxf(run, s_max[yy][x]);
      int first = kBlockK;
#pragma unroll
      for (int i = 0; i < kPer; ++i) {
        run = fmaxf(run, vals[i]);
        if (first == kBlockK && vals[i] != -INFINITY && b * (run_c - run) <= kHazardTilt) first = y * kPer + i;
      }
      s_first[y][x] = first;
      __syncthreads();
      if (y == 0) {
        int hz = kBlockK;
        for (int yy = 0; yy < kGroups; ++yy) hz = min(hz, s_first[yy][x]);
        if (!ch_ok || hz == kBlockK) hz = 0;  // no valid key: nothing to fix
        s_hz[x] = hz;
      }
      __syncthreads();
      if (y == 0) {
        // Rows r < hz_j of this tile need channel j recomputed.  Warp 0 of the
        // block appends one entry per hazardous row with the channel mask.
        int hz_max = s_hz[x];
        for (int off = 16; off; off >>= 1) hz_max = max(hz_max, __shfl_xor_sync(0xffffffffu, hz_max, off));
        const int t0 = kt * kBlockQ;
        const int n_rows = min(hz_max, T - t0);
        if (n_rows > 0) {
          int base = 0;
          if (x == 0) base = atomicAdd(fixup_count, n_rows);
          base = __shfl_sync(0xffffffffu, base, 0);
          for (int r = x; r < n_rows; r += 32) {
            unsigned mask = 0;
            for (int c = 0; c < 32; ++c) mask |= (s_hz[c] > r ? 1u : 0u) << c;
            FixupEntry e;
            e.row = bh * T + t0 + r;
            e.group = g;
            e.mask = mask;
            e.pad = 0;
            fixups[base + r] = e;
          }
        }
      }
    }
    __syncthreads();
  }
  if (y == 0 && ch_ok) {
    ChanInfo ci;
    const float mean = gsum / static_cast<float>(T);
    if (b > 0.f) {
      const float hi = gmin + kLinearLowTilt / b;
      const float lo = gmax - log1pf(kLinearBankMax * b) / b;
      ci.linear = lo <= hi ? 1.f : 0.f;
      ci.c_lin = fminf(fmaxf(mean, lo), hi);
    } else {
      ci.linear = 1.f;
      ci.c_lin = mean;
    }
    chan[bh * d + ch] = ci;
  }
}

cudaError_t launch_value_stats(const void *v, const float *beta, int BH, int H, int T, int d, int causal,
                               ChanInfo *chan, float *cpre, FixupEntry *fixups, int *fixup_count,
                               cudaStream_t stream) {
  const dim3 grid(BH, (d + 31) / 32), block(32, 8);
  value_stats_kernel<<<grid, block, 0, stream>>>(static_cast<const __nv_bfloat16 *>(v), beta, H, T, d, causal, chan,
                                                 cpre, fixups, fixup_count);
  return cudaGetLastError();
}

}  // namespace fem
