// Exact fp32 recompute of the (row, channel) entries listed by the pre-pass.
//
// These are causal rows of a diagonal tile whose visible values all lie far
// below the tile's shared bank shift (the shift includes keys the row cannot
// see).  For each entry the kernel evaluates the read's definition directly,
//   o_{t,j} = (LSE_i(s_{t,i} + beta_j v_{i,j}) - LSE_i s_{t,i}) / beta_j,
// with both log-sum-exps kept online in fp32, each stabilised by its own
// running maximum (App. E, "Numerical stability").  Listed channels always
// have beta_j * (spread of their tilt) > kHazardTilt, so beta_j is large
// enough that the difference of the two LSEs loses nothing in fp32.
//
// Persistent grid; one 128-thread block per entry at a time.  Scores are
// formed 128 keys at a time (thread per key), then each warp folds 32 keys of
// the chunk into per-channel partial LSEs (lane per channel); the four warps
// are merged at the end.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

__device__ __forceinline__ void lse_push(float &m, float &s, float a) {
  if (a == -INFINITY) return;
  if (a > m) {
    s = s * expf(m - a) + 1.f;
    m = a;
  } else {
    s += expf(a - m);
  }
}

__device__ __forceinline__ void lse_merge(float &m, float &s, float m2, float s2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) {
    m = m2;
    s = s2;
    return;
  }
  const float mm = fmaxf(m, m2);
  s = s * expf(m - mm) + s2 * expf(m2 - mm);
  m = mm;
}

__global__ void __launch_bounds__(128) fixup_kernel(const __nv_bfloat16 *__restrict__ q,
                                                     const __nv_bfloat16 *__restrict__ k,
                                                     const __nv_bfloat16 *__restrict__ v,
                                                     const float *__restrict__ beta, float *__restrict__ out, int H,
                                                     int T, int d, const FixupEntry *__restrict__ entries,
                                                     const int *__restrict__ count, int *__restrict__ last_count) {
  __shared__ float s_q[256];
  __shared__ float s_s[128];
  __shared__ float s_pm[4][32], s_ps[4][32], s_lm[4][32], s_ls[4][32];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n = *count;
  if (blockIdx.x == 0 && tid == 0 && last_count) *last_count = n;
  const float inv_sqrt_d = rsqrtf(static_cast<float>(d));

  for (int e = blockIdx.x; e < n; e += gridDim.x) {
    const FixupEntry ent = entries[e];
    const int row = ent.row;
    const int bh = row / T, t = row % T, h = bh % H;
    const int ch = ent.group * 32 + lane;
    const bool active = ch < d && ((ent.mask >> lane) & 1u);
    const float b = ch < d ? beta[h * d + ch] : 0.f;
    const __nv_bfloat16 *kb = k + static_cast<size_t>(bh) * T * d;
    const __nv_bfloat16 *vb = v + static_cast<size_t>(bh) * T * d;
    for (int c = tid; c < d; c += 128) s_q[c] = __bfloat162float(q[static_cast<size_t>(row) * d + c]);
    __syncthreads();

    float gm = -INFINITY, gs = 0.f;  // LSE of s + beta v (this warp's keys)
    float lm = -INFINITY, ls = 0.f;  // LSE of s (this warp's keys)
    for (int kc = 0; kc <= t; kc += 128) {
      const int key = kc + tid;
      float sc = -INFINITY;
      if (key <= t) {
        const __nv_bfloat16 *kr = kb + static_cast<size_t>(key) * d;
        float acc = 0.f;
        for (int c = 0; c < d; c += 8) {
          const uint4 raw = *reinterpret_cast<const uint4 *>(kr + c);
          const __nv_bfloat162 *p2 = reinterpret_cast<const __nv_bfloat162 *>(&raw);
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const float2 f = __bfloat1622float2(p2[u]);
            acc = fmaf(s_q[c + 2 * u], f.x, acc);
            acc = fmaf(s_q[c + 2 * u + 1], f.y, acc);
          }
        }
        sc = acc * inv_sqrt_d;
      }
      s_s[tid] = sc;
      __syncthreads();
      for (int i = warp * 32; i < warp * 32 + 32; ++i) {
        const int kk = kc + i;
        if (kk > t) break;
        const float s = s_s[i];
        lse_push(lm, ls, s);
        if (active) lse_push(gm, gs, s + b * __bfloat162float(vb[static_cast<size_t>(kk) * d + ch]));
      }
      __syncthreads();
    }
    s_pm[warp][lane] = gm;
    s_ps[warp][lane] = gs;
    s_lm[warp][lane] = lm;
    s_ls[warp][lane] = ls;
    __syncthreads();
    if (warp == 0) {
      float m1 = s_pm[0][lane], s1 = s_ps[0][lane], m2 = s_lm[0][lane], s2 = s_ls[0][lane];
      for (int w = 1; w < 4; ++w) {
        lse_merge(m1, s1, s_pm[w][lane], s_ps[w][lane]);
        lse_merge(m2, s2, s_lm[w][lane], s_ls[w][lane]);
      }
      if (active) {
        const float G = m1 + logf(s1);
        const float L = m2 + logf(s2);
        out[static_cast<size_t>(row) * d + ch] = (G - L) / b;
      }
    }
    __syncthreads();
  }
}

cudaError_t launch_fixup(const void *q, const void *k, const void *v, const float *beta, float *out, int H, int T,
                         int d, const FixupEntry *entries, const int *count, int *last_count, int num_sms,
                         cudaStream_t stream) {
  fixup_kernel<<<num_sms * 8, 128, 0, stream>>>(static_cast<const __nv_bfloat16 *>(q),
                                                static_cast<const __nv_bfloat16 *>(k),
                                                static_cast<const __nv_bfloat16 *>(v), beta, out, H, T, d, entries,
                                                count, last_count);
  return cudaGetLastError();
}

}  // namespace fem
