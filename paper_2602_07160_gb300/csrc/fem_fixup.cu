// Exact fp32 recompute of the (row, channel) entries listed by the pre-pass.
//
// These are causal rows of a diagonal tile whose visible values all lie far
// below the tile's shared bank shift (the shift includes keys the row cannot
// see).  For each listed row t and channel j the kernel evaluates the read's
// definition directly,
//   o_{t,j} = (LSE_i(s_{t,i} + beta_j v_{i,j}) - LSE_i s_{t,i}) / beta_j,
// each log-sum-exp stabilised by its own maximum (App. E, "Numerical
// stability"), in base 2 with fp32 accumulation.  Listed channels always have
// beta_j * (spread of their tilt) > kHazardTilt, so beta_j is large enough that
// the difference of the two LSEs loses nothing in fp32.
//
// One 512-thread block per listed row (persistent grid).  Keys are taken in
// chunks of kChunk: the block forms the chunk's scores s_i * log2(e) in shared
// memory (four threads per key) and stages the chunk's values there (rows
// padded by one 32-bit word so a column read is free of bank conflicts).
// The row's own LSE is folded by a block reduction.  Then the listed channels
// are dealt round-robin to the 16 warps; for each one the warp's lanes walk the
// chunk's keys and fold max and sum of 2^(s_i log2e + beta_j v_ij log2e) into
// the channel's running (max, sum) kept in shared memory.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

constexpr int kFixThreads = 512;
constexpr int kFixWarps = kFixThreads / 32;
constexpr int kChunk = 128;
constexpr int kVStride = 128 + 2;  // staged row stride in bf16 elements (d <= 128)

// (m, s) <- (m, s) (+) (m2, s2) for sums of 2^(x - m)
__device__ __forceinline__ void lse2_merge(float &m, float &s, float m2, float s2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) {
    m = m2;
    s = s2;
    return;
  }
  const float mm = fmaxf(m, m2);
  s = s * ex2_approx(m - mm) + s2 * ex2_approx(m2 - mm);
  m = mm;
}

__device__ __forceinline__ float warp_max(float x) {
  for (int off = 16; off; off >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, off));
  return x;
}

__device__ __forceinline__ float warp_sum(float x) {
  for (int off = 16; off; off >>= 1) x += __shfl_xor_sync(0xffffffffu, x, off);
  return x;
}

template <int D>
__global__ void __launch_bounds__(kFixThreads) fixup_kernel(const __nv_bfloat16 *__restrict__ q,
                                                            const __nv_bfloat16 *__restrict__ k,
                                                            const __nv_bfloat16 *__restrict__ v,
                                                            const float *__restrict__ beta, float *__restrict__ out,
                                                            int H, int T, const FixupEntry *__restrict__ entries,
                                                            const int *__restrict__ count, int *__restrict__ last_count) {
  constexpr int CPR = D / 8;                  // 16-byte chunks per row
  constexpr int RPP = kFixThreads / CPR;      // rows staged per pass
  constexpr int NPASS = kChunk / RPP;         // staging passes per chunk
  constexpr int KQ = D / 4 / 8;               // 16-byte chunks of a key quarter
  __shared__ float s_q[D];
  __shared__ float s_s[kChunk];                        // scores of the chunk, log2 units
  __shared__ __align__(16) uint32_t s_v[kChunk * kVStride / 2];  // values of the chunk, padded rows
  __shared__ float s_cm[D], s_cs[D];                   // running (max, sum) of each listed channel
  __shared__ float s_lm, s_ls;                         // the row's running (max, sum) of scores
  __shared__ int s_list[D], s_nlist;                   // listed channels of the row
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n = *count;
  if (blockIdx.x == 0 && tid == 0 && last_count) *last_count = n;
  const float scale = kLog2e * rsqrtf(static_cast<float>(D));
  const __nv_bfloat16 *sv = reinterpret_cast<const __nv_bfloat16 *>(s_v);

  for (int e = blockIdx.x; e < n; e += gridDim.x) {
    const FixupEntry ent = entries[e];
    const int row = ent.row;
    const int bh = row / T, t = row % T, h = bh % H;
    const __nv_bfloat16 *kb = k + static_cast<size_t>(bh) * T * D;
    const __nv_bfloat16 *vb = v + static_cast<size_t>(bh) * T * D;
    if (tid < D) {
      s_q[tid] = __bfloat162float(q[static_cast<size_t>(row) * D + tid]);
      s_cm[tid] = -INFINITY;
      s_cs[tid] = 0.f;
    }
    if (warp == 0) {
      // compact the listed channels in order
      int nl = 0;
#pragma unroll
      for (int g = 0; g < D / 32; ++g) {
        const unsigned m = ent.mask[g];
        if ((m >> lane) & 1u) s_list[nl + __popc(m & ((1u << lane) - 1u))] = 32 * g + lane;
        nl += __popc(m);
      }
      if (lane == 0) {
        s_nlist = nl;
        s_lm = -INFINITY;
        s_ls = 0.f;
      }
    }
    __syncthreads();
    const int nlist = s_nlist;

    for (int kc = 0; kc <= t; kc += kChunk) {
      const int nkeys = min(kChunk, t + 1 - kc);
      // every global load of the chunk in flight at once: the key quarter this
      // thread scores and the value chunks it stages
      const int si = tid >> 2, part = tid & 3;
      uint4 kraw[KQ];
#pragma unroll
      for (int c = 0; c < KQ; ++c)
        kraw[c] = si < nkeys
                      ? reinterpret_cast<const uint4 *>(kb + static_cast<size_t>(kc + si) * D + part * (D / 4))[c]
                      : make_uint4(0, 0, 0, 0);
      uint4 vraw[NPASS];
#pragma unroll
      for (int u = 0; u < NPASS; ++u) {
        const int r = tid / CPR + u * RPP;
        vraw[u] = r < nkeys ? reinterpret_cast<const uint4 *>(vb + static_cast<size_t>(kc + r) * D)[tid % CPR]
                            : make_uint4(0, 0, 0, 0);
      }
      float acc = 0.f;
#pragma unroll
      for (int c = 0; c < KQ; ++c) {
        const __nv_bfloat162 *p2 = reinterpret_cast<const __nv_bfloat162 *>(&kraw[c]);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const float2 f = __bfloat1622float2(p2[u]);
          const int cq = part * (D / 4) + c * 8 + 2 * u;
          acc = fmaf(s_q[cq], f.x, acc);
          acc = fmaf(s_q[cq + 1], f.y, acc);
        }
      }
      acc += __shfl_xor_sync(0xffffffffu, acc, 1);
      acc += __shfl_xor_sync(0xffffffffu, acc, 2);
      if (part == 0 && si < nkeys) s_s[si] = acc * scale;
#pragma unroll
      for (int u = 0; u < NPASS; ++u) {
        uint32_t *dst = s_v + ((tid / CPR + u * RPP) * kVStride) / 2 + (tid % CPR) * 4;
        dst[0] = vraw[u].x;
        dst[1] = vraw[u].y;
        dst[2] = vraw[u].z;
        dst[3] = vraw[u].w;
      }
      __syncthreads();
      // the row's score LSE over the chunk
      if (warp == 0) {
        float mx = -INFINITY;
        for (int i = lane; i < nkeys; i += 32) mx = fmaxf(mx, s_s[i]);
        mx = warp_max(mx);
        float sm = 0.f;
        for (int i = lane; i < nkeys; i += 32) sm += ex2_approx(s_s[i] - mx);
        sm = warp_sum(sm);
        if (lane == 0) {
          float m = s_lm, s = s_ls;
          lse2_merge(m, s, mx, sm);
          s_lm = m;
          s_ls = s;
        }
      }
      // the tilted LSE of each listed channel over the chunk
      for (int li = warp; li < nlist; li += kFixWarps) {
        const int j = s_list[li];
        const float bl = beta[h * D + j] * kLog2e;
        float a[kChunk / 32];
        float mx = -INFINITY;
#pragma unroll
        for (int u = 0; u < kChunk / 32; ++u) {
          const int i = lane + 32 * u;
          a[u] = i < nkeys ? fmaf(bl, __bfloat162float(sv[i * kVStride + j]), s_s[i]) : -INFINITY;
          mx = fmaxf(mx, a[u]);
        }
        mx = warp_max(mx);
        float sm = 0.f;
#pragma unroll
        for (int u = 0; u < kChunk / 32; ++u) sm += a[u] == -INFINITY ? 0.f : ex2_approx(a[u] - mx);
        sm = warp_sum(sm);
        if (lane == 0) {
          float m = s_cm[j], s = s_cs[j];
          lse2_merge(m, s, mx, sm);
          s_cm[j] = m;
          s_cs[j] = s;
        }
      }
      __syncthreads();
    }
    // o = (G - L) / beta for the listed channels
    for (int li = tid; li < nlist; li += kFixThreads) {
      const int j = s_list[li];
      const float G2 = s_cm[j] + log2f(s_cs[j]);  // log2 of sum_i 2^(s_i log2e + beta v log2e)
      const float L2 = s_lm + log2f(s_ls);        // log2 of sum_i 2^(s_i log2e)
      out[static_cast<size_t>(row) * D + j] = (G2 - L2) * kLn2 / beta[h * D + j];
    }
    __syncthreads();
  }
}

cudaError_t launch_fixup(const void *q, const void *k, const void *v, const float *beta, float *out, int H, int T,
                         int d, const FixupEntry *entries, const int *count, int *last_count, int num_sms,
                         cudaStream_t stream) {
  const __nv_bfloat16 *qb = static_cast<const __nv_bfloat16 *>(q), *kb = static_cast<const __nv_bfloat16 *>(k),
                      *vb = static_cast<const __nv_bfloat16 *>(v);
  if (d == 64)
    fixup_kernel<64><<<num_sms * 3, kFixThreads, 0, stream>>>(qb, kb, vb, beta, out, H, T, entries, count, last_count);
  else if (d == 128)
    fixup_kernel<128><<<num_sms * 3, kFixThreads, 0, stream>>>(qb, kb, vb, beta, out, H, T, entries, count, last_count);
  else
    return cudaErrorInvalidValue;
  return cudaGetLastError();
}

}  // namespace fem
