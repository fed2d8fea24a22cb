// Completion of the (row, channel) entries listed by the pre-pass.
//
// These are rows t of a causal diagonal key tile whose visible values of a
// shifted channel all lie far below the tile's bank shift (the shift includes
// keys the row cannot see), so the bank underflows for them on that tile
// only.  The tensor-core kernel leaves, for each entry, the state over the
// key tiles before the diagonal one: the row's running maximum m and sum l of
// 2^(s' - m) (s' = s log2 e, in the entry), and, in place of each listed
// channel's output, its accumulator
//   a_j = sum_{i < k0} 2^(s'_i - m) exp(beta_j (v_ij - c_j) + kappa),
// c_j the bank shift of tile kt - 1.  This kernel takes the diagonal tile's
// keys k0 .. t exactly in fp32 and merges, in base 2,
//   G_j = log2 sum_{i <= t} 2^(s'_i + beta_j v_ij log2 e)
//       = log2( 2^(m + log2 a_j + (beta_j c_j - kappa) log2 e) + sum_{k0 <= i <= t} 2^(s'_i + beta_j v_ij log2 e) )
//   L   = log2( 2^m l + sum_{k0 <= i <= t} 2^(s'_i) )
// and writes o_tj = (G_j - L) ln 2 / beta_j, the read's definition
// (Sec. 2.3, Eq. "fem-free-energy-main", with the softmax prior of App. C),
// each log-sum-exp stabilised by its own maximum (App. E, "Numerical
// stability").
//
// One 128-thread block per entry (grid-stride over the device-side count):
// thread i scores key k0 + i; the row's diagonal log-sum-exp is one warp
// reduction; the listed channels are dealt round-robin to the four warps,
// whose lanes walk the keys.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

constexpr int kFixThreads = 128;

__device__ __forceinline__ float warp_max(float x) {
  for (int off = 16; off; off >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, off));
  return x;
}

__device__ __forceinline__ float warp_sum(float x) {
  for (int off = 16; off; off >>= 1) x += __shfl_xor_sync(0xffffffffu, x, off);
  return x;
}

// log2(2^a + 2^b) for a, b possibly -inf
__device__ __forceinline__ float lse2_pair(float a, float b) {
  const float mx = fmaxf(a, b);
  if (mx == -INFINITY) return -INFINITY;
  return mx + log2f(exp2f(a - mx) + exp2f(b - mx));
}

template <int D>
__global__ void __launch_bounds__(kFixThreads) fixup_kernel(const __nv_bfloat16 *__restrict__ q,
                                                            const __nv_bfloat16 *__restrict__ k,
                                                            const __nv_bfloat16 *__restrict__ v,
                                                            const float *__restrict__ beta,
                                                            const float *__restrict__ shift, float *__restrict__ out,
                                                            int H, int T, const FixupEntry *__restrict__ entries,
                                                            const int *__restrict__ count, int *__restrict__ last_count) {
  __shared__ float s_q[D];
  __shared__ float s_s[kBlockK];  // diagonal scores, log2 units (-inf past t)
  __shared__ float s_L;           // log2 of the row's score sum over all its keys
  __shared__ int s_list[D], s_nlist;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n = *count;
  if (blockIdx.x == 0 && tid == 0 && last_count) *last_count = n;
  const float scale = kLog2e * rsqrtf(static_cast<float>(D));
  const int n_kt = (T + kBlockK - 1) / kBlockK;

  for (int e = blockIdx.x; e < n; e += gridDim.x) {
    const FixupEntry ent = entries[e];
    const int row = ent.row;
    const int bh = row / T, t = row % T, h = bh % H;
    const int kt = t / kBlockK, k0 = kt * kBlockK, nkeys = t + 1 - k0;
    for (int j = tid; j < D; j += kFixThreads) s_q[j] = __bfloat162float(q[static_cast<size_t>(row) * D + j]);
    if (warp == 0) {
      // compact the listed channels in order
      int nl = 0;
#pragma unroll
      for (int g = 0; g < D / 32; ++g) {
        const unsigned m = ent.mask[g];
        if ((m >> lane) & 1u) s_list[nl + __popc(m & ((1u << lane) - 1u))] = 32 * g + lane;
        nl += __popc(m);
      }
      if (lane == 0) s_nlist = nl;
    }
    __syncthreads();
    // scores of the diagonal keys
    {
      float acc = -INFINITY;
      if (tid < nkeys) {
        const uint4 *kr = reinterpret_cast<const uint4 *>(k + (static_cast<size_t>(bh) * T + k0 + tid) * D);
        uint4 raw[D / 8];
#pragma unroll
        for (int c = 0; c < D / 8; ++c) raw[c] = kr[c];
        acc = 0.f;
#pragma unroll
        for (int c = 0; c < D / 8; ++c) {
          const __nv_bfloat162 *p2 = reinterpret_cast<const __nv_bfloat162 *>(&raw[c]);
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const float2 f = __bfloat1622float2(p2[u]);
            acc = fmaf(s_q[8 * c + 2 * u], f.x, acc);
            acc = fmaf(s_q[8 * c + 2 * u + 1], f.y, acc);
          }
        }
        acc *= scale;
      }
      s_s[tid] = acc;
    }
    __syncthreads();
    if (warp == 0) {
      float x[kBlockK / 32];
      float mx = -INFINITY;
#pragma unroll
      for (int u = 0; u < kBlockK / 32; ++u) {
        x[u] = s_s[lane + 32 * u];
        mx = fmaxf(mx, x[u]);
      }
      mx = warp_max(mx);
      float sm = 0.f;
#pragma unroll
      for (int u = 0; u < kBlockK / 32; ++u) sm += x[u] == -INFINITY ? 0.f : exp2f(x[u] - mx);
      sm = warp_sum(sm);
      if (lane == 0) {
        const float pre = ent.l_pre > 0.f ? ent.m_pre + log2f(ent.l_pre) : -INFINITY;
        s_L = lse2_pair(pre, mx + log2f(sm));
      }
    }
    __syncthreads();
    const int nlist = s_nlist;
    const float L = s_L;
    for (int li = warp; li < nlist; li += kFixThreads / 32) {
      const int j = s_list[li];
      const float bj = beta[h * D + j];
      const float bl = bj * kLog2e;
      float x[kBlockK / 32];
      float mx = -INFINITY;
#pragma unroll
      for (int u = 0; u < kBlockK / 32; ++u) {
        const int i = lane + 32 * u;
        x[u] = i < nkeys ? fmaf(bl, __bfloat162float(v[(static_cast<size_t>(bh) * T + k0 + i) * D + j]), s_s[i])
                         : -INFINITY;
        mx = fmaxf(mx, x[u]);
      }
      mx = warp_max(mx);
      float sm = 0.f;
#pragma unroll
      for (int u = 0; u < kBlockK / 32; ++u) sm += x[u] == -INFINITY ? 0.f : exp2f(x[u] - mx);
      sm = warp_sum(sm);
      if (lane == 0) {
        const size_t o = static_cast<size_t>(row) * D + j;
        const float a = out[o];  // accumulator over the earlier key tiles
        float pre = -INFINITY;
        if (kt > 0 && a > 0.f && ent.l_pre > 0.f) {
          const float c = shift[(static_cast<size_t>(bh) * n_kt + kt - 1) * D + j];
          pre = ent.m_pre + log2f(a) + (bj * c - kBankOffset) * kLog2e;
        }
        const float G = lse2_pair(pre, mx + log2f(sm));
        out[o] = (G - L) * kLn2 / bj;
      }
    }
    __syncthreads();
  }
}

cudaError_t launch_fixup(const void *q, const void *k, const void *v, const float *beta, const float *shift,
                         float *out, int H, int T, int d, const FixupEntry *entries, const int *count, int *last_count,
                         int num_sms, cudaStream_t stream) {
  const __nv_bfloat16 *qb = static_cast<const __nv_bfloat16 *>(q), *kb = static_cast<const __nv_bfloat16 *>(k),
                      *vb = static_cast<const __nv_bfloat16 *>(v);
  const int grid = num_sms * 16;
  if (d == 64)
    fixup_kernel<64><<<grid, kFixThreads, 0, stream>>>(qb, kb, vb, beta, shift, out, H, T, entries, count, last_count);
  else if (d == 128)
    fixup_kernel<128><<<grid, kFixThreads, 0, stream>>>(qb, kb, vb, beta, shift, out, H, T, entries, count,
                                                        last_count);
  else
    return cudaErrorInvalidValue;
  return cudaGetLastError();
}

}  // namespace fem
