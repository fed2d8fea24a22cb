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
// Entries come in chunks of 8 consecutive rows of one diagonal tile (the
// pre-pass pads each tile's entries to a multiple of 8 with rows -1).  One
// 256-thread block takes a chunk at a time (grid-stride): it stages the tile's
// K and V rows k0 .. k0+r_max in shared memory (rows padded by one 32-bit
// word, so reading one column across rows is free of bank conflicts), then
// each warp completes one entry: its lanes score four keys each and reduce
// the row's log-sum-exp and, channel by channel, each listed channel's with
// warp shuffles; a 32-channel group with three or more listed channels is
// done with lane = channel instead, walking the keys in turn.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

constexpr int kFixChunk = 8;                // entries per chunk = warps per block
constexpr int kFixThreads = 32 * kFixChunk;

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
                                                            const int *__restrict__ count,
                                                            const int *__restrict__ rows_listed,
                                                            int *__restrict__ last_rows) {
  constexpr int KS = D + 2;  // staged row stride in bf16 elements (an odd number of 32-bit words)
  extern __shared__ __align__(16) uint8_t fix_smem[];
  __nv_bfloat16 *sK = reinterpret_cast<__nv_bfloat16 *>(fix_smem);
  __nv_bfloat16 *sV = sK + kBlockK * KS;
  __shared__ float sQ[kFixChunk][D];
  __shared__ float sS[kFixChunk][kBlockK];  // each warp's row scores, for the channel-parallel form
  __shared__ int s_nk;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n_chunks = *count / kFixChunk;
  if (blockIdx.x == 0 && tid == 0 && last_rows) *last_rows = *rows_listed;
  const float scale = kLog2e * rsqrtf(static_cast<float>(D));
  const int n_kt = (T + kBlockK - 1) / kBlockK;

  for (int ch = blockIdx.x; ch < n_chunks; ch += gridDim.x) {
    const FixupEntry ent = entries[ch * kFixChunk + warp];
    const int row0 = entries[ch * kFixChunk].row;  // the chunk's first entry is a real row
    const int bh = row0 / T, h = bh % H;
    const int kt = (row0 % T) / kBlockK, k0 = kt * kBlockK;
    const int r = ent.row >= 0 ? ent.row - bh * T - k0 : -1;  // this warp's row in the tile
    if (tid == 0) s_nk = 0;
    __syncthreads();
    if (lane == 0 && r >= 0) atomicMax(&s_nk, r + 1);
    __syncthreads();
    const int nk = s_nk;  // keys k0 .. k0+nk-1 serve every row of the chunk
    for (int idx = tid; idx < nk * (D / 8); idx += kFixThreads) {
      const int i = idx / (D / 8), c = idx % (D / 8);
      const size_t g = (static_cast<size_t>(bh) * T + k0 + i) * D + 8 * c;
      const uint4 kr = *reinterpret_cast<const uint4 *>(k + g);
      const uint4 vr = *reinterpret_cast<const uint4 *>(v + g);
      uint32_t *dk = reinterpret_cast<uint32_t *>(sK + i * KS + 8 * c);
      uint32_t *dv = reinterpret_cast<uint32_t *>(sV + i * KS + 8 * c);
      dk[0] = kr.x;
      dk[1] = kr.y;
      dk[2] = kr.z;
      dk[3] = kr.w;
      dv[0] = vr.x;
      dv[1] = vr.y;
      dv[2] = vr.z;
      dv[3] = vr.w;
    }
    if (r >= 0)
      for (int d = lane; d < D; d += 32) sQ[warp][d] = __bfloat162float(q[static_cast<size_t>(ent.row) * D + d]);
    __syncthreads();
    if (r >= 0) {
      // scores of keys i = lane + 32u (log2 units), -inf past the row
      float s[kBlockK / 32];
#pragma unroll
      for (int u = 0; u < kBlockK / 32; ++u) {
        const int i = lane + 32 * u;
        float acc = -INFINITY;
        if (i <= r) {
          acc = 0.f;
          const __nv_bfloat162 *kr = reinterpret_cast<const __nv_bfloat162 *>(sK + i * KS);
          const float2 *qr = reinterpret_cast<const float2 *>(sQ[warp]);
#pragma unroll 8
          for (int d2 = 0; d2 < D / 2; ++d2) {
            const float2 kf = __bfloat1622float2(kr[d2]);
            const float2 qf = qr[d2];
            acc = fmaf(qf.x, kf.x, acc);
            acc = fmaf(qf.y, kf.y, acc);
          }
          acc *= scale;
        }
        s[u] = acc;
      }
#pragma unroll
      for (int u = 0; u < kBlockK / 32; ++u) sS[warp][lane + 32 * u] = s[u];
      __syncwarp();
      // the row's score log-sum-exp over all its keys
      float mx = s[0];
#pragma unroll
      for (int u = 1; u < kBlockK / 32; ++u) mx = fmaxf(mx, s[u]);
      mx = warp_max(mx);
      float sm = 0.f;
#pragma unroll
      for (int u = 0; u < kBlockK / 32; ++u) sm += s[u] == -INFINITY ? 0.f : exp2f(s[u] - mx);
      sm = warp_sum(sm);
      const float L = lse2_pair(ent.l_pre > 0.f ? ent.m_pre + log2f(ent.l_pre) : -INFINITY, mx + log2f(sm));
      // each listed channel's tilted log-sum-exp, merged with the tensor-core
      // kernel's state over the earlier key tiles: the row's stashed
      // accumulators, the previous tile's shifts and beta, lane l holding
      // channels l + 32 g, all loaded at once
      float a_reg[D / 32], c_reg[D / 32], b_reg[D / 32];
#pragma unroll
      for (int gi = 0; gi < D / 32; ++gi) {
        const int j = lane + 32 * gi;
        a_reg[gi] = ent.mask[gi] ? out[static_cast<size_t>(ent.row) * D + j] : 0.f;
        c_reg[gi] = (ent.mask[gi] && kt > 0) ? shift[(static_cast<size_t>(bh) * n_kt + kt - 1) * D + j] : 0.f;
        b_reg[gi] = beta[h * D + j];
      }
#pragma unroll
      for (int gi = 0; gi < D / 32; ++gi) {
        unsigned m = ent.mask[gi];
        if (__popc(m) >= 3) {
          // many listed channels in this group: lane = channel, keys walked in turn
          const int j = 32 * gi + lane;
          const float bl = b_reg[gi] * kLog2e;
          float mj = -INFINITY;
          for (int i = 0; i <= r; ++i) mj = fmaxf(mj, fmaf(bl, __bfloat162float(sV[i * KS + j]), sS[warp][i]));
          float sj = 0.f;
          for (int i = 0; i <= r; ++i) sj += exp2f(fmaf(bl, __bfloat162float(sV[i * KS + j]), sS[warp][i]) - mj);
          if ((m >> lane) & 1u) {
            float pre = -INFINITY;
            if (kt > 0 && a_reg[gi] > 0.f && ent.l_pre > 0.f)
              pre = ent.m_pre + log2f(a_reg[gi]) + (b_reg[gi] * c_reg[gi] - kBankOffset) * kLog2e;
            const float G = lse2_pair(pre, mj + log2f(sj));
            out[static_cast<size_t>(ent.row) * D + j] = (G - L) * kLn2 / b_reg[gi];
          }
          m = 0;
        }
        while (m) {
          const int jl = __ffs(m) - 1, j = 32 * gi + jl;
          m &= m - 1;
          const float bj = __shfl_sync(0xffffffffu, b_reg[gi], jl);
          const float a = __shfl_sync(0xffffffffu, a_reg[gi], jl);  // accumulator over the earlier key tiles
          const float c = __shfl_sync(0xffffffffu, c_reg[gi], jl);
          const size_t o = static_cast<size_t>(ent.row) * D + j;
          const float bl = bj * kLog2e;
          float x[kBlockK / 32];
          float mj = -INFINITY;
#pragma unroll
          for (int u = 0; u < kBlockK / 32; ++u) {
            const int i = lane + 32 * u;
            x[u] = i <= r ? fmaf(bl, __bfloat162float(sV[i * KS + j]), s[u]) : -INFINITY;
            mj = fmaxf(mj, x[u]);
          }
          mj = warp_max(mj);
          float sj = 0.f;
#pragma unroll
          for (int u = 0; u < kBlockK / 32; ++u) sj += x[u] == -INFINITY ? 0.f : exp2f(x[u] - mj);
          sj = warp_sum(sj);
          if (lane == 0) {
            float pre = -INFINITY;
            if (kt > 0 && a > 0.f && ent.l_pre > 0.f) pre = ent.m_pre + log2f(a) + (bj * c - kBankOffset) * kLog2e;
            const float G = lse2_pair(pre, mj + log2f(sj));
            out[o] = (G - L) * kLn2 / bj;
          }
        }
      }
    }
    __syncthreads();  // the staged rows are rewritten by the next chunk
  }
}

cudaError_t launch_fixup(const void *q, const void *k, const void *v, const float *beta, const float *shift,
                         float *out, int H, int T, int d, const FixupEntry *entries, const int *count,
                         const int *rows, int *last_rows, int num_sms, cudaStream_t stream) {
  const __nv_bfloat16 *qb = static_cast<const __nv_bfloat16 *>(q), *kb = static_cast<const __nv_bfloat16 *>(k),
                      *vb = static_cast<const __nv_bfloat16 *>(v);
  const int grid = num_sms * 3;
  if (d == 64) {
    const size_t smem = 2 * kBlockK * (64 + 2) * sizeof(__nv_bfloat16);
    fixup_kernel<64><<<grid, kFixThreads, smem, stream>>>(qb, kb, vb, beta, shift, out, H, T, entries, count, rows,
                                                          last_rows);
  } else if (d == 128) {
    const size_t smem = 2 * kBlockK * (128 + 2) * sizeof(__nv_bfloat16);
    cudaError_t e = cudaFuncSetAttribute(fixup_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    fixup_kernel<128><<<grid, kFixThreads, smem, stream>>>(qb, kb, vb, beta, shift, out, H, T, entries, count, rows,
                                                           last_rows);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace fem
