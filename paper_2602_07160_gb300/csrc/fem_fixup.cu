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
// 256-thread block takes a chunk at a time, claimed from a counter so that
// blocks that drew cheap chunks take more of them: it stages the tile's
// K and V rows k0 .. k0+r_max and the chunk's 8 query rows in shared memory,
// scores the 8 rows against the keys with warp-level bf16 MMAs (16 keys per
// warp, fp32 accumulation), then each warp completes one entry: its lanes
// take four keys each and reduce
// the row's log-sum-exp and, channel by channel, each listed channel's with
// warp shuffles; a 32-channel group with three or more listed channels is
// done with lane = channel instead, walking the keys in turn.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

constexpr int kFixChunk = 8;                // entries per chunk = warps per block

// The entry's output: F itself, or for the one-pass gated read
// g (mu + lambda (F - mu)) with the mu the tensor-core kernel left aside.
__device__ __forceinline__ float fix_gated(const TcGate &gate, size_t o, float F) {
  if (!gate.lam) return F;
  const float mu = gate.mu_side[o];
  return gate.g[o] * fmaf(gate.lam[o], F - mu, mu);
}
constexpr int kFixThreads = 32 * kFixChunk;

__device__ __forceinline__ float warp_max(float x) {
  for (int off = 16; off; off >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, off));
  return x;
}

__device__ __forceinline__ float warp_sum(float x) {
  for (int off = 16; off; off >>= 1) x += __shfl_xor_sync(0xffffffffu, x, off);
  return x;
}

// Four 8x8 bf16 matrices from shared memory (lane l gives the address of row
// l % 8 of matrix l / 8), in the mma fragment layout.
__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}

// c += A (16x16, row-major) B (16x8, column-major), bf16 in, fp32 accumulate.
__device__ __forceinline__ void mma_bf16_16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Asynchronous global -> shared copies (16 bytes: both addresses 16-byte
// aligned; 4 bytes: both 4-byte aligned), so that every staged row is in
// flight at once.
__device__ __forceinline__ void fix_cp16(uint32_t dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void fix_cp4(uint32_t dst, const void *src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void fix_cp_wait_all() {
  asm volatile("cp.async.commit_group;" ::: "memory");
  asm volatile("cp.async.wait_group 0;" ::: "memory");
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
                                                            int *__restrict__ next_chunk,
                                                            int *__restrict__ last_rows, TcGate gate) {
  // staged row strides in bf16 elements: K and Q rows 16-byte aligned for
  // ldmatrix with consecutive rows four banks apart; V rows an odd number of
  // 32-bit words, so one column read across rows is free of bank conflicts
  constexpr int KS = D + 8, VS = D + 2;
  extern __shared__ __align__(16) uint8_t fix_smem[];
  __nv_bfloat16 *sK = reinterpret_cast<__nv_bfloat16 *>(fix_smem);
  __nv_bfloat16 *sV = sK + kBlockK * KS;
  __nv_bfloat16 *sQ = sV + kBlockK * VS;  // 16 rows (8 entries, 8 unused) of KS
  __shared__ float sS[kFixChunk][kBlockK];  // the chunk's scores, log2 units
  __shared__ int s_nk, s_ch;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n_chunks = *count / kFixChunk;
  if (blockIdx.x == 0 && tid == 0 && last_rows) *last_rows = *rows_listed;
  const float scale = kLog2e * rsqrtf(static_cast<float>(D));
  const int n_kt = (T + kBlockK - 1) / kBlockK;

  for (;;) {
    if (tid == 0) {
      s_ch = atomicAdd(next_chunk, 1);
      s_nk = 0;
    }
    __syncthreads();
    const int ch = s_ch;
    if (ch >= n_chunks) break;
    const FixupEntry ent = entries[ch * kFixChunk + warp];
    const int row0 = entries[ch * kFixChunk].row;  // the chunk's first entry is a real row
    const int bh = row0 / T, h = bh % H;
    const int kt = (row0 % T) / kBlockK, k0 = kt * kBlockK;
    const int r = ent.row >= 0 ? ent.row - bh * T - k0 : -1;  // this warp's row in the tile
    if (lane == 0 && r >= 0) atomicMax(&s_nk, r + 1);
    // the entry's stashed accumulators over the earlier key tiles, the
    // previous tile's shifts and beta, lane l holding channels l + 32 g: loaded
    // now so that they arrive while the chunk's rows are staged and scored
    float a_reg[D / 32], c_reg[D / 32], b_reg[D / 32];
#pragma unroll
    for (int gi = 0; gi < D / 32; ++gi) {
      const int j = lane + 32 * gi;
      const bool listed = r >= 0 && ent.mask[gi];
      a_reg[gi] = listed ? out[static_cast<size_t>(ent.row) * D + j] : 0.f;
      c_reg[gi] = (listed && kt > 0) ? shift[(static_cast<size_t>(bh) * n_kt + kt - 1) * D + j] : 0.f;
      b_reg[gi] = beta[h * D + j];
    }
    __syncthreads();
    const int nk = s_nk;  // keys k0 .. k0+nk-1 serve every row of the chunk
    for (int idx = tid; idx < nk * (D / 8); idx += kFixThreads) {
      const int i = idx / (D / 8), c = idx % (D / 8);
      const size_t g = (static_cast<size_t>(bh) * T + k0 + i) * D + 8 * c;
      fix_cp16(smem_u32(sK + i * KS + 8 * c), k + g);
      const uint32_t dv = smem_u32(sV + i * VS + 8 * c);
#pragma unroll
      for (int w = 0; w < 4; ++w) fix_cp4(dv + 4 * w, v + g + 2 * w);
    }
    for (int idx = tid; idx < kFixChunk * (D / 8); idx += kFixThreads) {
      const int w = idx / (D / 8), c = idx % (D / 8);
      const int erow = entries[ch * kFixChunk + w].row;
      *reinterpret_cast<uint4 *>(sQ + w * KS + 8 * c) =
          erow >= 0 ? *reinterpret_cast<const uint4 *>(q + static_cast<size_t>(erow) * D + 8 * c) : make_uint4(0, 0, 0, 0);
    }
    fix_cp_wait_all();
    __syncthreads();
    // S[8 x nk] = Q K^T: warp w takes keys 16w .. 16w+15 (two n8 blocks) over
    // D/16 k-steps of m16n8k16 (rows 8..15 of A are unused)
    if (16 * warp < nk) {
      float c0[4] = {0.f, 0.f, 0.f, 0.f}, c1[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int ks = 0; ks < D / 16; ++ks) {
        uint32_t a[4], bfr[4];
        ldmatrix_x4(a, smem_u32(sQ + (lane % 16) * KS + 16 * ks + (lane / 16) * 8));
        const int mm = lane / 8;  // matrices: (keys lo, d lo) (keys lo, d hi) (keys hi, d lo) (keys hi, d hi)
        ldmatrix_x4(bfr, smem_u32(sK + (16 * warp + (mm / 2) * 8 + lane % 8) * KS + 16 * ks + (mm % 2) * 8));
        mma_bf16_16816(c0, a, bfr[0], bfr[1]);
        mma_bf16_16816(c1, a, bfr[2], bfr[3]);
      }
      // fragment rows lane/4 (and lane/4 + 8, unused), columns 2 (lane % 4) + {0, 1}
      const int rr = lane / 4, cc = 16 * warp + 2 * (lane % 4);
      sS[rr][cc] = c0[0] * scale;
      sS[rr][cc + 1] = c0[1] * scale;
      sS[rr][cc + 8] = c1[0] * scale;
      sS[rr][cc + 9] = c1[1] * scale;
    }
    __syncthreads();
    if (r >= 0) {
      // scores of keys i = lane + 32u (log2 units), -inf past the row
      float s[kBlockK / 32];
#pragma unroll
      for (int u = 0; u < kBlockK / 32; ++u) {
        const int i = lane + 32 * u;
        s[u] = i <= r ? sS[warp][i] : -INFINITY;
      }
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
      // kernel's state over the earlier key tiles (a_reg, c_reg, b_reg)
#pragma unroll
      for (int gi = 0; gi < D / 32; ++gi) {
        unsigned m = ent.mask[gi];
        if (__popc(m) >= 3) {
          // many listed channels in this group: lane = channel, keys walked in turn
          const int j = 32 * gi + lane;
          const float bl = b_reg[gi] * kLog2e;
          float mj = -INFINITY;
          for (int i = 0; i <= r; ++i) mj = fmaxf(mj, fmaf(bl, __bfloat162float(sV[i * VS + j]), sS[warp][i]));
          float sj = 0.f;
          for (int i = 0; i <= r; ++i) sj += exp2f(fmaf(bl, __bfloat162float(sV[i * VS + j]), sS[warp][i]) - mj);
          if ((m >> lane) & 1u) {
            float pre = -INFINITY;
            if (kt > 0 && a_reg[gi] > 0.f && ent.l_pre > 0.f)
              pre = ent.m_pre + log2f(a_reg[gi]) + (b_reg[gi] * c_reg[gi] - kBankOffset) * kLog2e;
            const float G = lse2_pair(pre, mj + log2f(sj));
            const size_t o = static_cast<size_t>(ent.row) * D + j;
            out[o] = fix_gated(gate, o, (G - L) * kLn2 / b_reg[gi]);
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
            x[u] = i <= r ? fmaf(bl, __bfloat162float(sV[i * VS + j]), s[u]) : -INFINITY;
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
            out[o] = fix_gated(gate, o, (G - L) * kLn2 / bj);
          }
        }
      }
    }
    __syncthreads();  // the staged rows are rewritten by the next chunk
  }
}

cudaError_t launch_fixup(const void *q, const void *k, const void *v, const float *beta, const float *shift,
                         float *out, int H, int T, int d, const FixupEntry *entries, const int *count,
                         const int *rows, int *next_chunk, int *last_rows, const TcGate *gate, int num_sms,
                         cudaStream_t stream) {
  const TcGate g = gate ? *gate : TcGate{nullptr, nullptr, nullptr, nullptr};
  const __nv_bfloat16 *qb = static_cast<const __nv_bfloat16 *>(q), *kb = static_cast<const __nv_bfloat16 *>(k),
                      *vb = static_cast<const __nv_bfloat16 *>(v);
  const int grid = num_sms * 3;
  if (d == 64) {
    const size_t smem = (kBlockK * (64 + 8) + kBlockK * (64 + 2) + 16 * (64 + 8)) * sizeof(__nv_bfloat16);
    fixup_kernel<64><<<grid, kFixThreads, smem, stream>>>(qb, kb, vb, beta, shift, out, H, T, entries, count, rows,
                                                          next_chunk, last_rows, g);
  } else if (d == 128) {
    const size_t smem = (kBlockK * (128 + 8) + kBlockK * (128 + 2) + 16 * (128 + 8)) * sizeof(__nv_bfloat16);
    cudaError_t e = cudaFuncSetAttribute(fixup_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    fixup_kernel<128><<<grid, kFixThreads, smem, stream>>>(qb, kb, vb, beta, shift, out, H, T, entries, count, rows,
                                                           next_chunk, last_rows, g);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace fem
