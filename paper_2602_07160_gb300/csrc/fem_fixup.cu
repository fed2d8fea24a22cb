// Exact completion of the (row, channel) entries the tensor-core kernel's
// underflow guard rejected.
//
// For an entry of row t (b, h) the kernel restarts the read of the listed
// channels from the entry's key tile kt0 and takes every later key the row
// sees exactly in fp32, the way the fp32 read does: with the row's running
// maximum m of s' = s log2 e, P_i = 2^(s'_i - m), and per channel j a running
// shift c_j (the largest visible value so far) and
//   L   = sum_i P_i
//   A_j = sum_i P_i exp(beta_j (v_ij - c_j))
//   W_j = sum_i P_i expm1(beta_j (v_ij - c_j)) / beta_j   (v_ij - c_j at beta 0)
// The read is then o = c + log1p(beta W / L) / beta when beta W / L > -1/2
// (W is kept for beta < kFixWBeta only), c + log(A / L) / beta otherwise,
// c + W / L at beta = 0: the read's
// definition (Sec. 2.3, Eq. "fem-free-energy-main", with the softmax prior of
// App. C), free of the cancellation in the LSE difference at small beta and
// each sum stabilised by its own maximum (App. E, "Numerical stability").
//
// kt0 > 0: the row's earlier key tiles passed the guard, and the kernel
// starts from the state the tensor-core kernel left before tile kt0 (m, L in
// the entry; channel j's accumulator a_j in out[row][j], over the bank of tile
// kt0 - 1: shifted, A = a e^-kappa at that tile's shift and W = (A - L)/beta;
// linear, W = a at the anchor and A = L + beta W).  kt0 = 0: from nothing.
// The one-pass gated read's entries are gated, o = g (mu + lambda (F - mu)),
// with the mu the tensor-core kernel left aside, or, when the mean bank's own
// guard rejected it (kt0 = 0 and l_pre = 1), with mu recomputed as
// sum_i P_i (v_ij - c0_j) / L + c0_j.
//
// Entries come in chunks of kFixChunk = 8 rows of one query tile with the
// same kt0 (the tensor-core kernel pads each block to a multiple of 8 with
// rows -1).  One 256-thread block (three per SM at d = 128, four at d = 64, their
// register budgets set for it) takes a chunk at a time,
// claimed from a counter (the next claim already in flight while the current
// chunk runs) so that blocks that drew cheap chunks take more of them, and
// walks its key tiles: it stages the chunk's query rows and the tile's K and V
// rows in shared memory with asynchronous copies, scores the 8 rows against
// them with warp-level bf16 MMAs (16 keys per warp, fp32 accumulation), then
// each warp folds the tile into one entry's state: its
// lanes take four keys each for the row's sums and, channel by channel, for
// each listed channel's; a 32-channel group with three or more listed
// channels is folded with lane = channel instead, walking the keys in turn in
// one pass.
//
// At 128 key tiles or more (SPLIT), a chunk that recomputes its rows from the
// first key tile over 2 kseg tiles or more (kseg = fix_seg_tiles) is split: the
// block that draws it registers it in a slot and works through its segments of
// kseg tiles, other blocks take the remaining segments once the list is
// exhausted, each segment leaves the rows' partial states (m, L and per listed
// channel c, A, W, M, all from an empty start) in the slot's pool, and the block
// that finishes the last segment folds them in key order, each scaled to the
// common row maximum and shifted like a key tile's sums, and reads the rows out.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

// Channels with beta below this carry W (the read o = c + log1p(beta W / L) / beta,
// free of cancellation when A / L is near 1); from here on log(A / L) / beta
// loses at most a few fp32 ulps of A / L over beta and W is not needed.
constexpr float kFixWBeta = 0.25f;
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

// expm1(y)/beta for y = beta x <= 0, given e = exp(y): the series of
// expm1(y)/y times x for |y| < 1/2 (truncation below 4e-6 relative), (e - 1)
// times 1/beta beyond; x itself at beta = 0.
__device__ __forceinline__ float em1_over_beta(float x, float y, float e, float rb) {
  if (fabsf(y) < 0.5f) {
    float p = fmaf(y, 1.f / 720.f, 1.f / 120.f);
    p = fmaf(y, p, 1.f / 24.f);
    p = fmaf(y, p, 1.f / 6.f);
    p = fmaf(y, p, 0.5f);
    p = fmaf(y, p, 1.f);
    return x * p;
  }
  return (e - 1.f) * rb;
}

// The running state of one channel moves from shift c to c_new >= c:
// A <- r A, W <- r W + expm1(beta (c - c_new))/beta L with r = exp(beta (c - c_new)).
__device__ __forceinline__ void shift_state(float &c, float &A, float &W, float c_new, float b, float rb, float L) {
  if (!(c_new > c)) return;
  if (c == -INFINITY) {
    A = 0.f;
    W = 0.f;
  } else {
    const float x = c - c_new, y = b * x, e = exp2f(y * kLog2e);
    W = fmaf(e, W, em1_over_beta(x, y, e, rb) * L);
    A *= e;
  }
  c = c_new;
}

// Folds a tile's sums (a, w) over keys of prior mass lt, taken at the tile's
// own shift vt, into the running state (c, A, W) of prior mass L.
__device__ __forceinline__ void fold_tile(float &c, float &A, float &W, float L, float vt, float a, float w, float lt,
                                          float b, float rb) {
  float A2 = a, W2 = w, c2 = vt;
  if (vt >= c) {
    shift_state(c, A, W, vt, b, rb, L);
  } else {
    shift_state(c2, A2, W2, c, b, rb, lt);
  }
  A += A2;
  W += W2;
}

// SPLIT: long recomputations go over key-tile segments (part != null); otherwise
// every chunk runs whole and the kernel carries none of that machinery.
template <int D, bool SPLIT>
__global__ void __launch_bounds__(kFixThreads, D == 64 ? 4 : 3) fixup_kernel(const __nv_bfloat16 *__restrict__ q,
                                                            const __nv_bfloat16 *__restrict__ k,
                                                            const __nv_bfloat16 *__restrict__ v,
                                                            const float *__restrict__ beta,
                                                            const ChanInfo *__restrict__ chan,
                                                            const float *__restrict__ shift, float *__restrict__ out,
                                                            int H, int T, int causal,
                                                            const FixupEntry *__restrict__ entries,
                                                            const int *__restrict__ count,
                                                            const int *__restrict__ rows_listed,
                                                            int *__restrict__ next_chunk,
                                                            int *__restrict__ last_rows, TcGate gate,
                                                            int *__restrict__ fix_long, FixSlot *__restrict__ slots,
                                                            float *__restrict__ part) {
  // staged row strides in bf16 elements: K and Q rows 16-byte aligned for
  // ldmatrix with consecutive rows four banks apart; V rows an odd number of
  // 32-bit words, so one column read across rows is free of bank conflicts
  constexpr int KS = D + 8, VS = D + 2, G = D / 32;
  grid_dep_wait();  // the entry list and the accumulators the tensor-core kernel left in out
  extern __shared__ __align__(16) uint8_t fix_smem[];
  __nv_bfloat16 *sK = reinterpret_cast<__nv_bfloat16 *>(fix_smem);
  __nv_bfloat16 *sV = sK + kBlockK * KS;
  __nv_bfloat16 *sQ = sV + kBlockK * VS;  // 16 rows (8 entries, 8 unused) of KS
  __shared__ float sS[kFixChunk][kBlockK];  // the chunk's scores (log2 units), then the tile's P
  __shared__ int s_ch, s_slot, s_seg, s_merge, s_split;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n_chunks = *count / kFixChunk;
  if (blockIdx.x == 0 && tid == 0 && last_rows) *last_rows = *rows_listed;
  const float scale = kLog2e * rsqrtf(static_cast<float>(D));
  const int n_kt = (T + kBlockK - 1) / kBlockK;
  const bool gated = gate.lam != nullptr;
  const int kseg = fix_seg_tiles(n_kt), max_seg = fix_max_segs(n_kt);
  constexpr int kPart = 2 + 4 * D;  // floats of one row's partial state: m, L, then c, A, W, M per channel

  // warp 0 claims the work; lane 0 keeps the list's next chunk claimed one ahead and the
  // chunk this block split
  int claim = n_chunks, my_slot = -1, my_nseg = 0, my_chunk = 0;
  if (tid == 0) claim = atomicAdd(next_chunk, 1);
  for (;;) {
    // the next piece: (1) the next segment of the chunk this block split; (2) the list's
    // next chunk; (3) once the list is exhausted, a segment of a chunk another block split
    if (!SPLIT) {
      if (tid == 0) {
        s_ch = claim;
        s_slot = -1;
        s_seg = 0;
        if (claim < n_chunks) claim = atomicAdd(next_chunk, 1);
      }
    } else if (warp == 0) {
      int ch = n_chunks, slot = -1, seg = 0;
      if (lane == 0) {
        if (my_slot >= 0) {
          const int sg = atomicAdd(&slots[my_slot].next, 1);
          if (sg < my_nseg) {
            ch = my_chunk;
            slot = my_slot;
            seg = sg;
          } else {
            my_slot = -1;
          }
        }
        if (slot < 0 && claim < n_chunks) {
          ch = claim;
          claim = atomicAdd(next_chunk, 1);
        }
      }
      ch = __shfl_sync(0xffffffffu, ch, 0);
      slot = __shfl_sync(0xffffffffu, slot, 0);
      seg = __shfl_sync(0xffffffffu, seg, 0);
      if (slot < 0 && ch >= n_chunks) {
        // lanes over the slots, 32 at a time; the lowest lane holding one with segments left claims
        const int nl = min(*reinterpret_cast<volatile int *>(fix_long), kFixPoolSlots);
        for (int b0 = 0; b0 < nl && slot < 0; b0 += 32) {
          const int li = b0 + lane;
          bool cand = false;
          if (li < nl) {
            volatile FixSlot *fs = slots + li;
            if (fs->ready != 0) {
              __threadfence();  // the slot's fields, written before ready
              cand = fs->next < fs->n_seg;
            }
          }
          unsigned bal = __ballot_sync(0xffffffffu, cand);
          while (bal && slot < 0) {
            const int src = __ffs(bal) - 1;
            bal &= bal - 1;
            int got = -1, gch = 0;
            if (lane == src) {
              volatile FixSlot *fs = slots + li;
              const int sg = atomicAdd(&slots[li].next, 1);
              if (sg < fs->n_seg) {
                got = sg;
                gch = fs->chunk;
              }
            }
            got = __shfl_sync(0xffffffffu, got, src);
            gch = __shfl_sync(0xffffffffu, gch, src);
            if (got >= 0) {
              ch = gch;
              slot = b0 + src;
              seg = got;
            }
          }
        }
      }
      if (lane == 0) {
        s_ch = ch;
        s_slot = slot;
        s_seg = seg;
      }
    }
    __syncthreads();
    const int ch = s_ch;
    int slot = SPLIT ? s_slot : -1, seg = SPLIT ? s_seg : 0;
    if (ch >= n_chunks) break;
    const FixupEntry ent = entries[ch * kFixChunk + warp];
    const FixupEntry ent0 = entries[ch * kFixChunk];  // the chunk's first entry is a real row
    const int bh = ent0.row / T, h = bh % H;
    const int qt = (ent0.row % T) / kBlockQ, kt0 = ent0.kt0;
    const int kt_end = causal ? qt : n_kt - 1;
    if (SPLIT && slot < 0 && kt0 == 0 && kt_end + 1 >= 2 * kseg) {
      // a recomputation from the first key tile over 2 kseg tiles or more: split into segments
      // that other blocks may take, this block taking the first (the whole chunk when no slot is free)
      if (tid == 0) {
        const int li = atomicAdd(fix_long, 1);
        int got = -1;
        if (li < kFixPoolSlots) {
          FixSlot *fs = slots + li;
          my_nseg = (kt_end + kseg) / kseg;
          my_chunk = ch;
          fs->chunk = ch;
          fs->n_seg = my_nseg;
          fs->next = 1;
          fs->done = 0;
          __threadfence();
          atomicExch(&fs->ready, 1);
          my_slot = got = li;
        }
        s_split = got;
      }
      __syncthreads();
      slot = s_split;
      seg = 0;
    }
    // the key tiles of this piece: the whole chunk, or one segment of it
    const int kt_lo = slot < 0 ? kt0 : seg * kseg, kt_hi = slot < 0 ? kt_end : min(kt_end, kt_lo + kseg - 1);
    const int t = ent.row >= 0 ? ent.row - bh * T : -1;  // this warp's row
    const bool need_mu = gated && kt0 == 0 && ent.l_pre > 0.f;  // the gated read's mean recomputed too
    // the entry's state, lane l holding channels l + 32 g
    float m = -INFINITY, L = 0.f;
    float c_reg[G], A_reg[G], W_reg[G], M_reg[G], b_reg[G], rb_reg[G], c0_reg[G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const int j = lane + 32 * g;
      const float bj = beta[h * D + j];
      b_reg[g] = bj;
      rb_reg[g] = bj != 0.f ? 1.f / bj : 0.f;
      c_reg[g] = -INFINITY;
      A_reg[g] = W_reg[g] = M_reg[g] = 0.f;
      c0_reg[g] = need_mu ? gate.chan0[bh * D + j].c_lin : 0.f;  // the mean's anchor
    }
    if (t >= 0 && kt0 > 0) {
      m = ent.m_pre;
      L = ent.l_pre;
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const int j = lane + 32 * g;
        if (!((ent.mask[g] >> lane) & 1u)) continue;
        const float a = out[static_cast<size_t>(ent.row) * D + j];
        const ChanInfo ci = chan[bh * D + j];
        if (ci.linear != 0.f) {
          c_reg[g] = ci.c_lin;
          W_reg[g] = a;
          A_reg[g] = fmaf(b_reg[g], a, L);
        } else {
          c_reg[g] = shift[(static_cast<size_t>(bh) * n_kt + kt0 - 1) * D + j];
          A_reg[g] = a * 0.018315638888734f;  // e^-kappa
          W_reg[g] = (A_reg[g] - L) * rb_reg[g];
        }
      }
    }
    // the chunk's query rows, once, in flight with the first tile's K and V
    // (a padding row scores the chunk's first row and is never read)
    for (int idx = tid; idx < kFixChunk * (D / 8); idx += kFixThreads) {
      const int w = idx / (D / 8), c = idx % (D / 8);
      const int erow = entries[ch * kFixChunk + w].row;
      fix_cp16(smem_u32(sQ + w * KS + 8 * c), q + static_cast<size_t>(erow >= 0 ? erow : ent0.row) * D + 8 * c);
    }
    // the chunk's last row (every warp from the entries' rows, no barrier)
    int t_last = lane < kFixChunk ? entries[ch * kFixChunk + lane].row : -1;
#pragma unroll
    for (int off = 16; off; off >>= 1) t_last = max(t_last, __shfl_xor_sync(0xffffffffu, t_last, off));
    t_last -= bh * T;
    for (int kt = kt_lo; kt <= kt_hi; ++kt) {
      const int k0 = kt * kBlockK;
      const bool diag = causal && kt == qt;
      // keys k0 .. k0+nk-1 serve every row of the chunk
      const int nk = diag ? t_last - k0 + 1 : min(kBlockK, T - k0);
      for (int idx = tid; idx < nk * (D / 8); idx += kFixThreads) {
        const int i = idx / (D / 8), c = idx % (D / 8);
        const size_t gk = (static_cast<size_t>(bh) * T + k0 + i) * D + 8 * c;
        fix_cp16(smem_u32(sK + i * KS + 8 * c), k + gk);
        const uint32_t dv = smem_u32(sV + i * VS + 8 * c);
#pragma unroll
        for (int w = 0; w < 4; ++w) fix_cp4(dv + 4 * w, v + gk + 2 * w);
      }
      fix_cp_wait_all();
      __syncthreads();
      // S[16 x nk] = Q K^T: warp w takes keys 16w .. 16w+15 (two n8 blocks) over
      // D/16 k-steps of m16n8k16; keys past nk read stale rows and are masked below
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
        // fragment rows lane/4 and lane/4 + 8, columns 2 (lane % 4) + {0, 1}
        const int rr = lane / 4, cc = 16 * warp + 2 * (lane % 4);
        sS[rr][cc] = c0[0] * scale;
        sS[rr][cc + 1] = c0[1] * scale;
        sS[rr][cc + 8] = c1[0] * scale;
        sS[rr][cc + 9] = c1[1] * scale;
        if (kFixChunk > 8) {
          sS[rr + 8][cc] = c0[2] * scale;
          sS[rr + 8][cc + 1] = c0[3] * scale;
          sS[rr + 8][cc + 8] = c1[2] * scale;
          sS[rr + 8][cc + 9] = c1[3] * scale;
        }
      }
      __syncthreads();
      if (t >= 0) {
        // keys i = lane + 32u visible to the row: i < nk, and k0 + i <= t when causal
        const int n_vis = diag ? t - k0 + 1 : nk;
        float s[kBlockK / 32];
        float mt = -INFINITY;
#pragma unroll
        for (int u = 0; u < kBlockK / 32; ++u) {
          const int i = lane + 32 * u;
          s[u] = i < n_vis ? sS[warp][i] : -INFINITY;
          mt = fmaxf(mt, s[u]);
        }
        mt = warp_max(mt);
        if (mt > m) {  // the row maximum moves: every sum scales by 2^(m_old - m_new)
          const float al = exp2f(m - mt);
          L *= al;
#pragma unroll
          for (int g = 0; g < G; ++g) {
            A_reg[g] *= al;
            W_reg[g] *= al;
            M_reg[g] *= al;
          }
          m = mt;
        }
        float p[kBlockK / 32], lt = 0.f;
#pragma unroll
        for (int u = 0; u < kBlockK / 32; ++u) {
          p[u] = s[u] == -INFINITY ? 0.f : exp2f(s[u] - m);
          lt += p[u];
        }
        lt = warp_sum(lt);
        __syncwarp();
#pragma unroll
        for (int u = 0; u < kBlockK / 32; ++u) sS[warp][lane + 32 * u] = p[u];  // this row's P, for the walks
        __syncwarp();
#pragma unroll
        for (int g = 0; g < G; ++g) {
          unsigned mk = ent.mask[g];
          if (__popc(mk) >= 3) {
            // many listed channels in this group: lane = channel, keys walked in
            // turn, first for the visible maximum, then for the sums at it
            const int j = 32 * g + lane;
            float vt = -INFINITY;
            for (int i = 0; i < n_vis; ++i) vt = fmaxf(vt, __bfloat162float(sV[i * VS + j]));
            float c = c_reg[g], A = A_reg[g], W = W_reg[g];
            const float b = b_reg[g], rb = rb_reg[g], bl = b * kLog2e;
            const bool with_w = b < kFixWBeta;
            shift_state(c, A, W, vt, b, rb, L);
            float sm = 0.f;
            for (int i = 0; i < n_vis; ++i) {
              const float pi = sS[warp][i], x = __bfloat162float(sV[i * VS + j]);
              const float xs = x - c, e = exp2f(bl * xs);
              A = fmaf(pi, e, A);
              if (with_w) W = fmaf(pi, em1_over_beta(xs, b * xs, e, rb), W);
              if (need_mu) sm = fmaf(pi, x - c0_reg[g], sm);
            }
            if ((mk >> lane) & 1u) {
              c_reg[g] = c;
              A_reg[g] = A;
              W_reg[g] = W;
              M_reg[g] += sm;
            }
            mk = 0;
          }
          while (mk) {
            // lanes = keys for one listed channel: the tile's sums at the tile's
            // own maximum vt, folded into the state by the lane holding it (jl)
            const int jl = __ffs(mk) - 1, j = 32 * g + jl;
            mk &= mk - 1;
            const float b = __shfl_sync(0xffffffffu, b_reg[g], jl), rb = b != 0.f ? 1.f / b : 0.f;
            const float c0 = need_mu ? __shfl_sync(0xffffffffu, c0_reg[g], jl) : 0.f;
            float x[kBlockK / 32], vt = -INFINITY;
#pragma unroll
            for (int u = 0; u < kBlockK / 32; ++u) {
              const int i = lane + 32 * u;
              x[u] = i < n_vis ? __bfloat162float(sV[i * VS + j]) : -INFINITY;
              vt = fmaxf(vt, x[u]);
            }
            vt = warp_max(vt);
            const float bl = b * kLog2e;
            float sa = 0.f, sw = 0.f, sm = 0.f;
#pragma unroll
            for (int u = 0; u < kBlockK / 32; ++u) {
              if (p[u] == 0.f) continue;
              const float xs = x[u] - vt, y = b * xs, e = exp2f(bl * xs);
              sa = fmaf(p[u], e, sa);
              if (b < kFixWBeta) sw = fmaf(p[u], em1_over_beta(xs, y, e, rb), sw);
              if (need_mu) sm = fmaf(p[u], x[u] - c0, sm);
            }
            sa = warp_sum(sa);
            if (b < kFixWBeta) sw = warp_sum(sw);
            if (need_mu) sm = warp_sum(sm);
            if (lane == jl) {
              fold_tile(c_reg[g], A_reg[g], W_reg[g], L, vt, sa, sw, lt, b, rb);
              M_reg[g] += sm;
            }
          }
        }
        L += lt;
      }
      __syncthreads();  // the staged rows are rewritten by the next tile or chunk
    }
    bool read_out = !SPLIT || slot < 0;
    if (SPLIT && slot >= 0) {
      // a segment: its partial state to the pool; the last segment to finish merges them all
      float *pp = part + ((static_cast<size_t>(slot) * max_seg + seg) * kFixChunk + warp) * kPart;
      if (t >= 0) {
        if (lane == 0) {
          pp[0] = m;
          pp[1] = L;
        }
#pragma unroll
        for (int g = 0; g < G; ++g) {
          if (!((ent.mask[g] >> lane) & 1u)) continue;
          const int j = lane + 32 * g;
          pp[2 + j] = c_reg[g];
          pp[2 + D + j] = A_reg[g];
          pp[2 + 2 * D + j] = W_reg[g];
          pp[2 + 3 * D + j] = M_reg[g];
        }
      }
      __threadfence();
      __syncthreads();
      if (tid == 0) {
        const int n_seg = reinterpret_cast<volatile FixSlot *>(slots)[slot].n_seg;
        s_merge = atomicAdd(&slots[slot].done, 1) == n_seg - 1;
      }
      __syncthreads();
      read_out = s_merge != 0;
      if (read_out && t >= 0) {
        // every segment's state, in key order, each at its own row maximum and shifts:
        // scaled to the common maximum and folded like a key tile's sums
        __threadfence();
        const int n_seg = reinterpret_cast<volatile FixSlot *>(slots)[slot].n_seg;
        m = -INFINITY;
        L = 0.f;
#pragma unroll
        for (int g = 0; g < G; ++g) {
          c_reg[g] = -INFINITY;
          A_reg[g] = W_reg[g] = M_reg[g] = 0.f;
        }
        for (int sg = 0; sg < n_seg; ++sg) {
          const float *ps = part + ((static_cast<size_t>(slot) * max_seg + sg) * kFixChunk + warp) * kPart;
          const float ms = __ldcg(ps), mn = fmaxf(m, ms);
          const float al = exp2f(m - mn), as = exp2f(ms - mn), ls = __ldcg(ps + 1) * as;
          L *= al;
#pragma unroll
          for (int g = 0; g < G; ++g) {
            if (!((ent.mask[g] >> lane) & 1u)) continue;
            const int j = lane + 32 * g;
            A_reg[g] *= al;
            W_reg[g] *= al;
            M_reg[g] = fmaf(M_reg[g], al, __ldcg(ps + 2 + 3 * D + j) * as);
            fold_tile(c_reg[g], A_reg[g], W_reg[g], L, __ldcg(ps + 2 + j), __ldcg(ps + 2 + D + j) * as,
                      __ldcg(ps + 2 + 2 * D + j) * as, ls, b_reg[g], rb_reg[g]);
          }
          L += ls;
          m = mn;
        }
      }
    }
    if (read_out && t >= 0) {
#pragma unroll
      for (int g = 0; g < G; ++g) {
        if (!((ent.mask[g] >> lane) & 1u)) continue;
        const int j = lane + 32 * g;
        const float b = b_reg[g], c = c_reg[g];
        float o;
        if (b == 0.f) {
          o = c + W_reg[g] / L;
        } else {
          const float z = b * W_reg[g] / L;
          o = (b < kFixWBeta && z > -0.5f) ? c + log1pf(z) * rb_reg[g] : c + logf(A_reg[g] / L) * rb_reg[g];
        }
        const size_t oi = static_cast<size_t>(ent.row) * D + j;
        if (gated) {
          const float mu = (kt0 == 0 && ent.l_pre > 0.f) ? c0_reg[g] + M_reg[g] / L : gate.mu_side[oi];
          o = gate.g[oi] * fmaf(gate.lam[oi], o - mu, mu);
        }
        out[oi] = o;
      }
    }
    __syncthreads();  // s_ch and the staged query rows are rewritten by the next chunk
  }
}

cudaError_t launch_fixup(const void *q, const void *k, const void *v, const float *beta, const ChanInfo *chan,
                         const float *shift, float *out, int H, int T, int d, int causal, const FixupEntry *entries,
                         const int *count, const int *rows, int *next_chunk, int *last_rows, const TcGate *gate,
                         int *fix_long, FixSlot *fix_slots, float *fix_part, int num_sms, cudaStream_t stream,
                         bool pdl) {
  const TcGate g = gate ? *gate : TcGate{nullptr, nullptr, nullptr, nullptr, nullptr};
  const __nv_bfloat16 *qb = static_cast<const __nv_bfloat16 *>(q), *kb = static_cast<const __nv_bfloat16 *>(k),
                      *vb = static_cast<const __nv_bfloat16 *>(v);
  const int grid = num_sms * (d == 64 ? 4 : 3);
  if (d == 64) {
    const size_t smem = (kBlockK * (64 + 8) + kBlockK * (64 + 2) + 16 * (64 + 8)) * sizeof(__nv_bfloat16);
    cudaError_t e = launch_kernel(fix_part ? fixup_kernel<64, true> : fixup_kernel<64, false>, dim3(grid),
                                  dim3(kFixThreads), smem, stream, pdl, qb, kb, vb, beta, chan, shift, out, H, T,
                                  causal, entries, count, rows, next_chunk, last_rows, g, fix_long, fix_slots, fix_part);
    if (e != cudaSuccess) return e;
  } else if (d == 128) {
    const size_t smem = (kBlockK * (128 + 8) + kBlockK * (128 + 2) + 16 * (128 + 8)) * sizeof(__nv_bfloat16);
    const auto kern = fix_part ? fixup_kernel<128, true> : fixup_kernel<128, false>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    // three blocks per SM need the largest shared-memory carveout
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
    e = launch_kernel(kern, dim3(grid), dim3(kFixThreads), smem, stream, pdl, qb, kb, vb, beta, chan, shift, out, H, T,
                      causal, entries, count, rows, next_chunk, last_rows, g, fix_long, fix_slots, fix_part);
    if (e != cudaSuccess) return e;
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace fem
