// Tensor-core kernel of the FEM read for bf16 inputs (sm_103a, tcgen05).
//
// One CTA reads two 128-row query tiles (A = rows [256p, 256p+128), B = the
// next 128) of one (b, h) against the key tiles they see, with the value bank
// E (fp16, built once per key tile by the pre-pass) in place of V:
//
//   warp 0        TMA producer: Q_A, Q_B once; K and E tiles through a
//                 two-stage ring (full / empty mbarriers)
//   warp 1 (2)    MMA issuer of tile A (B): S = Q K^T (both operands in shared
//                 memory) into TMEM, then, once the softmax has written P,
//                 acc += P E with P read from TMEM.  Two issuers keep the
//                 tensor pipe busy while either softmax runs.
//   warp 3        TMEM allocation
//   warps 4-7     softmax of tile A (thread = row), warps 8-11 of tile B:
//                 S -> P = exp(s - m) (row max m raised lazily), P rounded to
//                 fp16 and written over S in TMEM, row sum L; when m or a
//                 channel shift moved, acc is rescaled element-wise by
//                 exp(m_old - m_new) * exp(beta_j (c_old - c_new)) before the
//                 next P E (the previous P E is complete: this tile's S was
//                 committed after it by the same issuer); epilogue
//                 o = c + log1p(beta acc/L)/beta (linear bank) or
//                 o = c + (log(acc/L) - kappa)/beta (shifted bank), lse = m + log L.
//
// sum_i exp(s_i - m) E_ij is the free energy's numerator up to the
// stabilising shifts and L its normaliser (Sec. 2.3, Eq.
// "fem-free-energy-main", with the softmax prior of App. C); the value bank
// is mixed with the same prior weights in one pass (App. E, "One-pass
// implementation").
//
// TMEM (512 columns): S_A [0,128) S_B [128,256) acc_A [256,256+D)
// acc_B [256+D, 256+2D); P overwrites the first 64 columns of its S.
// Shared memory: Q_A, Q_B, K[2], E[2] tiles of [128 x D] 16-bit elements in the
// 128-byte-swizzle layout TMA writes (64-element column blocks of 128 rows x
// 128 bytes, chunk c of row r at chunk c ^ (r & 7)), then barriers and
// per-channel state.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

template <int D>
struct TcLayout {
  static constexpr uint32_t kTile = D * 128 * 2;
  static constexpr uint32_t kQ = 0;            // Q_A, Q_B
  static constexpr uint32_t kK = 2 * kTile;    // K[0], K[1]
  static constexpr uint32_t kE = 4 * kTile;    // E[0], E[1]
  static constexpr uint32_t kBar = 6 * kTile;  // 16 mbarriers
  static constexpr uint32_t kTmemSlot = kBar + 16 * 8;
  static constexpr uint32_t kAbort = kTmemSlot + 4;
  static constexpr uint32_t kChan = kBar + 256;  // beta, linear flag, anchor
  static constexpr uint32_t kMoveBits = kChan + 3 * D * 4;  // 1 bit per key tile: a shift moved
  static constexpr int kMaxKeyTiles = 8192;                  // T <= 1M keys
  static constexpr uint32_t kBytes = kMoveBits + kMaxKeyTiles / 8;
  static constexpr uint32_t kAlloc = kBytes + 1024;
};

// mbarrier indices
enum : int {
  kBarQ = 0,
  kBarKFull = 1,    // + stage
  kBarKEmpty = 3,   // + stage
  kBarEFull = 5,    // + stage
  kBarEEmpty = 7,   // + stage
  kBarSFull = 9,    // + query tile
  kBarPFull = 11,   // + query tile
  kBarAccDone = 13  // + query tile
};

// Bounded wait that also gives up as soon as another role has given up.
__device__ __forceinline__ bool wait_or_abort(uint32_t bar, uint32_t parity, unsigned *err, unsigned code,
                                              volatile int *abort_flag) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = global_timer_ns();
  while (true) {
    if (mbar_try_wait_sleep(bar, parity, 200000u)) return true;
    if (*abort_flag) return false;
    if (global_timer_ns() - t0 > kWaitLimitNs) {
      atomicOr(err, code);
      *abort_flag = 1;
      return false;
    }
  }
}

__device__ __forceinline__ uint32_t pack_half2(float lo, float hi) {
  const __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<const uint32_t *>(&v);
}

template <int D>
__global__ void __launch_bounds__(384, 1)
    fem_tc_kernel(const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_k,
                  const __grid_constant__ CUtensorMap tmap_e, const float *__restrict__ beta,
                  const ChanInfo *__restrict__ chan, const float *__restrict__ shift,
                  const float *__restrict__ rfac, const unsigned *__restrict__ colmask, float *__restrict__ out,
                  float *__restrict__ lse, int H, int T, int causal, unsigned *__restrict__ err) {
  using Lay = TcLayout<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + Lay::kAbort);
  float *c_beta = reinterpret_cast<float *>(smem + Lay::kChan);
  float *c_lin = c_beta + D;
  float *c_anchor = c_lin + D;
  unsigned *move_bits = reinterpret_cast<unsigned *>(smem + Lay::kMoveBits);
  const uint32_t bars = sbase + Lay::kBar;
#define FEM_BAR(i) (bars + 8u * static_cast<uint32_t>(i))

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n_qt = (T + kBlockQ - 1) / kBlockQ;
  const int n_kt_all = (T + kBlockK - 1) / kBlockK;
  const int n_pairs = (n_qt + 1) / 2;
  const int pair = n_pairs - 1 - static_cast<int>(blockIdx.x);  // heaviest causal pairs first
  const int bh = blockIdx.y, h = bh % H;
  const int qt0 = 2 * pair;
  const int n_tiles = (qt0 + 1 < n_qt) ? 2 : 1;  // query tiles in this CTA
  const int nk0 = causal ? qt0 + 1 : n_kt_all;   // key tiles tile A reads
  const int nk1 = causal ? qt0 + 2 : n_kt_all;   // key tiles tile B reads
  const int nk_load = n_tiles == 2 ? nk1 : nk0;

  if (warp == 3) {
    tmem_alloc(sbase + Lay::kTmemSlot, 512);
    tmem_relinquish();
  }
  if (tid == 0) {
    mbar_init(FEM_BAR(kBarQ), 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(FEM_BAR(kBarKFull + s), 1);
      mbar_init(FEM_BAR(kBarKEmpty + s), n_tiles);
      mbar_init(FEM_BAR(kBarEFull + s), 1);
      mbar_init(FEM_BAR(kBarEEmpty + s), n_tiles);
    }
    for (int q = 0; q < 2; ++q) {
      mbar_init(FEM_BAR(kBarSFull + q), 1);
      mbar_init(FEM_BAR(kBarPFull + q), 128);
      mbar_init(FEM_BAR(kBarAccDone + q), 1);
    }
    fence_mbar_init();
    *abort_flag = 0;
  }
  for (int j = tid; j < D; j += 384) {
    const ChanInfo ci = chan[bh * D + j];
    c_beta[j] = beta[h * D + j];
    c_lin[j] = ci.linear;
    c_anchor[j] = ci.c_lin;
  }
  for (int w = tid; w < (n_kt_all + 31) / 32; w += 384) {
    unsigned bits = 0;
    for (int b = 0; b < 32 && 32 * w + b < n_kt_all; ++b) {
      const uint4 m = reinterpret_cast<const uint4 *>(colmask)[static_cast<size_t>(bh) * n_kt_all + 32 * w + b];
      bits |= ((m.x | m.y | m.z | m.w) != 0u ? 1u : 0u) << b;
    }
    move_bits[w] = bits;
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(smem + Lay::kTmemSlot);

  if (warp < 4) {
  // registers move from this warpgroup to the softmax warpgroups, which hold a
  // 128-float score row per thread
  setmaxnreg_dec56();
  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      prefetch_tensormap(&tmap_q);
      prefetch_tensormap(&tmap_k);
      prefetch_tensormap(&tmap_e);
      mbar_arrive_expect_tx(FEM_BAR(kBarQ), n_tiles * Lay::kTile);
      for (int q = 0; q < n_tiles; ++q)
        for (int b = 0; b < D / 64; ++b)
          tma_load_3d(sbase + Lay::kQ + q * Lay::kTile + b * 16384, &tmap_q, FEM_BAR(kBarQ), b * 64,
                      (qt0 + q) * kBlockQ, bh);
      for (int kt = 0; kt < nk_load; ++kt) {
        const int st = kt & 1;
        const uint32_t use = static_cast<uint32_t>(kt >> 1);
        if (kt >= 2 && !wait_or_abort(FEM_BAR(kBarKEmpty + st), (use - 1) & 1, err, kErrWaitMma, abort_flag)) break;
        mbar_arrive_expect_tx(FEM_BAR(kBarKFull + st), Lay::kTile);
        for (int b = 0; b < D / 64; ++b)
          tma_load_3d(sbase + Lay::kK + st * Lay::kTile + b * 16384, &tmap_k, FEM_BAR(kBarKFull + st), b * 64,
                      kt * kBlockK, bh);
        if (kt >= 2 && !wait_or_abort(FEM_BAR(kBarEEmpty + st), (use - 1) & 1, err, kErrWaitMma, abort_flag)) break;
        mbar_arrive_expect_tx(FEM_BAR(kBarEFull + st), Lay::kTile);
        for (int b = 0; b < D / 64; ++b)
          tma_load_3d(sbase + Lay::kE + st * Lay::kTile + b * 16384, &tmap_e, FEM_BAR(kBarEFull + st), b * 64,
                      kt * kBlockK, bh);
      }
    }
  } else if (warp == 1 || warp == 2) {
    // ---------------------------------------------------------------- MMA issuers
    const int q = warp - 1;
    if (q < n_tiles && lane == 0) {
      const int nk = q == 0 ? nk0 : nk1;
      const uint32_t tS = tmem + q * 128;
      const uint32_t tAcc = tmem + 256 + q * D;
      const uint32_t sQ = sbase + Lay::kQ + q * Lay::kTile;
      constexpr uint32_t idesc_qk = idesc_f16(128, 128, true, false);
      constexpr uint32_t idesc_pv = idesc_f16(128, D, false, true);
      bool ok = wait_or_abort(FEM_BAR(kBarQ), 0, err, kErrWaitTma, abort_flag);
      for (int kt = 0; ok && kt < nk; ++kt) {
        const int st = kt & 1;
        const uint32_t ph = static_cast<uint32_t>(kt >> 1) & 1;
        if (!(ok = wait_or_abort(FEM_BAR(kBarKFull + st), ph, err, kErrWaitTma, abort_flag))) break;
        tc_fence_after_sync();
        const uint32_t sK = sbase + Lay::kK + st * Lay::kTile;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * 16384 + (kk & 3) * 32;
          mma_f16_ss(tS, smem_desc_sw128(sQ + off, 16, 1024), smem_desc_sw128(sK + off, 16, 1024), idesc_qk,
                     kk > 0 ? 1u : 0u);
        }
        mma_commit(FEM_BAR(kBarSFull + q));
        mma_commit(FEM_BAR(kBarKEmpty + st));
        if (!(ok = wait_or_abort(FEM_BAR(kBarPFull + q), kt & 1, err, kErrWaitMma, abort_flag))) break;
        if (!(ok = wait_or_abort(FEM_BAR(kBarEFull + st), ph, err, kErrWaitTma, abort_flag))) break;
        tc_fence_after_sync();
        const uint32_t sE = sbase + Lay::kE + st * Lay::kTile;
#pragma unroll
        for (int kk = 0; kk < kBlockK / 16; ++kk)
          mma_f16_ts(tAcc, tS + kk * 8, smem_desc_sw128(sE + kk * 2048, 16384, 1024), idesc_pv,
                     (kt > 0 || kk > 0) ? 1u : 0u);
        mma_commit(FEM_BAR(kBarEEmpty + st));
      }
      mma_commit(FEM_BAR(kBarAccDone + q));  // completes once everything this thread issued is done
    }
  } else if (warp == 3 && lane == 0) {
    // make sure no MMA is still in flight before the allocation is released
    for (int q = 0; q < n_tiles; ++q) wait_or_abort(FEM_BAR(kBarAccDone + q), 0, err, kErrWaitMma, abort_flag);
  }
  } else {
    setmaxnreg_inc224();
    // ---------------------------------------------------------------- softmax + epilogue
    const int q = (warp - 4) >> 2;      // query tile of this warpgroup
    const int r = tid - 128 - 128 * q;  // row within the tile
    if (q < n_tiles) {
      const int nk = q == 0 ? nk0 : nk1;
      const int qt = qt0 + q;
      const int t_row = qt * kBlockQ + r;
      const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;
      const uint32_t tS = tmem + q * 128 + lane_off;
      const uint32_t tAcc = tmem + 256 + q * D + lane_off;
      const float qk_scale = kLog2e * rsqrtf(static_cast<float>(D));
      const float *shift_bh = shift + static_cast<size_t>(bh) * n_kt_all * D;
      const float *rfac_bh = rfac + static_cast<size_t>(bh) * n_kt_all * D;
      float m_row = -INFINITY, L_row = 0.f;
      bool ok = true;
      for (int kt = 0; kt < nk; ++kt) {
        const bool colmv = (move_bits[kt >> 5] >> (kt & 31)) & 1u;  // some channel's shift moved
        // every lane takes the same branch: the wait's outcome is made warp-uniform
        ok = __all_sync(0xffffffffu, wait_or_abort(FEM_BAR(kBarSFull + q), kt & 1, err, kErrWaitMma, abort_flag));
        if (!ok) break;
        tc_fence_after_sync();
        // the whole 128-column score row: four loads in flight, one wait
        uint32_t sr[128];
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld32(tS + c * 32, *reinterpret_cast<uint32_t(*)[32]>(&sr[c * 32]));
        tmem_ld_wait();
        float *s = reinterpret_cast<float *>(sr);
        const int k0 = kt * kBlockK;
        if ((causal && kt == qt) || k0 + kBlockK > T) {
          // keys k0 + n are visible for n < lim (key < T, and key <= row when causal)
          const int lim = min(T, causal ? t_row + 1 : T) - k0;
#pragma unroll
          for (int n = 0; n < 128; ++n) s[n] = n < lim ? s[n] : -INFINITY;
        }
        float mx[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) mx[u] = s[u];
#pragma unroll
        for (int n = 8; n < 128; ++n) mx[n & 7] = fmaxf(mx[n & 7], s[n]);
        float tmax = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])), fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
        tmax *= qk_scale;  // log2-domain row maximum of this tile
        float alpha = 1.f;
        if (tmax > m_row + kRowMaxLag) {
          alpha = ex2_approx(m_row - tmax);  // 0 on the first tile
          m_row = tmax;
        }
        // P = exp2(s * scale - m) as fp16 over the first 64 columns of S; L from the fp32 values
        const float2 scale2 = make_float2(qk_scale, qk_scale), negm2 = make_float2(-m_row, -m_row);
        float2 ls[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) ls[u] = make_float2(0.f, 0.f);
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          uint32_t p[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float2 x = __ffma2_rn(make_float2(s[c * 32 + 2 * i], s[c * 32 + 2 * i + 1]), scale2, negm2);
            const float2 e = make_float2(ex2_approx(x.x), ex2_approx(x.y));
            ls[i & 3] = __fadd2_rn(ls[i & 3], e);
            p[i] = pack_half2(e.x, e.y);
          }
          tmem_st16(tS + c * 16, p);
        }
        const float lsum = (ls[0].x + ls[0].y) + (ls[1].x + ls[1].y) + (ls[2].x + ls[2].y) + (ls[3].x + ls[3].y);
        // joint online rescale of acc (the previous P E has completed): every
        // column when a row maximum moved, else only the moved channels
        if (kt > 0) {
          const float *rf = rfac_bh + kt * D;  // exp(beta_j (c_old - c_new)), 1 for unmoved channels
          if (__any_sync(0xffffffffu, alpha != 1.f)) {
#pragma unroll 1
            for (int c = 0; c < D / 32; ++c) {
              uint32_t v[32];
              tmem_ld32(tAcc + c * 32, v);
              tmem_ld_wait();
              if (colmv) {
#pragma unroll
                for (int i = 0; i < 32; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) * alpha * rf[c * 32 + i]);
              } else {
#pragma unroll
                for (int i = 0; i < 32; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) * alpha);
              }
              tmem_st32(tAcc + c * 32, v);
            }
          } else if (colmv) {
            const uint4 m4 = reinterpret_cast<const uint4 *>(colmask)[static_cast<size_t>(bh) * n_kt_all + kt];
            const unsigned mw[4] = {m4.x, m4.y, m4.z, m4.w};
#pragma unroll 1
            for (int g = 0; g < D / 32; ++g) {
              unsigned m = mw[g];
              while (m) {
                const int j = 32 * g + __ffs(m) - 1;
                m &= m - 1;
                const uint32_t x = tmem_ld1(tAcc + j);
                tmem_ld_wait();
                tmem_st1(tAcc + j, __float_as_uint(__uint_as_float(x) * rf[j]));
              }
            }
          }
        }
        L_row = L_row * alpha + lsum;
        tmem_st_wait();
        tc_fence_before_sync();
        mbar_arrive(FEM_BAR(kBarPFull + q));
      }
      // ---- epilogue
      if (ok) ok = __all_sync(0xffffffffu, wait_or_abort(FEM_BAR(kBarAccDone + q), 0, err, kErrWaitMma, abort_flag));
      if (ok) {
        const float *c_last = shift_bh + (nk - 1) * D;
        tc_fence_after_sync();
        const bool store = t_row < T;
        const size_t orow = static_cast<size_t>(bh) * T + t_row;
        const float invL = 1.f / L_row;
#pragma unroll 1
        for (int c = 0; c < D / 32; ++c) {
          uint32_t v[32];
          tmem_ld32(tAcc + c * 32, v);
          tmem_ld_wait();
          if (store) {
            float4 *dst = reinterpret_cast<float4 *>(out + orow * D + c * 32);
#pragma unroll
            for (int i4 = 0; i4 < 8; ++i4) {
              float o4[4];
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                const int j = c * 32 + i4 * 4 + u;
                const float a = __uint_as_float(v[i4 * 4 + u]) * invL;
                const float b = c_beta[j];
                if (c_lin[j] != 0.f)
                  o4[u] = b != 0.f ? c_anchor[j] + log1pf(b * a) / b : c_anchor[j] + a;
                else
                  o4[u] = c_last[j] + (logf(a) - kBankOffset) / b;
              }
              dst[i4] = make_float4(o4[0], o4[1], o4[2], o4[3]);
            }
          }
        }
        if (store && lse) lse[orow] = m_row * kLn2 + logf(L_row);
      }
    }
  }

  tc_fence_before_sync();
  __syncthreads();
  if (warp == 3) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, 512);
  }
#undef FEM_BAR
}

template <int D>
static cudaError_t launch_tc_d(const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &te, const float *beta,
                               const ChanInfo *chan, const float *shift, const float *rfac, const unsigned *colmask,
                               float *out, float *lse, int BH, int H, int T, int causal, unsigned *err,
                               cudaStream_t stream) {
  if ((T + kBlockK - 1) / kBlockK > TcLayout<D>::kMaxKeyTiles) return cudaErrorInvalidValue;
  const uint32_t smem = TcLayout<D>::kAlloc;
  cudaError_t e = cudaFuncSetAttribute(fem_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const int n_qt = (T + kBlockQ - 1) / kBlockQ;
  const dim3 grid((n_qt + 1) / 2, BH);
  fem_tc_kernel<D><<<grid, 384, smem, stream>>>(tq, tk, te, beta, chan, shift, rfac, colmask, out, lse, H, T, causal,
                                                err);
  return cudaGetLastError();
}

cudaError_t launch_tc(int d, const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &te, const float *beta,
                      const ChanInfo *chan, const float *shift, const float *rfac, const unsigned *colmask, float *out,
                      float *lse, int BH, int H, int T, int causal, unsigned *err, cudaStream_t stream) {
  if (d == 64)
    return launch_tc_d<64>(tq, tk, te, beta, chan, shift, rfac, colmask, out, lse, BH, H, T, causal, err, stream);
  if (d == 128)
    return launch_tc_d<128>(tq, tk, te, beta, chan, shift, rfac, colmask, out, lse, BH, H, T, causal, err, stream);
  return cudaErrorInvalidValue;
}

}  // namespace fem
