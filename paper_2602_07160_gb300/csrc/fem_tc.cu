// Tensor-core kernel of the FEM read for bf16 inputs (sm_103a, tcgen05).
//
// One CTA reads one 128-row query tile of one (b, h) against the key tiles it
// sees, with the value bank E (fp16, built once per key tile by the
// pre-pass) in place of V.  Three score buffers in TMEM let the score
// contraction of later key tiles and the value contraction of the previous
// one run on the tensor pipe while the softmax works on the current tile:
//
//   warp 0       TMA producer of Q and of the K tiles (three-stage ring)
//   warp 1       S issuer: S_k = Q K_k^T (both operands in shared memory) into
//                score buffer k mod 3, up to two key tiles ahead of the
//                softmax; it waits only for the P E that last read the buffer
//   warp 2       PV issuer: acc += P_k E_k with P_k read from TMEM, once the
//                softmax has written P_k and the correction has rescaled acc.
//                The two issuers are different warps, so their instruction
//                streams overlap on the tensor pipe
//   warp 3       TMEM allocation; TMA producer of the E tiles (two-stage ring)
//   warps 4-7    softmax (thread = row): the tile's row maximum and the factor
//                alpha = exp(m_old - m_new) of a lazily raised running maximum
//                m (handed to the correction at once), then P = exp(s - m)
//                rounded to fp16 over the first 64 columns of the tile's score
//                buffer, and the row sum L
//   warps 8-11   correction (thread = row): once the previous P E completed,
//                the joint online rescale of acc by alpha * exp(beta_j (c_old -
//                c_new)), over every column when a row maximum moved, over the
//                moved channels when only channel shifts moved.  Off the
//                softmax's path, it overlaps the next tile's exponentials.
//                Thread j also keeps channel j's sum of |bank| over the key
//                tiles read, rescaled with the shifts (the guard's Ecol_j)
//   warps 4-11   epilogue, half the columns each:
//                o = c + log1p(beta acc/L)/beta (linear bank) or
//                o = c + (log(acc/L) - kappa)/beta (shifted bank); lse = m + log L;
//                the underflow guard (kGuardTau) on every entry, and the
//                rejected entries listed for the exact fix-up.
//
// Causal diagonal tile (the last key tile of a query tile, when there are
// earlier ones): its P E goes into a free score buffer instead of acc, and
// the epilogue adds acc (rescaled by that tile's alpha and shift factors) to
// it.  acc therefore still holds the state before the diagonal tile, from
// which the fix-up restarts rows whose final state fails the guard but whose
// earlier state passes it.
//
// sum_i exp(s_i - m) E_ij is the free energy's numerator up to the
// stabilising shifts and L its normaliser (Sec. 2.3, Eq.
// "fem-free-energy-main", with the softmax prior of App. C); the value bank is
// mixed with the same prior weights in one pass (App. E, "One-pass
// implementation").
//
// TMEM (512 columns): score buffers [0,128) [128,256) [256,384), acc
// [384, 384 + D); the diagonal tile's P E goes to score buffer nk mod 3.
// Shared memory: Q, K[kStagesK], E[kSlotsE] tiles of [128 x D] 16-bit
// elements in the 128-byte-swizzle layout TMA writes (64-element column
// blocks of 128 rows x 128 bytes, chunk c of row r at chunk c ^ (r & 7)),
// then barriers and per-channel state.  Every mbarrier completes once per use
// of what it guards, and no waiter can fall two phases behind: a buffer's
// next use always waits for the previous one.
#include "fem_common.cuh"
#include "fem_launch.h"
#include "fem_order.h"

namespace fem {

// GATED: the two-level gated read in one pass -- two banks per key tile (the
// mean's, beta = 0, and beta_max's) into two accumulators of D columns each.
template <int D, bool GATED>
struct TcLayout {
  static constexpr int kNB = GATED ? 2 : 1;  // banks per key tile
  static constexpr uint32_t kTile = D * 128 * 2;
  // 512 TMEM columns: kBufS score buffers of 128 and kNB * D accumulator columns
  static constexpr int kBufS = (GATED && D == 128) ? 2 : 3;
  // at d = 128 the bank ring takes the third 32 KB slot: the score contractions run up to two key
  // tiles ahead of the P E, so a bank tile is needed later than its K tile and waits on its load
  // more often (three K stages and two bank slots ran 0.5 % slower per step)
  static constexpr int kStagesK = D == 128 ? 2 : 3;
  static constexpr int kSlotsE = GATED ? (D == 128 ? 3 : 6) : (D == 128 ? 3 : 2);  // one bank tile per slot
  static constexpr uint32_t kQ = 0;
  static constexpr uint32_t kK = kTile;                    // K stages
  static constexpr uint32_t kE = kK + kStagesK * kTile;    // E slots
  static constexpr uint32_t kBar = kE + kSlotsE * kTile;   // mbarriers
  static constexpr int kNumBars = 41;
  static constexpr uint32_t kTmemSlot = kBar + kNumBars * 8;
  static constexpr uint32_t kAbort = kTmemSlot + 4;
  static constexpr uint32_t kChan = kBar + 512;               // per-channel epilogue coefficients
  static constexpr uint32_t kMoveBits = kChan + 4 * D * 4 + (GATED ? 4 * D : 0);
  static constexpr int kMaxKeyTiles = kMaxSeqLen / kBlockK;  // T <= 1M keys
  // side ring: per key tile its rescale factors exp(beta_j (c_old - c_new)) [D],
  // the bank's column sums [D] (GATED: also the mean bank's [D]) and the
  // moved-channel mask [4], loaded with the K tile, kSideStages tiles deep
  static constexpr int kSideStages = 8;
  static constexpr int kSideArrays = GATED ? 3 : 2;
  static constexpr uint32_t kSide = kMoveBits;
  static constexpr uint32_t kSideMask = kSideArrays * D * 4;  // offset of the mask in a slot
  static constexpr uint32_t kSideStride = kSideMask + 128;
  static constexpr uint32_t kAlpha = kSide + kSideStages * kSideStride;  // alpha per row, per score buffer
  static constexpr uint32_t kInvL = kAlpha + kBufS * 128 * 4;         // 1/L per row, for the epilogue
  static constexpr uint32_t kPre = kInvL + 128 * 4;  // per row (m, L) before the diagonal tile
  static constexpr uint32_t kGco = kPre + 128 * 8;   // per channel guard coefficients {X, Z, Y, Zp}
  static constexpr uint32_t kThr = kGco + D * 16;    // per channel: the guard as a < A + B / L, {A, B}
  static constexpr uint32_t kFlag = kThr + D * 8;    // per row and 32-channel group: entries the guard rejects
  static constexpr uint32_t kBad = kFlag + 128 * 16;  // per row: restart from the diagonal tile not possible
  static constexpr uint32_t kMisc = kBad + 128 * 4;   // entry counts and bases, guard bounds, row flags
  // 1/L of row 4 k + q at [32 q + k]: the transform's batch of 8 rows in two 16-byte loads
  static constexpr uint32_t kInvLT = kMisc + 128;
  static constexpr uint32_t kBytes = kInvLT + 128 * 4;
  static constexpr uint32_t kAlloc = kBytes + 1024;
  static constexpr uint32_t kAccCol = kBufS * 128;
  static constexpr uint32_t kAccB = kAccCol + (GATED ? D : 0);  // the beta (or beta_max) read's accumulator
  static_assert(kAccCol + kNB * D <= 512, "TMEM columns");
  static_assert(kBytes <= 227 * 1024 - 1024, "shared memory");
  static_assert(kNB * D / 32 * 16384 <= (kStagesK * kTile + kSlotsE * kTile),
                "epilogue staging fits the idle K and E rings");
};

// mbarrier indices
enum : int {
  kBarQ = 0,
  kBarKFull = 1,     // + K stage (up to 3)
  kBarKEmpty = 4,    // + K stage (up to 3)
  kBarEFull = 7,     // + E slot (up to 6)
  kBarEEmpty = 13,   // + E slot (up to 6)
  kBarSFull = 19,    // + score buffer (up to 3): S_k complete
  kBarPFull = 22,    // + score buffer: P_k written and acc rescaled (256 arrivals)
  kBarPvDone = 25,   // + score buffer: P_k E_k complete
  kBarAccDone = 28,  // every P E complete
  kBarSDone = 29,    // every score contraction the S issuer started is complete
  kBarAlpha = 30,    // + score buffer: the softmax's alpha of tile k is in shared memory (128 arrivals)
  kBarSide = 33      // + side slot (8): tile k's rescale factors and moved-channel mask are in shared memory
};


__device__ __forceinline__ int pad_chunk(int n) { return (n + kFixChunk - 1) / kFixChunk * kFixChunk; }

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

__device__ __forceinline__ uint32_t pack_bf162(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t *>(&v);
}

// ATTN: the attention-mode comparator -- plain softmax attention
// o = sum_i p_t(i) v_i, the same kernel with V itself (bf16) as the second
// operand and P in bf16: no value bank, no shifts, no guard.
template <int D, bool GATED, bool ATTN = false>
__global__ void __launch_bounds__(384, 1)
    fem_tc_kernel(const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_k,
                  const __grid_constant__ CUtensorMap tmap_e, const __grid_constant__ CUtensorMap tmap_e0,
                  float *__restrict__ out, const float *__restrict__ beta, const BankWorkspace w,
                  float *__restrict__ lse, int H, int T, int causal, TcGate gate, unsigned *__restrict__ err) {
  using Lay = TcLayout<D, GATED>;
  constexpr int kNB = Lay::kNB, kBufS = Lay::kBufS, kStagesK = Lay::kStagesK, kSlotsE = Lay::kSlotsE;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + Lay::kAbort);
  // per channel, for the epilogue: shifted bank {0, c - kappa/beta, ln2/beta, 1}
  // with c the last shift; linear bank {beta, c, ln2/beta (0 at beta = 0), 0}
  // with c the anchor
  float4 *c_coef = reinterpret_cast<float4 *>(smem + Lay::kChan);
  const uint32_t bars = sbase + Lay::kBar;
#define FEM_BAR(i) (bars + 8u * static_cast<uint32_t>(i))

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int wg = __shfl_sync(0xffffffffu, tid >> 7, 0);  // warpgroup, provably warp-uniform
  const int n_qt = (T + kBlockQ - 1) / kBlockQ;
  const int n_kt_all = (T + kBlockK - 1) / kBlockK;
  // CTAs in launch order take the heads in groups of kHeadGroup: within a
  // group the query tiles go heaviest first across its heads (causal), so the
  // launch ends on the lightest tiles and the SMs finish together, while the
  // CTAs in flight share the K and E of at most two groups (64 MB at d = 128,
  // T = 8192) in L2: sixteen-head groups doubled that and raised the DRAM reads by 60 %
  const int rank = static_cast<int>(blockIdx.y * gridDim.x + blockIdx.x), BH = static_cast<int>(gridDim.y);
  int bh, qt;
  tc_tile_of_rank(rank, BH, n_qt, causal, bh, qt);
  const int h = bh % H;
  const int nk = causal ? qt + 1 : n_kt_all;  // key tiles this query tile reads
  // causal with earlier key tiles: the diagonal tile's P E (of the beta bank)
  // goes to the score buffer no other tile uses from then on, so acc keeps
  // the state before it
  const bool split = !ATTN && causal && nk > 1;

  // K tile kt into K stage kt % kStagesK, with its side data into side slot
  // kt % 8.  Side slot kt % 8 was last read by the correction of tile kt - 8,
  // which finished before PV(kt - 8), hence before S(kt - kStagesK) (which
  // waited for PV(kt - kStagesK - kBufS)) released this K stage.
  auto load_k = [&](int kt) {
    const int st = kt % kStagesK, ss = kt % Lay::kSideStages;
    mbar_arrive_expect_tx(FEM_BAR(kBarKFull + st), Lay::kTile);
    for (int b = 0; b < D / 64; ++b)
      tma_load_3d(sbase + Lay::kK + st * Lay::kTile + b * 16384, &tmap_k, FEM_BAR(kBarKFull + st), b * 64,
                  kt * kBlockK, bh);
    const size_t row = static_cast<size_t>(bh) * n_kt_all + kt;
    if (ATTN) return;  // no bank, no side data
    const uint32_t slot = sbase + Lay::kSide + ss * Lay::kSideStride;
    mbar_arrive_expect_tx(FEM_BAR(kBarSide + ss), Lay::kSideMask + 16);
    bulk_load(slot, w.rfac + row * D, D * 4, FEM_BAR(kBarSide + ss));
    bulk_load(slot + D * 4, w.colsum + row * D, D * 4, FEM_BAR(kBarSide + ss));
    if (GATED) bulk_load(slot + 2 * D * 4, gate.colsum0 + row * D, D * 4, FEM_BAR(kBarSide + ss));
    bulk_load(slot + Lay::kSideMask, w.colmask + row * 4, 16, FEM_BAR(kBarSide + ss));
  };
  // E item e (key tile e / kNB; bank e % kNB, the mean's first when GATED)
  // into E slot e % kSlotsE
  auto load_e = [&](int e) {
    const int st = e % kSlotsE, kt = e / kNB;
    const CUtensorMap *map = (GATED && e % kNB == 0) ? &tmap_e0 : &tmap_e;
    mbar_arrive_expect_tx(FEM_BAR(kBarEFull + st), Lay::kTile);
    for (int b = 0; b < D / 64; ++b)
      tma_load_3d(sbase + Lay::kE + st * Lay::kTile + b * 16384, map, FEM_BAR(kBarEFull + st), b * 64,
                  kt * kBlockK, bh);
  };
  constexpr int kPreK = kStagesK, kPreE = kSlotsE;  // loads the prologue issues (the rings' depths)
  const int ne = nk * kNB;                           // E items

  grid_dep_launch_dependents();
  if (warp == 3) {
    tmem_alloc(sbase + Lay::kTmemSlot, 512);
    tmem_relinquish();
  }
  grid_dep_wait();  // the value bank, its plan and column sums; the fix-up list's counters
  if (tid == 0) {
    mbar_init(FEM_BAR(kBarQ), 1);
    for (int s = 0; s < kStagesK; ++s) {
      mbar_init(FEM_BAR(kBarKFull + s), 1);
      mbar_init(FEM_BAR(kBarKEmpty + s), 1);
    }
    for (int s = 0; s < kBufS; ++s) {
      mbar_init(FEM_BAR(kBarSFull + s), 1);
      mbar_init(FEM_BAR(kBarPFull + s), 256);
      mbar_init(FEM_BAR(kBarAlpha + s), 128);
      mbar_init(FEM_BAR(kBarPvDone + s), 1);
    }
    for (int s = 0; s < kSlotsE; ++s) {
      mbar_init(FEM_BAR(kBarEFull + s), 1);
      mbar_init(FEM_BAR(kBarEEmpty + s), 1);
    }
    for (int s = 0; s < Lay::kSideStages; ++s) mbar_init(FEM_BAR(kBarSide + s), 1);
    mbar_init(FEM_BAR(kBarAccDone), 1);
    mbar_init(FEM_BAR(kBarSDone), 1);
    fence_mbar_init();
    *abort_flag = 0;
    // the first loads leave before the rest of the prologue: Q, the first
    // kPreK K tiles with their side data, the first kPreE E tiles
    mbar_arrive_expect_tx(FEM_BAR(kBarQ), Lay::kTile);
    for (int b = 0; b < D / 64; ++b)
      tma_load_3d(sbase + Lay::kQ + b * 16384, &tmap_q, FEM_BAR(kBarQ), b * 64, qt * kBlockQ, bh);
    for (int kt = 0; kt < min(nk, kPreK); ++kt) load_k(kt);
    for (int e = 0; e < min(ne, kPreE); ++e) load_e(e);
  }
  if (tid == 0) {
    reinterpret_cast<float *>(smem + Lay::kMisc)[4] = 0.f;        // the mean bank's largest guard bound
  }
  if (tid < 128) reinterpret_cast<unsigned *>(smem + Lay::kBad)[tid] = 0u;
  // rows with listed entries [16..19], rows with candidate entries [20..23]
  if (tid < 8) reinterpret_cast<unsigned *>(smem + Lay::kMisc)[16 + tid] = 0u;
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(smem + Lay::kTmemSlot);
  const uint32_t tDiag = tmem + static_cast<uint32_t>((nk % kBufS) * 128);

  // Every warp keeps the launch's register count: moving registers from the
  // producer warps to the softmax (setmaxnreg) made the compiled code spill
  // more and ran slower.
  if (wg == 0) {
  if (warp == 0) {
    // ---------------------------------------------------------------- TMA: Q and K
    if (lane == 0) {
      for (int kt = kPreK; kt < nk; ++kt) {
        const uint32_t use = static_cast<uint32_t>(kt / kStagesK);
        if (!wait_or_abort(FEM_BAR(kBarKEmpty + kt % kStagesK), (use - 1) & 1, err, kErrWaitMma, abort_flag)) break;
        load_k(kt);
      }
    }
  } else if (warp == 3) {
    // ---------------------------------------------------------------- TMA: E
    if (lane == 0) {
      for (int e = kPreE; e < ne; ++e) {
        const uint32_t use = static_cast<uint32_t>(e / kSlotsE);
        if (!wait_or_abort(FEM_BAR(kBarEEmpty + e % kSlotsE), (use - 1) & 1, err, kErrWaitMma, abort_flag)) break;
        load_e(e);
      }
      // no contraction may be in flight when the TMEM allocation is released:
      // both issuers commit these barriers on every exit path
      mbar_wait(FEM_BAR(kBarSDone), 0, err, kErrWaitMma);
      mbar_wait(FEM_BAR(kBarAccDone), 0, err, kErrWaitMma);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- S issuer
    if (lane == 0) {
      constexpr uint32_t idesc_qk = idesc_f16(128, 128, true, false);
      bool ok = wait_or_abort(FEM_BAR(kBarQ), 0, err, kErrWaitTma, abort_flag);
      for (int kt = 0; ok && kt < nk; ++kt) {
        const int b = kt % kBufS, ks = kt % kStagesK;
        const uint32_t use = static_cast<uint32_t>(kt / kBufS);
        if (!(ok = wait_or_abort(FEM_BAR(kBarKFull + ks), (kt / kStagesK) & 1, err, kErrWaitTma, abort_flag))) break;
        // the buffer's previous tile must have been consumed by its P E
        if (use > 0 && !(ok = wait_or_abort(FEM_BAR(kBarPvDone + b), (use - 1) & 1, err, kErrWaitMma, abort_flag)))
          break;
        tc_fence_after_sync();
        const uint32_t sK = sbase + Lay::kK + ks * Lay::kTile;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * 16384 + (kk & 3) * 32;
          mma_f16_ss(tmem + b * 128, smem_desc_sw128(sbase + Lay::kQ + off, 16, 1024),
                     smem_desc_sw128(sK + off, 16, 1024), idesc_qk, kk > 0 ? 1u : 0u);
        }
        mma_commit(FEM_BAR(kBarSFull + b));
        mma_commit(FEM_BAR(kBarKEmpty + ks));
      }
      mma_commit(FEM_BAR(kBarSDone));
    }
  } else if (warp == 2) {
    // ---------------------------------------------------------------- PV issuer
    if (lane == 0) {
      constexpr uint32_t idesc_pv = idesc_f16(128, D, ATTN, true);  // fp16 P and bank, or bf16 P and V
      const uint32_t tAcc = tmem + Lay::kAccCol;
      bool ok = true;
      for (int kt = 0; ok && kt < nk; ++kt) {
        const int b = kt % kBufS;
        if (!(ok = wait_or_abort(FEM_BAR(kBarPFull + b), (kt / kBufS) & 1, err, kErrWaitMma, abort_flag))) break;
        // each bank of the tile into its accumulator, D columns apart; the
        // beta bank of a split diagonal tile into its own buffer
#pragma unroll
        for (int part = 0; part < kNB; ++part) {
          const int e = kt * kNB + part, st = e % kSlotsE;
          if (!(ok = wait_or_abort(FEM_BAR(kBarEFull + st), (e / kSlotsE) & 1, err, kErrWaitTma, abort_flag))) break;
          tc_fence_after_sync();
          const uint32_t sE = sbase + Lay::kE + st * Lay::kTile;
          const bool to_diag = split && kt == nk - 1 && part == kNB - 1;
          // the diagonal tile's buffer was last read by the P E of tile nk - kBufS
          if (to_diag && nk >= kBufS &&
              !(ok = wait_or_abort(FEM_BAR(kBarPvDone + nk % kBufS), ((nk - kBufS) / kBufS) & 1, err, kErrWaitMma,
                                   abort_flag)))
            break;
          const uint32_t dst = to_diag ? tDiag : tAcc + part * D;
#pragma unroll
          for (int kk = 0; kk < kBlockK / 16; ++kk)
            mma_f16_ts(dst, tmem + b * 128 + kk * 8, smem_desc_sw128(sE + kk * 2048, 16384, 1024), idesc_pv,
                       ((kt > 0 && !to_diag) || kk > 0) ? 1u : 0u);
          mma_commit(FEM_BAR(kBarEEmpty + st));
        }
        if (!ok) break;
        mma_commit(FEM_BAR(kBarPvDone + b));
      }
      mma_commit(FEM_BAR(kBarAccDone));  // completes once everything this thread issued is done
    }
  }
  } else {
    // ---------------------------------------------------------------- softmax (warpgroup 1) or
    // correction (warpgroup 2), then the epilogue, which both run as one code path
    const bool is_sm = wg == 1;
    const int r = (tid - 128) & 127;  // row within the tile
    const int t_row = qt * kBlockQ + r;
    const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t tAcc = tmem + Lay::kAccCol + lane_off;  // every accumulator column
    const uint32_t tAccB = tmem + Lay::kAccB + lane_off;   // the beta read's
    const uint32_t tDiagL = tDiag + lane_off;
    float *s_alpha = reinterpret_cast<float *>(smem + Lay::kAlpha);
    float *s_invL = reinterpret_cast<float *>(smem + Lay::kInvL);
    float2 *s_pre = reinterpret_cast<float2 *>(smem + Lay::kPre);
    float4 *s_gco = reinterpret_cast<float4 *>(smem + Lay::kGco);
    unsigned *s_flag = reinterpret_cast<unsigned *>(smem + Lay::kFlag);  // [128][4]
    unsigned *s_bad = reinterpret_cast<unsigned *>(smem + Lay::kBad);
    int *s_misc = reinterpret_cast<int *>(smem + Lay::kMisc);
    float m_row = -INFINITY, L_row = 0.f;
    bool ok = true;
    if (is_sm) {
      // ------------------------------------------------------------ softmax
      const float qk_scale = kLog2e * rsqrtf(static_cast<float>(D));
      for (int kt = 0; kt < nk; ++kt) {
        const int b = kt % kBufS;
        const uint32_t tS = tmem + b * 128 + lane_off;
        // every lane takes the same branch: the wait's outcome is made warp-uniform
        ok = __all_sync(0xffffffffu,
                        wait_or_abort(FEM_BAR(kBarSFull + b), (kt / kBufS) & 1, err, kErrWaitMma, abort_flag));
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
        for (int u = 0; u < 8; ++u) mx[u] = fmax3(s[u], s[u + 8], s[u + 16]);
#pragma unroll
        for (int n = 24; n < 120; n += 16)
#pragma unroll
          for (int u = 0; u < 8; ++u) mx[u] = fmax3(mx[u], s[n + u], s[n + 8 + u]);
#pragma unroll
        for (int u = 0; u < 8; ++u) mx[u] = fmaxf(mx[u], s[120 + u]);
        float tmax = fmax3(fmax3(mx[0], mx[1], mx[2]), fmax3(mx[3], mx[4], mx[5]), fmaxf(mx[6], mx[7]));
        tmax *= qk_scale;  // log2-domain row maximum of this tile
        float alpha = 1.f;
        const float m_old = m_row;
        if (tmax > m_row + kRowMaxLag) {
          alpha = ex2_approx(m_row - tmax);  // 0 on the first tile
          m_row = tmax;
        }
        s_alpha[b * 128 + r] = alpha;
        mbar_arrive(FEM_BAR(kBarAlpha + b));
        if (kt == nk - 1) s_pre[r] = make_float2(m_old, L_row);  // the row's state before its last key tile
        // P = exp2(s * scale - m) as fp16 over the first 64 columns of the buffer; L from the fp32 values
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
            p[i] = ATTN ? pack_bf162(e.x, e.y) : pack_half2(e.x, e.y);
          }
          tmem_st16(tS + c * 16, p);
        }
        const float lsum = (ls[0].x + ls[0].y) + (ls[1].x + ls[1].y) + (ls[2].x + ls[2].y) + (ls[3].x + ls[3].y);
        L_row = L_row * alpha + lsum;
        tmem_st_wait();
        tc_fence_before_sync();
        mbar_arrive(FEM_BAR(kBarPFull + b));
      }
      s_invL[r] = 1.f / L_row;
      reinterpret_cast<float *>(smem + Lay::kInvLT)[(r & 3) * 32 + (r >> 2)] = 1.f / L_row;
      if (ok && lse && t_row < T) lse[static_cast<size_t>(bh) * T + t_row] = (m_row + lg2_approx(L_row)) * kLn2;
    }
    else {
      // ------------------------------------------------------------ correction
      // thread j < D: channel j's sum of |bank| over the key tiles read so far,
      // in the units of the current shift (and the mean bank's, GATED), and
      // the same before the diagonal tile
      float ecol = 0.f, ecol_pre = 0.f, ecol0 = 0.f;
      // channel r's epilogue coefficients, loaded now and stored after the loop
      // (the epilogue is the first reader): the bank's mode and anchor, the last
      // shift, beta and, GATED, the mean's anchor
      ChanInfo ci_r = {0.f, 1.f};
      float beta_r = 0.f, shift_r = 0.f, c0_r = 0.f;
      if (!ATTN && r < D) {
        ci_r = w.chan[bh * D + r];
        beta_r = beta[h * D + r];
        shift_r = w.shift[(static_cast<size_t>(bh) * n_kt_all + nk - 1) * D + r];
        if (GATED) c0_r = gate.chan0[bh * D + r].c_lin;
      }
      for (int kt = 0; kt < nk; ++kt) {
        const int b = kt % kBufS;
        ok = __all_sync(0xffffffffu,
                        wait_or_abort(FEM_BAR(kBarAlpha + b), (kt / kBufS) & 1, err, kErrWaitMma, abort_flag));
        if (!ok) break;
        const float alpha = s_alpha[b * 128 + r];
        // (colmv, some channel's shift moved at this tile, comes with the side data below)
        const bool rowmv = __any_sync(0xffffffffu, alpha != 1.f);
        const bool last_split = split && kt == nk - 1;  // acc keeps its state; the epilogue rescales
        // this tile's rescale factors exp(beta_j (c_old - c_new)), 1 for unmoved
        // channels, its column sums and its moved-channel mask, loaded tiles
        // ahead with K
        const float *rf =
            reinterpret_cast<const float *>(smem + Lay::kSide + (kt % Lay::kSideStages) * Lay::kSideStride);
        if (!ATTN) {
          ok = __all_sync(0xffffffffu, wait_or_abort(FEM_BAR(kBarSide + kt % Lay::kSideStages),
                                                     (kt / Lay::kSideStages) & 1, err, kErrWaitTma, abort_flag));
        }
        if (!ok) break;
        bool colmv = false;
        if (!ATTN) {
          const uint4 m4 = *reinterpret_cast<const uint4 *>(rf + Lay::kSideMask / 4);
          colmv = (m4.x | m4.y | m4.z | m4.w) != 0u;
        }
        if (!ATTN && r < D) {
          if (last_split) ecol_pre = ecol;
          ecol = fmaf(ecol, rf[r], rf[D + r]);
          if (GATED) ecol0 += rf[2 * D + r];
        }
        const bool do_b = !last_split && (rowmv || colmv);  // the beta accumulator needs a rescale
        const bool do_m = GATED && rowmv;                    // the mean's accumulator
        if (kt > 0 && (do_b || do_m)) {
          unsigned gm = 0;  // 32-column groups holding a moved channel
          int g0 = 0;
          float f0[32];  // factors of the first such group, read before acc is ready
          if (colmv && do_b) {
            const uint4 m4 = *reinterpret_cast<const uint4 *>(rf + Lay::kSideMask / 4);
            gm = (m4.x ? 1u : 0u) | (m4.y ? 2u : 0u) | (m4.z ? 4u : 0u) | (m4.w ? 8u : 0u);
            g0 = __ffs(gm) - 1;
#pragma unroll
            for (int i = 0; i < 32; ++i) f0[i] = rf[g0 * 32 + i];
          }
          // acc is final for tile kt-1 once its P E completed
          const int pb = (kt - 1) % kBufS;
          ok = __all_sync(0xffffffffu, wait_or_abort(FEM_BAR(kBarPvDone + pb), ((kt - 1) / kBufS) & 1, err,
                                                     kErrWaitMma, abort_flag));
          if (!ok) break;
          tc_fence_after_sync();
          if (do_m) {
            // the mean's accumulator: the row maximum's factor only
#pragma unroll 1
            for (int c = 0; c < D / 32; ++c) {
              uint32_t v[32];
              tmem_ld32(tAcc + c * 32, v);
              tmem_ld_wait();
#pragma unroll
              for (int i = 0; i < 32; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) * alpha);
              tmem_st32(tAcc + c * 32, v);
            }
          }
          if (do_b && rowmv) {
#pragma unroll 1
            for (int c = 0; c < D / 32; ++c) {
              uint32_t v[32];
              tmem_ld32(tAccB + c * 32, v);
              tmem_ld_wait();
              if (colmv) {
#pragma unroll
                for (int i = 0; i < 32; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) * alpha * rf[c * 32 + i]);
              } else {
#pragma unroll
                for (int i = 0; i < 32; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) * alpha);
              }
              tmem_st32(tAccB + c * 32, v);
            }
          } else if (do_b && colmv) {
            {
              uint32_t v[32];
              tmem_ld32(tAccB + g0 * 32, v);
              tmem_ld_wait();
#pragma unroll
              for (int i = 0; i < 32; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) * f0[i]);
              tmem_st32(tAccB + g0 * 32, v);
            }
#pragma unroll 1
            for (int c = g0 + 1; c < D / 32; ++c) {
              if (!((gm >> c) & 1u)) continue;
              uint32_t v[32];
              tmem_ld32(tAccB + c * 32, v);
              float f[32];
#pragma unroll
              for (int i = 0; i < 32; ++i) f[i] = rf[c * 32 + i];
              tmem_ld_wait();
#pragma unroll
              for (int i = 0; i < 32; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) * f[i]);
              tmem_st32(tAccB + c * 32, v);
            }
          }
          tmem_st_wait();
        }
        tc_fence_before_sync();
        mbar_arrive(FEM_BAR(kBarPFull + b));
      }
      // the guard's coefficients of channel j: an entry is rejected when
      //   X a + Z / L < Y          (final state, a = acc / L)
      //   X a_pre + Zp < Y L_pre   (state before the diagonal tile)
      // with X = tau beta, Z = -2^-25 Ecol, Zp = -2^-25 Ecol_pre and Y = 2^-25
      // (shifted bank) or -tau (linear bank); see kGuardTau
      if (r < D) {
        if (ATTN) {
          c_coef[r] = make_float4(0.f, 0.f, 0.f, 0.f);  // o = acc / L: the linear form at beta = 0 around 0
        } else if (ci_r.linear != 0.f) {
          c_coef[r] = make_float4(beta_r, ci_r.c_lin, beta_r != 0.f ? kLn2 / beta_r : 0.f, 0.f);
        } else {
          c_coef[r] = make_float4(0.f, shift_r - kBankOffset / beta_r, kLn2 / beta_r, 1.f);
        }
        // the mean's anchor: its bank holds v - c, so mu = c + acc/L
        if (GATED) reinterpret_cast<float *>(c_coef + D)[r] = c0_r;
      }
      if (!ATTN && r < D) {
        const bool lin = ci_r.linear != 0.f;
        const float4 g = make_float4(kGuardTau * beta_r, -kGuardUlp * ecol, lin ? -kGuardTau : kGuardUlp, -kGuardUlp * ecol_pre);
        s_gco[r] = g;
        // the same test on the final state as a < A + B / L: A = Y / X, B = -Z / X for
        // X > 0; at beta = 0 (X = 0, linear) it holds for no L >= 1 unless -Z > tau,
        // in which case every entry of the channel goes to the exact test
        reinterpret_cast<float2 *>(smem + Lay::kThr)[r] =
            g.x > 0.f ? make_float2(g.z / g.x, -g.y / g.x) : make_float2(-g.y > kGuardTau ? INFINITY : -INFINITY, 0.f);
        // the mean bank (linear, beta = 0): rejected when 2^-25 Ecol0 / L > tau;
        // the CTA keeps the largest 2^-25 Ecol0 (positive floats order as integers)
        if (GATED) atomicMax(reinterpret_cast<int *>(smem + Lay::kMisc) + 4, __float_as_int(kGuardUlp * ecol0));
      }
    }
    // ---- epilogue, half the channels per warpgroup.  acc/L is staged in
    // shared memory (the K and E rings are idle once every contraction
    // completed) as 32-column boxes, row r by thread r, and checked by the
    // underflow guard; the transform then runs column-parallel and writes each
    // row's 32 columns of a box as one coalesced 128-byte store.  GATED: boxes
    // 0 .. D/32-1 hold the mean's accumulator, boxes D/32 .. 2D/32-1 the
    // beta_max read's.
    if (ok) ok = __all_sync(0xffffffffu, wait_or_abort(FEM_BAR(kBarAccDone), 0, err, kErrWaitMma, abort_flag));
    ok = bar_and(1, 256, ok);  // both warpgroups went through every key tile
    if (ok) {
      tc_fence_after_sync();
      const float invL = s_invL[r];
      constexpr int NC = D / 64;             // 32-column chunks of this warpgroup
      constexpr int kBoxB = (kNB - 1) * (D / 32);  // first box of the beta read
      const int c_lo = is_sm ? 0 : NC;
      // GATED: the mean bank's guard for the whole row (its bound is per channel;
      // the largest one stands for all)
      const float mean_bound = GATED ? reinterpret_cast<const float *>(smem + Lay::kMisc)[4] : 0.f;
      const bool mean_bad = GATED && mean_bound * invL > kGuardTau;
      const float2 pre = s_pre[r];  // (m, L) before the last key tile
      const float alpha_last = split ? s_alpha[((nk - 1) % kBufS) * 128 + r] : 1.f;
      const float *rf_last =
          reinterpret_cast<const float *>(smem + Lay::kSide + ((nk - 1) % Lay::kSideStages) * Lay::kSideStride);
      unsigned bad = 0;  // a rejected entry whose state before the diagonal tile is rejected too
      const float2 *s_ab = reinterpret_cast<const float2 *>(smem + Lay::kThr);
      if (GATED) {
        uint32_t v[NC][32];
#pragma unroll
        for (int c = 0; c < NC; ++c) tmem_ld32(tAcc + (c_lo + c) * 32, v[c]);
        tmem_ld_wait();
#pragma unroll
        for (int c = 0; c < NC; ++c) {
          uint8_t *box = smem + Lay::kK + (c_lo + c) * 16384;  // 128 rows x 32 fp32, 128-byte swizzle
#pragma unroll
          for (int i4 = 0; i4 < 8; ++i4)
            *reinterpret_cast<float4 *>(box + sw128_offset(r, i4)) =
                make_float4(__uint_as_float(v[c][4 * i4]) * invL, __uint_as_float(v[c][4 * i4 + 1]) * invL,
                            __uint_as_float(v[c][4 * i4 + 2]) * invL, __uint_as_float(v[c][4 * i4 + 3]) * invL);
        }
      }
      // chunk by chunk: acc (before the diagonal tile when split) times the
      // diagonal tile's factors, alpha of the row and exp(beta (c_old - c_new))
      // of the channel (both exactly 1 unless the row maximum or the channel's
      // shift moved on it), plus the diagonal tile's P E, over L, staged
#pragma unroll 1
      for (int c = c_lo; c < c_lo + NC; ++c) {
        uint32_t va[32], vd[32];
        tmem_ld32(tAccB + c * 32, va);
        if (split) {
          tmem_ld32(tDiagL + c * 32, vd);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i)
            vd[i] = __float_as_uint(fmaf(__uint_as_float(va[i]), alpha_last * rf_last[c * 32 + i], __uint_as_float(vd[i])));
        } else {
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i) vd[i] = va[i];
        }
        uint8_t *box = smem + Lay::kK + (kBoxB + c) * 16384;
#pragma unroll
        for (int i4 = 0; i4 < 8; ++i4)
          *reinterpret_cast<float4 *>(box + sw128_offset(r, i4)) =
              make_float4(__uint_as_float(vd[4 * i4]) * invL, __uint_as_float(vd[4 * i4 + 1]) * invL,
                          __uint_as_float(vd[4 * i4 + 2]) * invL, __uint_as_float(vd[4 * i4 + 3]) * invL);
      }
      bar_sync(4, 256);  // every box is staged
      // Thread r takes column r % 32 of a chunk and rows r / 32 + 4k, so its
      // channel's coefficients stay in registers, each warp access is one
      // 128-byte row of the box, and 8 loads at a time are in flight before the math.
      //   shifted bank: c + (log a - kappa)/beta = lg2(a) ln2/beta + (c - kappa/beta)
      //   linear bank:  c + log1p(x)/beta with x = beta a, as lg2(1 + x) ln2/beta + c,
      //                 or, for |x| < 2^-6 (also beta = 0), as c + a times the
      //                 series of log1p(x)/x
      // GATED: mu = c_mean + a_mean, F the beta_max read as above, and
      // o = g (mu + lambda (F - mu)).  The underflow guard's test a < A + B / L
      // runs here too, thread per channel with A, B in registers; rows with a
      // candidate entry are marked for the exact test after the transform.
      const int col = r & 31, row0 = r >> 5;
      const int rows_left = T - qt * kBlockQ;
      const size_t tile_off = (static_cast<size_t>(bh) * T + static_cast<size_t>(qt) * kBlockQ) * D + col;
      float *out_tile = out + tile_off;
#pragma unroll 1
      for (int c = c_lo; c < c_lo + NC; ++c) {
        const float4 cf = c_coef[c * 32 + col];
        const float c_mean = GATED ? reinterpret_cast<const float *>(c_coef + D)[c * 32 + col] : 0.f;
        const float2 thr = ATTN ? make_float2(0.f, 0.f) : s_ab[c * 32 + col];
        const bool lin = cf.w == 0.f;
        // pairs of rows go through the packed fp32x2 pipe; the lg2 argument is
        // a (shifted) or 1 + beta a (linear)
        const float2 bx2 = make_float2(cf.x, cf.x), y2 = make_float2(cf.y, cf.y), z2 = make_float2(cf.z, cf.z);
        const float2 s12 = lin ? bx2 : make_float2(1.f, 1.f), s02 = make_float2(lin ? 1.f : 0.f, lin ? 1.f : 0.f);
        const uint8_t *box = smem + Lay::kK + (kBoxB + c) * 16384 + ((col & 3) << 2);
        const uint8_t *box_m = smem + Lay::kK + c * 16384 + ((col & 3) << 2);
#pragma unroll 1
        for (int k0 = 0; k0 < 32; k0 += 8) {
          float a[8];
#pragma unroll
          for (int k = 0; k < 8; ++k)
            a[k] = *reinterpret_cast<const float *>(box + sw128_offset(row0 + 4 * (k0 + k), col >> 2));
          // GATED: the 8 rows' gates, in flight together with the math below
          // (rows past T read the tile's last row and are not stored)
          float lamv[8], gv[8];
          if (GATED) {
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              const size_t oi =
                  tile_off + static_cast<size_t>(min(row0 + 4 * (k0 + k), rows_left - 1)) * D + c * 32;
              lamv[k] = __ldcs(gate.lam + oi);
              gv[k] = __ldcs(gate.g + oi);
            }
          }
          // the guard's quick test on the 8 rows (row0 + 4 (k0 + k) lies in word k0 / 8, bit row0 + 4 k)
          if (!ATTN) {
            const float4 il0 = *reinterpret_cast<const float4 *>(smem + Lay::kInvLT + (row0 * 32 + k0) * 4);
            const float4 il1 = *reinterpret_cast<const float4 *>(smem + Lay::kInvLT + (row0 * 32 + k0 + 4) * 4);
            const float il[8] = {il0.x, il0.y, il0.z, il0.w, il1.x, il1.y, il1.z, il1.w};
            // two rows per packed fma; the rows' own marks only when some entry of the batch is a candidate
            bool anyc = false;
#pragma unroll
            for (int k = 0; k < 8; k += 2) {
              const float2 t2 = __ffma2_rn(make_float2(thr.y, thr.y), make_float2(il[k], il[k + 1]),
                                           make_float2(thr.x, thr.x));
              anyc = anyc || a[k] < t2.x || a[k + 1] < t2.y;
              if (GATED) anyc = anyc || mean_bound * fmaxf(il[k], il[k + 1]) > kGuardTau;
            }
            if (__any_sync(0xffffffffu, anyc)) {
              unsigned cm = 0;
#pragma unroll
              for (int k = 0; k < 8; ++k) {
                bool cnd = a[k] < fmaf(thr.y, il[k], thr.x);
                if (GATED) cnd = cnd || mean_bound * il[k] > kGuardTau;
                cm |= (cnd && row0 + 4 * (k0 + k) < rows_left) ? 1u << (row0 + 4 * k) : 0u;
              }
              cm = __reduce_or_sync(0xffffffffu, cm);
              if (cm && lane == 0) atomicOr(reinterpret_cast<unsigned *>(smem + Lay::kMisc) + 20 + (k0 >> 3), cm);
            }
          }
          float o[8];
#pragma unroll
          for (int k = 0; k < 8; k += 2) {
            const float2 a2 = make_float2(a[k], a[k + 1]);
            const float2 x2 = __fmul2_rn(bx2, a2);
            const float2 g2 = __ffma2_rn(a2, s12, s02);
            const float2 lg = __ffma2_rn(make_float2(lg2_approx(g2.x), lg2_approx(g2.y)), z2, y2);
            float2 q = __ffma2_rn(x2, make_float2(0.2f, 0.2f), make_float2(-0.25f, -0.25f));
            q = __ffma2_rn(x2, q, make_float2(1.f / 3.f, 1.f / 3.f));
            q = __ffma2_rn(x2, q, make_float2(-0.5f, -0.5f));
            q = __ffma2_rn(x2, q, make_float2(1.f, 1.f));
            const float2 se = __ffma2_rn(a2, q, y2);
            o[k] = (lin && fabsf(x2.x) < 0.015625f) ? se.x : lg.x;
            o[k + 1] = (lin && fabsf(x2.y) < 0.015625f) ? se.y : lg.y;
          }
          if (GATED) {
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              const float mu =
                  c_mean + *reinterpret_cast<const float *>(box_m + sw128_offset(row0 + 4 * (k0 + k), col >> 2));
              o[k] = gv[k] * fmaf(lamv[k], o[k] - mu, mu);
            }
          }
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const int row = row0 + 4 * (k0 + k);
            if (row < rows_left) __stcs(out_tile + static_cast<size_t>(row) * D + c * 32, o[k]);
          }
        }
      }
      // ---- the exact guard on the marked rows, row r by thread r: a rejected
      // entry's accumulator before the diagonal tile replaces its output (the
      // fix-up's starting state; GATED: its mu goes to the gate's side buffer),
      // and whether that state passes the guard too decides where the fix-up starts
      bar_sync(4, 256);  // the transform's stores and marks are complete
      const unsigned *rowcand = reinterpret_cast<const unsigned *>(smem + Lay::kMisc) + 20;
      if ((rowcand[0] | rowcand[1] | rowcand[2] | rowcand[3]) != 0u) {
        const bool cand = (rowcand[r >> 5] >> (r & 31)) & 1u;
        if (__any_sync(0xffffffffu, cand)) {
#pragma unroll 1
          for (int c = c_lo; c < c_lo + NC; ++c) {
            uint32_t vp[32];
            tmem_ld32(tAccB + c * 32, vp);
            tmem_ld_wait();
            unsigned fm = 0;
            if (cand) {
              const uint8_t *box = smem + Lay::kK + (kBoxB + c) * 16384;
              const float4 *gco = s_gco + c * 32;
              const size_t orow = (static_cast<size_t>(bh) * T + t_row) * D + c * 32;
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                const float cell = *(reinterpret_cast<const float *>(box + sw128_offset(r, i >> 2)) + (i & 3));
                const float4 g = gco[i];
                const float2 t = s_ab[c * 32 + i];
                if (!(mean_bad || cell < fmaf(t.y, invL, t.x))) continue;
                fm |= 1u << i;
                const float a_pre = split ? __uint_as_float(vp[i]) : 0.f;
                if (split && fmaf(g.x, a_pre, g.w) < g.z * pre.y) bad = 1;
                out[orow + i] = a_pre;
                if (GATED)
                  gate.mu_side[orow + i] =
                      reinterpret_cast<const float *>(c_coef + D)[c * 32 + i] +
                      *(reinterpret_cast<const float *>(smem + Lay::kK + c * 16384 + sw128_offset(r, i >> 2)) + (i & 3));
              }
            }
            s_flag[r * 4 + c] = fm;
            if (fm) atomicOr(reinterpret_cast<unsigned *>(smem + Lay::kMisc) + 16 + (r >> 5), 1u << (r & 31));
          }
        } else {
#pragma unroll
          for (int c = c_lo; c < c_lo + NC; ++c) s_flag[r * 4 + c] = 0u;
        }
        if (bad) atomicOr(s_bad + r, 1u);
        bar_sync(4, 256);
      }
      // ---- list the rejected rows: one block of entries that restart from the
      // diagonal tile, one of entries recomputed over every key tile, each padded
      // to a multiple of kFixChunk rows (rows -1) for the fix-up's chunks
      const unsigned *rowflags = reinterpret_cast<const unsigned *>(smem + Lay::kMisc) + 16;
      const bool any_listed = (rowflags[0] | rowflags[1] | rowflags[2] | rowflags[3]) != 0u;
      int base = 0;  // thread 0 of the softmax warpgroup: the first reserved slot
      if (any_listed && is_sm) {
        const bool listed = (rowflags[r >> 5] >> (r & 31)) & 1u;
        const bool diag = listed && split && s_bad[r] == 0u;
        const unsigned bd = __ballot_sync(0xffffffffu, diag), bf = __ballot_sync(0xffffffffu, listed && !diag);
        if (lane == 0) {
          s_misc[8 + (warp & 3)] = __popc(bd);
          s_misc[12 + (warp & 3)] = __popc(bf);
        }
        bar_sync(2, 128);
        if (r == 0) {
          int nd = 0, nf = 0;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            nd += s_misc[8 + q];
            nf += s_misc[12 + q];
          }
          base = atomicAdd(w.fixup_count, pad_chunk(nd) + pad_chunk(nf));
          atomicAdd(w.fixup_rows, nd + nf);
        }
      }
      // ---- the listed rows' entries, in the reserved slots
      if (any_listed && is_sm) {
        if (r == 0) s_misc[0] = base;
        bar_sync(2, 128);
        const int b0 = s_misc[0], wq = warp & 3;
        int nd = 0, nf = 0, pd = 0, pf = 0;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int a = s_misc[8 + q], b = s_misc[12 + q];
          nd += a;
          nf += b;
          pd += q < wq ? a : 0;
          pf += q < wq ? b : 0;
        }
        const int sd = pad_chunk(nd), sf = pad_chunk(nf);
        const bool listed = (rowflags[r >> 5] >> (r & 31)) & 1u;
        const bool diag = listed && split && s_bad[r] == 0u;
        const unsigned bd = __ballot_sync(0xffffffffu, diag), bf = __ballot_sync(0xffffffffu, listed && !diag);
        const unsigned below = (1u << lane) - 1u;
        if (listed) {
          const float2 pr = s_pre[r];
          FixupEntry e;
          e.row = bh * T + t_row;
#pragma unroll
          for (int g = 0; g < 4; ++g) e.mask[g] = g < D / 32 ? s_flag[r * 4 + g] : 0u;
          e.m_pre = pr.x;
          e.l_pre = pr.y;
          e.kt0 = diag ? nk - 1 : 0;
          // a recomputation from the first key tile keeps the mean the kernel
          // left aside unless the mean bank's own guard rejected it (l_pre = 1)
          if (!diag)
            e.l_pre = (GATED && reinterpret_cast<const float *>(smem + Lay::kMisc)[4] * s_invL[r] > kGuardTau) ? 1.f
                                                                                                                : 0.f;
          w.fixups[diag ? b0 + pd + __popc(bd & below) : b0 + sd + pf + __popc(bf & below)] = e;
        }
        FixupEntry padding;
        padding.row = -1;
        padding.mask[0] = padding.mask[1] = padding.mask[2] = padding.mask[3] = 0u;
        padding.m_pre = -INFINITY;
        padding.l_pre = 0.f;
        if (r < sd - nd) {
          padding.kt0 = nk - 1;
          w.fixups[b0 + nd + r] = padding;
        }
        if (r < sf - nf) {
          padding.kt0 = 0;
          w.fixups[b0 + sd + nf + r] = padding;
        }
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

template <int D, bool GATED, bool ATTN = false>
static cudaError_t launch_tc_d(const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &te,
                               const CUtensorMap &te0, float *out, const float *beta, const BankWorkspace &w,
                               float *lse, int BH, int H, int T, int causal, const TcGate &gate, unsigned *err,
                               cudaStream_t stream, bool pdl) {
  using Lay = TcLayout<D, GATED>;
  const int n_qt = (T + kBlockQ - 1) / kBlockQ;
  if (n_qt > Lay::kMaxKeyTiles || BH > 65535) return cudaErrorInvalidValue;
  const uint32_t smem = Lay::kAlloc;
  cudaError_t e =
      cudaFuncSetAttribute(fem_tc_kernel<D, GATED, ATTN>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  e = launch_kernel(fem_tc_kernel<D, GATED, ATTN>, dim3(n_qt, BH), dim3(384), smem, stream, pdl, tq, tk, te, te0, out,
                    beta, w, lse, H, T, causal, gate, err);
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_tc(int d, const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &te,
                      const CUtensorMap *te0, float *out, const float *beta, const BankWorkspace &w, float *lse,
                      int BH, int H, int T, int causal, const TcGate *gate, unsigned *err, cudaStream_t stream,
                      bool pdl) {
  const TcGate none = {nullptr, nullptr, nullptr, nullptr, nullptr};
  if ((te0 != nullptr) != (gate != nullptr)) return cudaErrorInvalidValue;
  if (gate) {
    if (d == 64)
      return launch_tc_d<64, true>(tq, tk, te, *te0, out, beta, w, lse, BH, H, T, causal, *gate, err, stream, pdl);
    if (d == 128)
      return launch_tc_d<128, true>(tq, tk, te, *te0, out, beta, w, lse, BH, H, T, causal, *gate, err, stream, pdl);
    return cudaErrorInvalidValue;
  }
  if (d == 64)
    return launch_tc_d<64, false>(tq, tk, te, te, out, beta, w, lse, BH, H, T, causal, none, err, stream, pdl);
  if (d == 128)
    return launch_tc_d<128, false>(tq, tk, te, te, out, beta, w, lse, BH, H, T, causal, none, err, stream, pdl);
  return cudaErrorInvalidValue;
}

cudaError_t launch_attn(int d, const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &tv, float *out,
                        float *lse, int BH, int H, int T, int causal, unsigned *err, cudaStream_t stream) {
  const TcGate none = {nullptr, nullptr, nullptr, nullptr, nullptr};
  const BankWorkspace w = {};
  if (d == 64)
    return launch_tc_d<64, false, true>(tq, tk, tv, tv, out, nullptr, w, lse, BH, H, T, causal, none, err, stream,
                                        false);
  if (d == 128)
    return launch_tc_d<128, false, true>(tq, tk, tv, tv, out, nullptr, w, lse, BH, H, T, causal, none, err, stream,
                                         false);
  return cudaErrorInvalidValue;
}

}  // namespace fem
