// Tensor-core kernel of the FEM read for bf16 inputs (sm_103a, tcgen05).
//
// One CTA of 128 threads computes a tile of 128 query rows of one (b, h):
//
//   for each key tile of 128 keys (up to the diagonal when causal):
//     TMA    K, V tile -> shared memory (128-byte swizzle)
//     MMA    S = Q K^T -> TMEM (fp32), issued by one thread
//     value  E = bank(V) in place in shared memory, once per key tile:
//            linear channels  D = expm1(beta (v - c)) / beta   (c fixed)
//            shifted channels E = exp(beta (v - c) + kappa)     (c running)
//     row    P = exp(s - m) with a lazily raised row max m, rounded to fp16;
//            L accumulates the rounded P (the same values the MMA sees)
//     rescale acc_{t,j} *= exp(m_old - m_new) * exp(beta_j (c_old - c_new))
//            when a row max or a channel shift moved (joint online rescale)
//     MMA    acc += P E -> TMEM (fp32)
//   epilogue o = c + log1p(beta acc/L)/beta (linear) or
//            o = c + (log(acc/L) - kappa)/beta (shifted); lse = m + log L.
//
// The two contractions are the read's (Sec. 2.3, Eq. "fem-free-energy-main"
// with the softmax prior of App. C): sum_i exp(s_i - m) exp(beta_j (v_ij -
// c_j)) is the numerator of the free energy up to the stabilising shifts,
// and L is its normaliser.  The mixing of one value bank with the shared
// prior weights in one pass follows the one-pass form of App. E ("One-pass
// implementation").
//
// Shared memory (bytes, D = head dim): Q  D*256 | K  D*256 | V/E  D*256 |
// P 32768 | barriers, TMEM address, per-channel state.  Operands use the
// 128-byte swizzle layout TMA writes: 64-element column blocks of 128 rows x
// 128 bytes, 16-byte chunk c of row r stored at chunk c ^ (r & 7).
// TMEM: S in columns [0, 128), acc in [128, 128 + D).
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

template <int D>
struct TcLayout {
  static constexpr uint32_t kTileBytes = D * kBlockK * 2;  // one bf16/fp16 [128 x D] tile
  static constexpr uint32_t kQ = 0;
  static constexpr uint32_t kK = kQ + kTileBytes;
  static constexpr uint32_t kV = kK + kTileBytes;
  static constexpr uint32_t kP = kV + kTileBytes;
  static constexpr uint32_t kMisc = kP + kBlockQ * kBlockK * 2;
  static constexpr uint32_t kBarTma = kMisc;
  static constexpr uint32_t kBarMma = kMisc + 8;
  static constexpr uint32_t kBarQ = kMisc + 16;
  static constexpr uint32_t kTmemSlot = kMisc + 24;
  static constexpr uint32_t kFlags = kMisc + 32;  // [0] abort, [1] column moved
  static constexpr uint32_t kChan = kMisc + 64;   // 6 float arrays of D
  static constexpr uint32_t kBytes = kChan + 6 * D * 4;
  static constexpr uint32_t kAlloc = kBytes + 1024;  // slack for 1024-byte alignment
  static constexpr uint32_t kTmemCols = 256;
};

template <int D>
__global__ void __launch_bounds__(128, 1)
    fem_tc_kernel(const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_k,
                  const __grid_constant__ CUtensorMap tmap_v, const float *__restrict__ beta,
                  const ChanInfo *__restrict__ chan, const float *__restrict__ cpre, float *__restrict__ out,
                  float *__restrict__ lse, int H, int T, int causal, unsigned *__restrict__ err) {
  using Lay = TcLayout<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sQ = sbase + Lay::kQ, sK = sbase + Lay::kK, sV = sbase + Lay::kV, sP = sbase + Lay::kP;
  const uint32_t bar_tma = sbase + Lay::kBarTma, bar_mma = sbase + Lay::kBarMma, bar_q = sbase + Lay::kBarQ;
  volatile int *flags = reinterpret_cast<volatile int *>(smem + Lay::kFlags);
  float *c_beta = reinterpret_cast<float *>(smem + Lay::kChan);  // beta_j
  float *c_lin = c_beta + D;                                     // 1 = linear bank
  float *c_shift = c_lin + D;                                    // current c_j
  float *c_ea = c_shift + D;  // shifted bank: E = ex2(ea v + eb); linear bank: ea = 1/beta
  float *c_eb = c_ea + D;
  float *c_r = c_eb + D;  // column rescale factor of this key tile

  const int tid = threadIdx.x, warp = tid >> 5;
  const int n_qt = (T + kBlockQ - 1) / kBlockQ;
  const int n_kt_all = (T + kBlockK - 1) / kBlockK;
  const int qt = n_qt - 1 - static_cast<int>(blockIdx.x);  // heaviest causal tiles first
  const int bh = blockIdx.y, h = bh % H;
  const int t0 = qt * kBlockQ;
  const int n_kt = causal ? qt + 1 : n_kt_all;
  const int t_row = t0 + tid;

  if (warp == 0) {
    tmem_alloc(sbase + Lay::kTmemSlot, Lay::kTmemCols);
    tmem_relinquish();
  }
  if (tid == 0) {
    mbar_init(bar_tma, 1);
    mbar_init(bar_mma, 1);
    mbar_init(bar_q, 1);
    fence_mbar_init();
    flags[0] = 0;
    flags[1] = 0;
    prefetch_tensormap(&tmap_q);
    prefetch_tensormap(&tmap_k);
    prefetch_tensormap(&tmap_v);
  }
  if (tid < D) {
    const ChanInfo ci = chan[bh * D + tid];
    c_beta[tid] = beta[h * D + tid];
    c_lin[tid] = ci.linear;
    c_shift[tid] = ci.linear != 0.f ? ci.c_lin : -INFINITY;
    c_ea[tid] = c_beta[tid] > 0.f ? 1.f / c_beta[tid] : 0.f;
    c_r[tid] = 1.f;
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(smem + Lay::kTmemSlot);
  const uint32_t lane_off = static_cast<uint32_t>(warp * 32) << 16;
  const uint32_t tS = tmem, tAcc = tmem + 128;

  uint32_t tma_phase = 0, mma_phase = 0;
  if (tid == 0) {
    mbar_arrive_expect_tx(bar_q, Lay::kTileBytes);
#pragma unroll
    for (int b = 0; b < D / 64; ++b) tma_load_3d(sQ + b * 16384, &tmap_q, bar_q, b * 64, t0, bh);
  }

  constexpr uint32_t idesc_qk = idesc_f16(128, 128, true, false);
  constexpr uint32_t idesc_pv = idesc_f16(128, D, false, true);
  const float qk_scale = kLog2e * rsqrtf(static_cast<float>(D));  // log2-domain score scale
  float m_row = -INFINITY, L_row = 0.f;

  for (int kt = 0; kt < n_kt; ++kt) {
    // ---- [A] K, V tile in flight; per-channel shift schedule for this tile
    if (tid == 0) {
      mbar_arrive_expect_tx(bar_tma, 2 * Lay::kTileBytes);
#pragma unroll
      for (int b = 0; b < D / 64; ++b) tma_load_3d(sK + b * 16384, &tmap_k, bar_tma, b * 64, kt * kBlockK, bh);
#pragma unroll
      for (int b = 0; b < D / 64; ++b) tma_load_3d(sV + b * 16384, &tmap_v, bar_tma, b * 64, kt * kBlockK, bh);
    }
    if (tid < D) {
      const int j = tid;
      float r = 1.f;
      if (c_lin[j] == 0.f) {
        const float b = c_beta[j];
        const float cp = cpre[(static_cast<size_t>(bh) * n_kt_all + kt) * D + j];
        float cur = c_shift[j];
        if (cur == -INFINITY) {
          cur = cp;  // first tile: acc is not yet written
        } else if (b * (cp - cur) > kShiftLag) {
          r = expf(b * (cur - cp));
          cur = cp;
        }
        c_shift[j] = cur;
        c_ea[j] = b * kLog2e;
        c_eb[j] = (kBankOffset - b * cur) * kLog2e;
      }
      c_r[j] = r;
      if (r != 1.f) flags[1] = 1;
    }
    // Q (first pass) and this tile's K, V
    if (kt == 0 && !mbar_wait(bar_q, 0, err, kErrWaitTma)) flags[0] = 1;
    if (!mbar_wait(bar_tma, tma_phase, err, kErrWaitTma)) flags[0] = 1;
    tma_phase ^= 1;
    __syncthreads();
    if (flags[0]) break;

    // ---- [B] S = Q K^T on the tensor cores; value bank in place meanwhile
    if (tid == 0) {
      tc_fence_after_sync();
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint32_t off = (kk >> 2) * 16384 + (kk & 3) * 32;
        mma_f16_ss(tS, smem_desc_sw128(sQ + off, 16, 1024), smem_desc_sw128(sK + off, 16, 1024), idesc_qk,
                   kk > 0 ? 1u : 0u);
      }
      mma_commit(bar_mma);
    }
    {
      constexpr int kChunks = kBlockK * D / 8;  // 16-byte chunks of the V tile
      for (int c = tid; c < kChunks; c += 128) {
        const int blk = c >> 10, rem = c & 1023, row = rem >> 3, pos = rem & 7;
        const int ch0 = blk * 64 + ((pos ^ (row & 7)) << 3);
        const int key = kt * kBlockK + row;
        uint4 *p = reinterpret_cast<uint4 *>(smem + Lay::kV + blk * 16384 + row * 128 + pos * 16);
        uint4 raw = *p;
        const __nv_bfloat16 *vin = reinterpret_cast<const __nv_bfloat16 *>(&raw);
        __align__(16) __half e[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int j = ch0 + u;
          const float x = __bfloat162float(vin[u]);
          float val;
          if (key >= T) {
            val = 0.f;
          } else if (c_lin[j] != 0.f) {
            // D = expm1(y) / beta with y = beta (v - c) >= -1: a Taylor series of
            // expm1(y)/y for |y| < 1/2 (truncation < 4e-6 relative), e^y - 1 beyond.
            const float xs = x - c_shift[j];
            const float y = c_beta[j] * xs;
            if (fabsf(y) < 0.5f) {
              float poly = fmaf(y, 1.f / 720.f, 1.f / 120.f);
              poly = fmaf(y, poly, 1.f / 24.f);
              poly = fmaf(y, poly, 1.f / 6.f);
              poly = fmaf(y, poly, 0.5f);
              poly = fmaf(y, poly, 1.f);
              val = xs * poly;
            } else {
              val = (ex2_approx(y * kLog2e) - 1.f) * c_ea[j];
            }
          } else {
            val = ex2_approx(fmaf(c_ea[j], x, c_eb[j]));
          }
          e[u] = __float2half_rn(val);
        }
        *p = *reinterpret_cast<const uint4 *>(e);
      }
    }
    fence_proxy_async_smem();
    if (!mbar_wait(bar_mma, mma_phase, err, kErrWaitMma)) flags[0] = 1;
    mma_phase ^= 1;
    tc_fence_after_sync();

    // ---- [C] row softmax of S (thread = row), P -> shared memory as fp16
    float s[128];
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      uint32_t r[32];
      tmem_ld32(tS + lane_off + c * 32, r);
      tmem_ld_wait();
#pragma unroll
      for (int i = 0; i < 32; ++i) s[c * 32 + i] = __uint_as_float(r[i]);
    }
    float tmax = -INFINITY;
#pragma unroll
    for (int n = 0; n < 128; ++n) {
      const int key = kt * kBlockK + n;
      const bool valid = key < T && (!causal || key <= t_row);
      s[n] = valid ? s[n] * qk_scale : -INFINITY;
      tmax = fmaxf(tmax, s[n]);
    }
    float alpha = 1.f;
    if (tmax > m_row + kRowMaxLag) {
      alpha = ex2_approx(m_row - tmax);  // 0 on the first valid tile
      m_row = tmax;
    }
    const bool row_live = m_row != -INFINITY;
    float lsum = 0.f;
#pragma unroll
    for (int c8 = 0; c8 < 16; ++c8) {
      __align__(16) __half pk[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const float pv = row_live ? ex2_approx(s[c8 * 8 + u] - m_row) : 0.f;
        pk[u] = __float2half_rn(pv);
        lsum += __half2float(pk[u]);
      }
      *reinterpret_cast<uint4 *>(smem + Lay::kP + (c8 >> 3) * 16384 + sw128_offset(tid, c8 & 7)) =
          *reinterpret_cast<const uint4 *>(pk);
    }
    L_row = L_row * alpha + lsum;

    // joint online rescale of acc (after the previous P E has completed)
    if (kt > 0 && (__any_sync(0xffffffffu, alpha != 1.f) || flags[1])) {
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(tAcc + lane_off + c * 32, r);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha * c_r[c * 32 + i]);
        tmem_st32(tAcc + lane_off + c * 32, r);
      }
      tmem_st_wait();
    }
    fence_proxy_async_smem();
    tc_fence_before_sync();
    __syncthreads();
    if (tid == 0) flags[1] = 0;
    if (flags[0]) break;

    // ---- [D] acc += P E on the tensor cores
    if (tid == 0) {
      tc_fence_after_sync();
#pragma unroll
      for (int kk = 0; kk < kBlockK / 16; ++kk) {
        const uint32_t aoff = (kk >> 2) * 16384 + (kk & 3) * 32;
        mma_f16_ss(tAcc, smem_desc_sw128(sP + aoff, 16, 1024), smem_desc_sw128(sV + kk * 2048, 16384, 1024),
                   idesc_pv, (kt > 0 || kk > 0) ? 1u : 0u);
      }
      mma_commit(bar_mma);
    }
    if (!mbar_wait(bar_mma, mma_phase, err, kErrWaitMma)) flags[0] = 1;
    mma_phase ^= 1;
    tc_fence_after_sync();
    __syncthreads();
    if (flags[0]) break;
  }

  // ---- epilogue: o = c + (mode-specific log of acc / L) / beta; lse
  if (!flags[0]) {
    const bool store = t_row < T;
    const size_t orow = static_cast<size_t>(bh) * T + t_row;
    const float invL = 1.f / L_row;
#pragma unroll
    for (int c = 0; c < D / 32; ++c) {
      uint32_t r[32];
      tmem_ld32(tAcc + lane_off + c * 32, r);
      tmem_ld_wait();
      if (store) {
        __align__(16) float o[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int j = c * 32 + i;
          const float a = __uint_as_float(r[i]) * invL;
          const float b = c_beta[j];
          float val;
          if (c_lin[j] != 0.f)
            val = b != 0.f ? c_shift[j] + log1pf(b * a) / b : c_shift[j] + a;
          else
            val = c_shift[j] + (logf(a) - kBankOffset) / b;
          o[i] = val;
        }
        float4 *dst = reinterpret_cast<float4 *>(out + orow * D + c * 32);
#pragma unroll
        for (int i = 0; i < 8; ++i) dst[i] = reinterpret_cast<const float4 *>(o)[i];
      }
    }
    if (store && lse) lse[orow] = m_row * kLn2 + logf(L_row);
  }

  tc_fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, Lay::kTmemCols);
  }
}

template <int D>
static cudaError_t launch_tc_d(const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &tv, const float *beta,
                               const ChanInfo *chan, const float *cpre, float *out, float *lse, int BH, int H, int T,
                               int causal, unsigned *err, cudaStream_t stream) {
  const uint32_t smem = TcLayout<D>::kAlloc;
  cudaError_t e = cudaFuncSetAttribute(fem_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const dim3 grid((T + kBlockQ - 1) / kBlockQ, BH);
  fem_tc_kernel<D><<<grid, 128, smem, stream>>>(tq, tk, tv, beta, chan, cpre, out, lse, H, T, causal, err);
  return cudaGetLastError();
}

cudaError_t launch_tc(int d, const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &tv, const float *beta,
                      const ChanInfo *chan, const float *cpre, float *out, float *lse, int BH, int H, int T,
                      int causal, unsigned *err, cudaStream_t stream) {
  if (d == 64) return launch_tc_d<64>(tq, tk, tv, beta, chan, cpre, out, lse, BH, H, T, causal, err, stream);
  if (d == 128) return launch_tc_d<128>(tq, tk, tv, beta, chan, cpre, out, lse, BH, H, T, causal, err, stream);
  return cudaErrorInvalidValue;
}

}  // namespace fem
