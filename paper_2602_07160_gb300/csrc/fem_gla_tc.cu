// FEM over a gated-linear-attention prior, chunked on the tensor cores
// (App. "Gated Linear Attention (GLA) Prior", Eqs. "gla-score-appendix" and
// "gla-assoc"):
//
//   s_t(i) = K_{t,i} <qf_t, kf_i> (i <= t),  K_{t,i} = exp(g_{i+1} + ... + g_t),
//   p_t = s_t / Z_t,  o_{t,j} = (1/beta_j) log sum_i p_t(i) exp(beta_j v_{i,j}).
//
// Two CTAs per (b, h), 32 value channels each, walk the sequence in chunks of
// 128 steps (the score and mask work is repeated in both).  With gamma_t
// the running sum of g inside the chunk (so K_{t,i} = exp(gamma_t - gamma_i) for
// i, t in the chunk and exp(gamma_t) from the chunk start), a chunk is four
// contractions on tcgen05 (kind::f16, bf16 operands, fp32 accumulation in TMEM):
//
//   S     = Qf Kf^T                                  [128 x 128], K = m
//   intra = (S o decay-mask) E^T                     [128 x 48],  K = 128 keys
//   inter = Qf Shat^T                                [128 x 48],  K = m
//   U     = (Kf o exp(gamma_last - gamma_i))^T E^T   [m x 48],    K = 128 keys
//
// E holds, per channel j and key i, the value bank of the chunk; channel 32 is
// the constant 1 that gives the normaliser Z ("A one-pass implementation
// appends a constant channel to values").  Shat is the state, sum over earlier
// keys of K_{.,i} kf_i E_ij, kept in fp32 (the bf16 copy only feeds the
// contraction).  Per channel, two forms of the bank, fixed for the sequence:
//
//   beta_j <  1/4: linear, E = expm1(beta (v - c)) / beta with the anchor c the
//     mean of the values so far, at most 1/beta above their minimum; when c moves
//     to c', the state becomes e^{beta (c - c')} Shat_j + expm1(beta (c - c')) / beta
//     Shat_Z (the constant channel's state), and the read is o = c + log1p(beta num / Z) / beta (c + num / Z at
//     beta = 0);
//   beta_j >= 1/4: shifted, E = exp(beta v - lambda) with lambda the chunk's
//     largest beta v, the state carried as e^{mu} Shat with mu the log of its
//     scale, and the read o = (log num - log Z) / beta with log num the
//     log-sum-exp of the chunk's and the state's parts.
//
// The bf16 operands' relative error (2^-9) reaches o as about 2^-9 |v - c| (linear)
// or 2^-9 / beta (shifted), the same order as the bf16 softmax read's.  A shifted
// channel's in-chunk sum for row t uses the chunk's largest value as its shift,
// which may come after t; when that sum falls below 2^-100 of the row's in-chunk
// prior mass (terms under fp32's range could then carry it) the entry is
// recomputed exactly from the fp32 scores and the values, with the running
// maximum of the row's visible keys as the shift.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {
namespace {

constexpr int kGC = 128;        // steps per chunk (rows of S, TMEM lanes)
constexpr int kGM = 64;         // feature width
constexpr int kVD = 64;         // value channels of a head (the row width of v and out)
constexpr int kGD = 32;         // value channels of a CTA: two CTAs share a head
constexpr int kGN = 48;         // the CTA's channels, the constant channel, zero padding to a multiple of 16
constexpr int kQtr = 256 / kGD;  // groups of keys in the per-channel passes (thread = channel and group)
constexpr int kKg = kGC / kQtr;  // keys per group
constexpr float kGlaLinBeta = 0.25f;

struct GLay {
  static constexpr uint32_t kQ32 = 0, kK32 = 32768, kV32 = 65536;  // the chunk's fp32 inputs
  static constexpr uint32_t kGam = 98304;                          // gamma_t
  static constexpr uint32_t kDk = kGam + 512;                      // exp(gamma_last - gamma_i)
  static constexpr uint32_t kPart = kDk + 512;                     // per quarter of keys and channel: max, min, sum
  static constexpr uint32_t kQ16 = 103424;                         // 1024-aligned operands from here
  static constexpr uint32_t kK16 = kQ16 + 16384;
  static constexpr uint32_t kKT16 = kK16 + 16384;  // two boxes of 128 rows (64 features, 64 zero) x 64 keys
  static constexpr uint32_t kE16 = kKT16 + 32768;  // two boxes of kGN channels x 64 keys
  static constexpr uint32_t kEBox = kGN * 128;
  static constexpr uint32_t kS16 = kE16 + 2 * kEBox;    // kGN channels x 64 features
  static constexpr uint32_t kSf = kS16 + kGN * 128;     // fp32 state [channel][feature]
  static constexpr uint32_t kChan = kSf + kGN * kGM * 4;  // per channel: beta, anchor, mu, lambda, running min and sum, 1/beta
  static constexpr uint32_t kBar = kChan + 7 * kGN * 4;
  static constexpr uint32_t kTmemSlot = kBar + 32;
  static constexpr uint32_t kBytes = kTmemSlot + 32;
  static constexpr uint32_t kAlloc = kBytes + 1024;
  static_assert(kPart + 3 * kQtr * kGD * 4 <= kQ16, "partials fit below the operands");
  static_assert(kQ16 % 1024 == 0 && kK16 % 1024 == 0 && kKT16 % 1024 == 0 && kE16 % 1024 == 0 &&
                    kEBox % 1024 == 0 && kS16 % 1024 == 0,
                "swizzled operands on 1024-byte boundaries");
  static_assert(kAlloc <= 227 * 1024, "shared memory");
};

// TMEM columns (32-column aligned): S in fp32 (kept for the exact rows), the masked bf16 A,
// the three accumulators
constexpr uint32_t kColS = 0, kColA = 128, kColInter = 192, kColIntra = 288, kColU = 384;

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t *>(&v);
}

// expm1(y) / beta for y = beta x: x times the series of expm1(y) / y for |y| < 1/2
// (truncation below 4e-6 relative), (e^y - 1) / beta beyond (ex2.approx: the result
// is rounded to bf16); x itself at beta = 0.
__device__ __forceinline__ float em1_beta_fast(float x, float y, float rb) {
  float p = fmaf(y, 1.f / 720.f, 1.f / 120.f);  // both forms, then a select: no branch per element
  p = fmaf(y, p, 1.f / 24.f);
  p = fmaf(y, p, 1.f / 6.f);
  p = fmaf(y, p, 0.5f);
  p = fmaf(y, p, 1.f);
  const float far = (__expf(y) - 1.f) * rb;
  return fabsf(y) < 0.5f ? x * p : far;
}

// log1p(x) for x > -1: the series to x^5 for |x| < 2^-6 (truncation below 2^-36
// relative), lg2.approx of 1 + x beyond.
__device__ __forceinline__ float log1p_fast(float x) {
  float p = fmaf(x, 0.2f, -0.25f);  // both forms, then a select
  p = fmaf(x, p, 1.f / 3.f);
  p = fmaf(x, p, -0.5f);
  p = fmaf(x, p, 1.f);
  const float far = __logf(1.f + x);
  return fabsf(x) < 0.015625f ? x * p : far;
}

// 8 consecutive fp32 as bf16 into a 16-byte chunk of a 128-byte-swizzled row.
__device__ __forceinline__ void st_bf16x8(uint8_t *dst, const float *src, float scale) {
  const float4 a = *reinterpret_cast<const float4 *>(src), b = *reinterpret_cast<const float4 *>(src + 4);
  *reinterpret_cast<uint4 *>(dst) = make_uint4(pack_bf16x2(a.x * scale, a.y * scale), pack_bf16x2(a.z * scale, a.w * scale),
                                               pack_bf16x2(b.x * scale, b.y * scale), pack_bf16x2(b.z * scale, b.w * scale));
}

__global__ void __launch_bounds__(256, 1)
    gla_tc_kernel(const float *__restrict__ qf, const float *__restrict__ kf, const float *__restrict__ v,
                  const float *__restrict__ logdecay, const float *__restrict__ beta, float *__restrict__ out,
                  float *__restrict__ logz, int H, int T, unsigned *__restrict__ err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int bh = blockIdx.x, h = bh % H, jo = blockIdx.y * kGD;  // the head, its first channel here
  const int n_ch = (T + kGC - 1) / kGC;
  float *q32 = reinterpret_cast<float *>(smem + GLay::kQ32), *k32 = reinterpret_cast<float *>(smem + GLay::kK32),
        *v32 = reinterpret_cast<float *>(smem + GLay::kV32);
  float *gam = reinterpret_cast<float *>(smem + GLay::kGam), *dk = reinterpret_cast<float *>(smem + GLay::kDk);
  float *pmax = reinterpret_cast<float *>(smem + GLay::kPart), *pmin = pmax + kQtr * kGD, *psum = pmin + kQtr * kGD;
  float *Sf = reinterpret_cast<float *>(smem + GLay::kSf);
  float *c_beta = reinterpret_cast<float *>(smem + GLay::kChan), *c_anc = c_beta + kGN, *c_mu = c_anc + kGN,
        *c_lam = c_mu + kGN, *c_rmin = c_lam + kGN, *c_rsum = c_rmin + kGN, *c_rb = c_rsum + kGN;
  const uint32_t bar_in = sbase + GLay::kBar, bar_s = bar_in + 8, bar_a = bar_in + 16;
  const size_t base_row = static_cast<size_t>(bh) * T;

  auto issue_inputs = [&](int c) {  // the chunk's rows of qf, kf and v (contiguous in [B, H, T, .])
    const int rows = min(kGC, T - c * kGC);
    const size_t r0 = base_row + static_cast<size_t>(c) * kGC;
    const uint32_t bytes = static_cast<uint32_t>(rows) * kGM * 4, vbytes = static_cast<uint32_t>(rows) * kVD * 4;
    mbar_arrive_expect_tx(bar_in, 2 * bytes + vbytes);
    bulk_load(sbase + GLay::kQ32, qf + r0 * kGM, bytes, bar_in);
    bulk_load(sbase + GLay::kK32, kf + r0 * kGM, bytes, bar_in);
    bulk_load(sbase + GLay::kV32, v + r0 * kVD, vbytes, bar_in);  // whole rows: both CTAs' channels
  };

  if (tid == 0) {
    mbar_init(bar_in, 1);
    mbar_init(bar_s, 1);
    mbar_init(bar_a, 1);
    fence_mbar_init();
    issue_inputs(0);
  }
  if (warp == 1) {
    tmem_alloc(sbase + GLay::kTmemSlot, 512);
    tmem_relinquish();
  }
  // constant parts of the operands: KT16's rows 64..127, E16's channel 64 (ones) and 65..79
  // (zeros); the state and its bf16 copy start at zero
  for (int i = tid; i < 2 * 64 * 8; i += 256) {
    const int bx = i >> 9, r = 64 + ((i >> 3) & 63), ch = i & 7;
    *reinterpret_cast<uint4 *>(smem + GLay::kKT16 + bx * 16384 + sw128_offset(r, ch)) = make_uint4(0u, 0u, 0u, 0u);
  }
  for (int i = tid; i < 2 * (kGN - kGD) * 8; i += 256) {
    const int bx = i / ((kGN - kGD) * 8), r = kGD + (i >> 3) % (kGN - kGD), ch = i & 7;
    const uint32_t one = r == kGD ? pack_bf16x2(1.f, 1.f) : 0u;
    *reinterpret_cast<uint4 *>(smem + GLay::kE16 + bx * GLay::kEBox + sw128_offset(r, ch)) = make_uint4(one, one, one, one);
  }
  for (int i = tid; i < kGN * kGM; i += 256) Sf[i] = 0.f;
  for (int i = tid; i < kGN * 8; i += 256)
    *reinterpret_cast<uint4 *>(smem + GLay::kS16 + sw128_offset(i >> 3, i & 7)) = make_uint4(0u, 0u, 0u, 0u);
  for (int j = tid; j < kGN; j += 256) {
    c_beta[j] = j < kGD ? beta[h * kVD + jo + j] : 0.f;
    c_anc[j] = INFINITY;
    c_mu[j] = -INFINITY;
    c_lam[j] = 0.f;
    c_rmin[j] = INFINITY;
    c_rsum[j] = 0.f;
    c_rb[j] = c_beta[j] != 0.f ? 1.f / c_beta[j] : 0.f;
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(smem + GLay::kTmemSlot);
  const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;

  bool ok = true;
  for (int c = 0; c < n_ch && ok; ++c) {
    const int rows = min(kGC, T - c * kGC);
    const size_t r0 = base_row + static_cast<size_t>(c) * kGC;
    const uint32_t par = static_cast<uint32_t>(c & 1);
    // ---- the chunk's inputs; rows past T read as zero (no key weight, no output)
    ok = __syncthreads_and(mbar_wait(bar_in, par, err, kErrWaitTma));
    if (!ok) break;
    float g = 0.f;
    if (tid < kGC && tid < rows) g = logdecay[r0 + tid];
    if (rows < kGC) {
      for (int i = rows * 16 + tid; i < kGC * 16; i += 256) {
        const int rr = i >> 4, cc = (i & 15) * 4;
        *reinterpret_cast<float4 *>(q32 + rr * kGM + cc) = make_float4(0.f, 0.f, 0.f, 0.f);
        *reinterpret_cast<float4 *>(k32 + rr * kGM + cc) = make_float4(0.f, 0.f, 0.f, 0.f);
        *reinterpret_cast<float4 *>(v32 + rr * kVD + cc) = make_float4(0.f, 0.f, 0.f, 0.f);
      }
    }
    // ---- gamma_t = g_0 + ... + g_t over the chunk (warps 0-3, one step each)
    if (tid < kGC) {
      float x = g;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, x, off);
        if (lane >= off) x += y;
      }
      if (lane == 31) pmax[warp] = x;  // warp totals (the partials are free until the channel pass)
      gam[tid] = x;
    }
    __syncthreads();
    if (tid < kGC) {
      float add = 0.f;
      for (int w = 0; w < warp; ++w) add += pmax[w];
      gam[tid] += add;
    }
    __syncthreads();
    const float glast = gam[kGC - 1];
    if (tid < kGC) dk[tid] = expf(glast - gam[tid]);
    // ---- Qf and Kf as bf16 (K-major, 128-byte swizzle); the channels' extremes over the chunk
    for (int i = tid; i < kGC * 8; i += 256) {
      const int rr = i >> 3, ch = i & 7;
      st_bf16x8(smem + GLay::kQ16 + sw128_offset(rr, ch), q32 + rr * kGM + ch * 8, 1.f);
      st_bf16x8(smem + GLay::kK16 + sw128_offset(rr, ch), k32 + rr * kGM + ch * 8, 1.f);
    }
    {
      const int j = tid % kGD, qtr = tid / kGD;
      float mx = -INFINITY, mn = INFINITY, sm = 0.f;
      for (int i = qtr * kKg; i < min(qtr * kKg + kKg, rows); ++i) {
        const float x = v32[i * kVD + jo + j];
        mx = fmaxf(mx, x);
        mn = fminf(mn, x);
        sm += x;
      }
      pmax[qtr * kGD + j] = mx;
      pmin[qtr * kGD + j] = mn;
      psum[qtr * kGD + j] = sm;
    }
    __syncthreads();
    // decayed Kf transposed (features x keys) for the state's contraction
    for (int i = tid; i < kGM * 16; i += 256) {
      const int f = i & 63, kc = i >> 6;  // lanes over features: conflict-free column reads
      float tmp[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) tmp[u] = k32[(kc * 8 + u) * kGM + f] * dk[kc * 8 + u];
      *reinterpret_cast<uint4 *>(smem + GLay::kKT16 + (kc >> 3) * 16384 + sw128_offset(f, kc & 7)) =
          make_uint4(pack_bf16x2(tmp[0], tmp[1]), pack_bf16x2(tmp[2], tmp[3]), pack_bf16x2(tmp[4], tmp[5]),
                     pack_bf16x2(tmp[6], tmp[7]));
    }
    // per channel: the shifted form's lambda; the linear form's anchor, moving the state with it
    if (tid < kGD) {
      const int j = tid;
      const float b = c_beta[j];
      float mx = pmax[j], mn = pmin[j], sm = psum[j];
#pragma unroll
      for (int g = 1; g < kQtr; ++g) {
        mx = fmaxf(mx, pmax[g * kGD + j]);
        mn = fminf(mn, pmin[g * kGD + j]);
        sm += psum[g * kGD + j];
      }
      if (b >= kGlaLinBeta) {
        c_lam[j] = b * mx;
        pmax[j] = 1.f;  // no move of the state (see below)
        pmin[j] = 0.f;
      } else {
        // the anchor: the mean of the values so far, at most 1/beta above their minimum (so that
        // 1 + beta num / Z >= 1/e); the state moves with it (either way)
        const float rmin = fminf(c_rmin[j], mn);
        const float rsum = c_rsum[j] + sm;
        c_rmin[j] = rmin;
        c_rsum[j] = rsum;
        const float mean = rsum / static_cast<float>(c * kGC + rows);
        const float cn = b > 0.f ? fminf(mean, rmin + 1.f / b) : mean, co = c_anc[j];
        // the state's move with the anchor: factors here, the transform by every thread below
        float e = 1.f, w = 0.f;
        if (co != INFINITY && cn != co) {
          const float x = co - cn;
          e = expf(b * x);
          w = b != 0.f ? expm1f(b * x) / b : x;
        }
        pmax[j] = e;  // the chunk's extremes are consumed; their space holds the factors
        pmin[j] = w;
        c_anc[j] = cn;
      }
    }
    __syncthreads();
    for (int i = tid; i < kGD * kGM; i += 256) {
      const int j = i / kGM, f = i % kGM;
      const float e = pmax[j], w = pmin[j];
      if (e != 1.f || w != 0.f) Sf[i] = fmaf(e, Sf[i], w * Sf[kGD * kGM + f]);
    }
    __syncthreads();
    // the chunk's bank (channels x keys, K-major) and the state's bf16 copy (channels x features)
    {
      const int j = tid % kGD, qtr = tid / kGD;
      const float b = c_beta[j];
      const bool lin = b < kGlaLinBeta;
      const float sh = lin ? c_anc[j] : c_lam[j], rb = c_rb[j];
#pragma unroll 1
      for (int kc = qtr * (kKg / 8); kc < (qtr + 1) * (kKg / 8); ++kc) {
        float e[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int i = kc * 8 + u;
          const float x = v32[i * kVD + jo + j];
          float val;
          if (lin) val = em1_beta_fast(x - sh, b * (x - sh), rb);
          else val = __expf(b * x - sh);
          e[u] = i < rows ? val : 0.f;
        }
        *reinterpret_cast<uint4 *>(smem + GLay::kE16 + (kc >> 3) * GLay::kEBox + sw128_offset(j, kc & 7)) =
            make_uint4(pack_bf16x2(e[0], e[1]), pack_bf16x2(e[2], e[3]), pack_bf16x2(e[4], e[5]),
                       pack_bf16x2(e[6], e[7]));
      }
    }
    for (int i = tid; i < kGN * 8; i += 256) {
      const int j = i >> 3, fc = i & 7;
      st_bf16x8(smem + GLay::kS16 + sw128_offset(j, fc), Sf + j * kGM + fc * 8, 1.f);
    }
    fence_proxy_async_smem();  // the operands' generic writes, and the fp32 tiles' reads, before the async proxy
    __syncthreads();
    if (tid == 0) {
      if (c + 1 < n_ch) issue_inputs(c + 1);
      tc_fence_after_sync();
      constexpr uint32_t id_s = idesc_f16(128, 128, true, false), id_n = idesc_f16(128, kGN, true, false);
#pragma unroll
      for (int kk = 0; kk < kGM / 16; ++kk)
        mma_f16_ss(tmem + kColS, smem_desc_sw128(sbase + GLay::kQ16 + kk * 32, 16, 1024),
                   smem_desc_sw128(sbase + GLay::kK16 + kk * 32, 16, 1024), id_s, kk > 0 ? 1u : 0u);
#pragma unroll
      for (int kk = 0; kk < kGM / 16; ++kk)
        mma_f16_ss(tmem + kColInter, smem_desc_sw128(sbase + GLay::kQ16 + kk * 32, 16, 1024),
                   smem_desc_sw128(sbase + GLay::kS16 + kk * 32, 16, 1024), id_n, kk > 0 ? 1u : 0u);
      mma_commit(bar_s);
    }
    // ---- S o decay mask, as bf16 in A's 64 columns (thread = row of its warp's TMEM lane
    // quarter; warps 0-3 take keys 0..63, warps 4-7 keys 64..127)
    {
      ok = __all_sync(0xffffffffu, mbar_wait(bar_s, par, err, kErrWaitMma));
      if (ok) {
        tc_fence_after_sync();
        const int t = (warp & 3) * 32 + lane, kh = warp >> 2;  // row, half of the keys
        uint32_t s[2][32];
#pragma unroll
        for (int q = 0; q < 2; ++q) tmem_ld32(tmem + kColS + lane_off + (kh * 2 + q) * 32, s[q]);
        tmem_ld_wait();
        const float gt = gam[t];
#pragma unroll
        for (int q = 0; q < 2; ++q) {
          uint32_t p[16];
#pragma unroll
          for (int i2 = 0; i2 < 16; ++i2) {
            const int i = (kh * 2 + q) * 32 + 2 * i2;
            const float a0 = i <= t ? __uint_as_float(s[q][2 * i2]) * __expf(gt - gam[i]) : 0.f;
            const float a1 = i + 1 <= t ? __uint_as_float(s[q][2 * i2 + 1]) * __expf(gt - gam[i + 1]) : 0.f;
            p[i2] = pack_bf16x2(a0, a1);
          }
          tmem_st16(tmem + kColA + lane_off + (kh * 2 + q) * 16, p);
        }
        tmem_st_wait();
      }
    }
    tc_fence_before_sync();
    ok = __syncthreads_and(ok);
    if (!ok) break;
    if (tid == 0) {
      tc_fence_after_sync();
      constexpr uint32_t id_n = idesc_f16(128, kGN, true, false);
#pragma unroll
      for (int kk = 0; kk < kGC / 16; ++kk)
        mma_f16_ts(tmem + kColIntra, tmem + kColA + kk * 8,
                   smem_desc_sw128(sbase + GLay::kE16 + (kk >> 2) * GLay::kEBox + (kk & 3) * 32, 16, 1024), id_n,
                   kk > 0 ? 1u : 0u);
#pragma unroll
      for (int kk = 0; kk < kGC / 16; ++kk)
        mma_f16_ss(tmem + kColU, smem_desc_sw128(sbase + GLay::kKT16 + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024),
                   smem_desc_sw128(sbase + GLay::kE16 + (kk >> 2) * GLay::kEBox + (kk & 3) * 32, 16, 1024), id_n,
                   kk > 0 ? 1u : 0u);
      mma_commit(bar_a);
    }
    // ---- the outputs (thread = row of its warp's lane quarter; warps 4-7 take the CTA's channels
    // 0..15, warps 0-3 channels 16..31) and then the state (warps 0, 1, 4, 5, thread = feature)
    const bool state_warp = (warp & 3) < 2;
    ok = __all_sync(0xffffffffu, mbar_wait(bar_a, par, err, kErrWaitMma));
    if (ok) {
      tc_fence_after_sync();
      const int t = (warp & 3) * 32 + lane, q = warp < 4 ? 1 : 0;
      const float gt = gam[t], et = __expf(gt);
      const float zi = __uint_as_float(tmem_ld1(tmem + kColIntra + lane_off + kGD));
      const float zx = __uint_as_float(tmem_ld1(tmem + kColInter + lane_off + kGD));
      uint32_t ai[32], ax[32];
      tmem_ld32(tmem + kColIntra + lane_off, ai);
      tmem_ld32(tmem + kColInter + lane_off, ax);
      tmem_ld_wait();
      const float Z = fmaf(et, zx, zi), lz = __logf(Z), rZ = 1.f / Z;
      if (q == 0 && blockIdx.y == 0 && t < rows && logz) logz[r0 + t] = lz;
      // shifted channels whose in-chunk sum fell below 2^-100 of the row's in-chunk prior mass:
      // the chunk's shift may lie far above every key the row sees (the largest value came
      // later in the chunk), so terms under fp32's range may carry the sum; recomputed below
      unsigned flag = 0;
      float o[16];
      auto read = [&](int j, float in, float ix) {  // j: the CTA's channel
        const float b = c_beta[j], rb = c_rb[j];
        // both forms, then a select (the form is the channel's; no branch per element)
        const bool lin = b < kGlaLinBeta;
        const float num = fmaf(et, ix, in), x = b * num * rZ;
        const float o_lin = b != 0.f ? fmaf(log1p_fast(x), rb, c_anc[j]) : fmaf(num, rZ, c_anc[j]);
        const float la = in > 0.f ? c_lam[j] + __logf(in) : -INFINITY;
        const float lb = ix > 0.f ? c_mu[j] + gt + __logf(ix) : -INFINITY;
        const float hi = fmaxf(la, lb), lo = fminf(la, lb);
        const float ln = hi == -INFINITY ? -INFINITY : hi + __logf(1.f + __expf(lo - hi));
        flag |= (!lin && !(in >= 0x1p-100f * zi)) ? 1u << j : 0u;
        return lin ? o_lin : (ln - lz) * rb;
      };
      if (q == 0) {
#pragma unroll
        for (int u = 0; u < 16; ++u) o[u] = read(u, __uint_as_float(ai[u]), __uint_as_float(ax[u]));
      } else {
#pragma unroll
        for (int u = 0; u < 16; ++u) o[u] = read(16 + u, __uint_as_float(ai[16 + u]), __uint_as_float(ax[16 + u]));
      }
      if (t < rows) {
        float *orow = out + (r0 + t) * kVD + jo + q * 16;
#pragma unroll
        for (int u = 0; u < 16; u += 4) *reinterpret_cast<float4 *>(orow + u) = make_float4(o[u], o[u + 1], o[u + 2], o[u + 3]);
      }
      // the flagged entries exactly: the row's fp32 scores (still in TMEM) and the chunk's values,
      // one pass over the visible keys with the running maximum of beta v as the shift
      if (__any_sync(0xffffffffu, flag != 0u && t < rows)) {
        uint32_t sr[4][32];
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) tmem_ld32(tmem + kColS + lane_off + qq * 32, sr[qq]);
        tmem_ld_wait();
        unsigned fm = t < rows ? flag : 0u;
        while (fm) {
          const int j = __ffs(fm) - 1;  // the CTA's channel
          fm &= fm - 1;
          const float b = c_beta[j];
          const float *vcol = v + r0 * kVD + jo + j;
          float m = -INFINITY, acc = 0.f;
          // 32 keys' values in flight at a time (the chunk's staged values already hold the next
          // chunk's), then the walk over them
#pragma unroll
          for (int i0 = 0; i0 < kGC; i0 += 32) {
            if (i0 > t) break;
            float xv[32];
#pragma unroll
            for (int k2 = 0; k2 < 32; ++k2)
              xv[k2] = i0 + k2 < rows ? __ldg(vcol + static_cast<size_t>(i0 + k2) * kVD) : 0.f;
#pragma unroll
            for (int k2 = 0; k2 < 32; ++k2) {
              const int i = i0 + k2;
              if (i <= t) {
                const float x = b * xv[k2];
                const float a = __uint_as_float(sr[i >> 5][i & 31]) * expf(gt - gam[i]);
                if (x > m) {
                  acc = fmaf(acc, expf(m - x), a);
                  m = x;
                } else {
                  acc = fmaf(a, expf(x - m), acc);
                }
              }
            }
          }
          // the state's part from the fp32 state (unchanged until the barrier below)
          const float *qrow = qf + (r0 + t) * kGM;
          float ix = 0.f;
#pragma unroll 8
          for (int f = 0; f < kGM; ++f) ix = fmaf(__ldg(qrow + f), Sf[j * kGM + f], ix);
          const float la = acc > 0.f ? m + logf(acc) : -INFINITY;
          const float lb = ix > 0.f ? c_mu[j] + gt + logf(ix) : -INFINITY;
          const float hi = fmaxf(la, lb), lo = fminf(la, lb);
          const float ln = hi == -INFINITY ? -INFINITY : hi + log1pf(expf(lo - hi));
          out[(r0 + t) * kVD + jo + j] = (ln - lz) / b;
        }
      }
    }
    __syncthreads();  // the exact entries read the state before its update
    if (ok && state_warp) {
      // feature f = the warp's TMEM lane; warps 0, 1 take channels 0 .. kGN/2 - 1, warps 4, 5
      // the rest (columns 0..63 loaded)
      const int f = (warp & 1) * 32 + lane;
      const float eg = __expf(glast);
      uint32_t uu[2][32];
      auto update = [&](int j, float uv) {
        const float b = c_beta[j];
        float &st = Sf[j * kGM + f];
        if (j >= kGD || b < kGlaLinBeta) {
          st = fmaf(eg, st, uv);
        } else {
          const float mo = c_mu[j], lam = c_lam[j], mn = fmaxf(mo + glast, lam);
          st = fmaf(__expf(mo + glast - mn), st, __expf(lam - mn) * uv);
        }
      };
      tmem_ld32(tmem + kColU + lane_off, uu[0]);
      tmem_ld32(tmem + kColU + lane_off + 32, uu[1]);
      tmem_ld_wait();
      if (warp < 4) {
#pragma unroll
        for (int u = 0; u < kGN / 2; ++u) update(u, __uint_as_float(uu[u >> 5][u & 31]));
      } else {
#pragma unroll
        for (int u = kGN / 2; u < kGN; ++u) update(u, __uint_as_float(uu[u >> 5][u & 31]));
      }
    }
    tc_fence_before_sync();
    ok = __syncthreads_and(ok);
    if (tid < kGD && c_beta[tid] >= kGlaLinBeta) c_mu[tid] = fmaxf(c_mu[tid] + glast, c_lam[tid]);
    __syncthreads();
  }
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, 512);
  }
}

}  // namespace

cudaError_t launch_gla_tc(const float *qf, const float *kf, const float *v, const float *logdecay, const float *beta,
                          float *out, float *logz, int B, int H, int T, unsigned *err, cudaStream_t stream) {
  cudaError_t e = cudaFuncSetAttribute(gla_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, GLay::kAlloc);
  if (e != cudaSuccess) return e;
  gla_tc_kernel<<<dim3(B * H, kVD / kGD), 256, GLay::kAlloc, stream>>>(qf, kf, v, logdecay, beta, out, logz, H, T,
                                                                      err);
  return cudaGetLastError();
}

}  // namespace fem
