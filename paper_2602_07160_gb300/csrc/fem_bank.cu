// Value-bank pre-pass of the FEM read: statistics, shift schedule and the
// fp16 value bank, written once per key tile for every query tile to share.
//
//   tile_stats  (block per tile)   max, min and sum of v_.j over each tile of
//                                  128 keys (valid keys only)
//   plan        (B*H x 32-channel  per channel: bank mode and linear anchor
//                groups)           from the whole sequence; the running maximum
//                                  over tiles 0..kt; the shifted bank's shift
//                                  c[kt], raised lazily along it (only when
//                                  beta*(max - c) > kShiftLag); a per-tile mask
//                                  of the channels whose shift moved; the
//                                  bank's coefficients for every tile
//   bank        (persistent)       E = bank(v) in fp16 with the tile's shift,
//                                  and per channel the sum of |E| over the
//                                  tile's keys (the tensor-core kernel's bound
//                                  on the error of 16-bit prior weights)
//
// The shift is the per-channel LSE stabilisation of App. E ("Numerical
// stability"), made online over key tiles; only keys < T enter it.  On a
// causal diagonal tile it also includes keys later than some of the tile's
// rows; the tensor-core kernel's guard finds the rows for which that (or a
// peaked prior) leaves the 16-bit operands too little range, and the exact
// fix-up completes them.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

constexpr float kBankFastBeta = 1.f / 64.f;  // linear bank: (e^y - 1)/beta from here on

// Ring of key tiles a persistent bank block streams through shared memory:
// kStages slots, one mbarrier each, filled by copies that thread 0 issues
// kStages - 1 tiles ahead.  A block takes tiles_of_block() tiles, the i-th of
// them number blockIdx.x + i gridDim.x of the (b, h, key tile) list (key tile
// fastest), counted from its start or from its end.
constexpr int kStages = 3;

__device__ __forceinline__ int tiles_of_block(int n_tiles) {
  return blockIdx.x < n_tiles ? (n_tiles - 1 - static_cast<int>(blockIdx.x)) / static_cast<int>(gridDim.x) + 1 : 0;
}

// ---------------------------------------------------------------------------
// tile_stats: one 128-thread block per key tile; thread (cc, rg) loads 16-byte
// chunk cc of rows rg*RPG .. rg*RPG + RPG - 1 straight from V, all RPG loads in
// flight at once (consecutive lanes read consecutive chunks of a row), lanes
// holding the same chunk combine by shuffles, the four warps through shared
// memory.  Short blocks, many resident per SM: the loads of several tiles per
// SM are in flight together.
// ---------------------------------------------------------------------------
template <int D>
struct StatsMap {
  static constexpr int CPR = D / 8;        // chunks per row
  static constexpr int RG = 128 / CPR;     // row groups
  static constexpr int RPG = 128 / RG;     // rows per group
};

template <int D>
__global__ void __launch_bounds__(128) tile_stats_kernel(const __nv_bfloat16 *__restrict__ v, int T, int n_kt,
                                                          float4 *__restrict__ tstat) {
  using M = StatsMap<D>;
  __shared__ float s_part[3][4][D];  // [max, min, sum][warp][channel]
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int cc = tid % M::CPR, rg = tid / M::CPR;
  const int g = static_cast<int>(blockIdx.x), bh = g / n_kt, kt = g % n_kt;
  const int rows = min(kBlockK, T - kt * kBlockK);
  const uint4 *src = reinterpret_cast<const uint4 *>(v + (static_cast<size_t>(bh) * T + static_cast<size_t>(kt) * kBlockK) * D);
  uint4 rawv[M::RPG];
#pragma unroll
  for (int r = 0; r < M::RPG; ++r) {
    const int row = rg * M::RPG + r;
    rawv[r] = row < rows ? __ldg(src + row * M::CPR + cc) : make_uint4(0u, 0u, 0u, 0u);
  }
  float mx[8], mn[8], sm[8];
#pragma unroll
  for (int u = 0; u < 8; ++u) {
    mx[u] = -INFINITY;
    mn[u] = INFINITY;
    sm[u] = 0.f;
  }
#pragma unroll
  for (int r = 0; r < M::RPG; ++r) {
    const int row = rg * M::RPG + r;
    if (row < rows) {
      const uint4 raw = rawv[r];
      const __nv_bfloat162 *p2 = reinterpret_cast<const __nv_bfloat162 *>(&raw);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float2 f = __bfloat1622float2(p2[u]);
        mx[2 * u] = fmaxf(mx[2 * u], f.x);
        mx[2 * u + 1] = fmaxf(mx[2 * u + 1], f.y);
        mn[2 * u] = fminf(mn[2 * u], f.x);
        mn[2 * u + 1] = fminf(mn[2 * u + 1], f.y);
        sm[2 * u] += f.x;
        sm[2 * u + 1] += f.y;
      }
    }
  }
#pragma unroll
  for (int off = M::CPR; off < 32; off <<= 1) {
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      mx[u] = fmaxf(mx[u], __shfl_xor_sync(0xffffffffu, mx[u], off));
      mn[u] = fminf(mn[u], __shfl_xor_sync(0xffffffffu, mn[u], off));
      sm[u] += __shfl_xor_sync(0xffffffffu, sm[u], off);
    }
  }
  if (lane < M::CPR) {
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      s_part[0][warp][cc * 8 + u] = mx[u];
      s_part[1][warp][cc * 8 + u] = mn[u];
      s_part[2][warp][cc * 8 + u] = sm[u];
    }
  }
  __syncthreads();  // every partial of the tile is written
  for (int j = tid; j < D; j += 128) {
    float a = s_part[0][0][j], b = s_part[1][0][j], c = s_part[2][0][j];
#pragma unroll
    for (int w = 1; w < 4; ++w) {
      a = fmaxf(a, s_part[0][w][j]);
      b = fminf(b, s_part[1][w][j]);
      c += s_part[2][w][j];
    }
    tstat[static_cast<size_t>(g) * D + j] = make_float4(a, b, c, 0.f);
  }
}

// A channel's bank mode and linear anchor from its max, min and mean over the
// sequence's valid keys (beta > 0: linear when an anchor keeps both the tilt
// and the bank within their bounds; beta = 0: linear at the mean).
__device__ __forceinline__ ChanInfo chan_info(float gmax, float gmin, float mean, float b) {
  ChanInfo ci;
  if (b > 0.f) {
    const float hi = gmin + kLinearLowTilt / b;
    const float lo = gmax - log1pf(kLinearBankMax * b) / b;
    ci.linear = lo <= hi ? 1.f : 0.f;
    ci.c_lin = fminf(fmaxf(mean, lo), hi);
  } else {
    ci.linear = 1.f;
    ci.c_lin = mean;
  }
  return ci;
}

// BankCoef of a channel at shift (or anchor) c.
__device__ __forceinline__ float4 bank_coef(bool lin, float b, float c) {
  return lin ? make_float4(b > 0.f ? 1.f / b : 0.f, b, c, __int_as_float(0x7fc00000))
             : make_float4(b * kLog2e, (kBankOffset - b * c) * kLog2e, c, 0.f);
}

// ---------------------------------------------------------------------------
// plan: one block per (b, h) and group of 32 channels, four threads per
// channel, each holding a quarter of a window of 64 key tiles in registers so
// every load of a window is in flight at once.  The lazy shift is a sequential
// recurrence over tiles: one lane per channel walks it over the window's tile
// maxima in shared memory, then the four lanes write the window's schedule in
// parallel.  Besides the schedule it writes the bank's per-tile coefficients
// (BankCoef) and the moved-channel word of its group.
// ---------------------------------------------------------------------------
template <int D>
__global__ void __launch_bounds__(128) plan_kernel(const float4 *__restrict__ tstat, const float *__restrict__ beta,
                                                   int H, int T, int n_kt, ChanInfo *__restrict__ chan,
                                                   float *__restrict__ shift, float *__restrict__ rfac,
                                                   unsigned *__restrict__ colmask, float4 *__restrict__ bcoef) {
  constexpr int kParts = 4, kPer = 16, kWin = kParts * kPer;
  __shared__ unsigned s_mask[kWin];
  __shared__ float s_tm[kWin][33];      // the window's tile maxima per channel of the block
  __shared__ float s_cl[kWin + 1][33];  // the shift before the window and after each of its tiles
  const int tid = threadIdx.x, part = tid % kParts, lane = tid & 31;
  const int grp = blockIdx.y, j = grp * 32 + tid / kParts;
  const int bh = blockIdx.x, h = bh % H;
  const float b = beta[h * D + j];
  const float4 *ts = tstat + static_cast<size_t>(bh) * n_kt * D + j;
  // pass 1: the channel's max, min and sum over every key tile
  float gmax = -INFINITY, gmin = INFINITY, gsum = 0.f;
  for (int w0 = 0; w0 < n_kt; w0 += kWin) {
    float4 st[kPer];
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int kt = w0 + part * kPer + u;
      st[u] = kt < n_kt ? ts[static_cast<size_t>(kt) * D] : make_float4(-INFINITY, INFINITY, 0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      gmax = fmaxf(gmax, st[u].x);
      gmin = fminf(gmin, st[u].y);
      gsum += st[u].z;
    }
  }
#pragma unroll
  for (int off = 1; off < kParts; off <<= 1) {
    gmax = fmaxf(gmax, __shfl_xor_sync(0xffffffffu, gmax, off));
    gmin = fminf(gmin, __shfl_xor_sync(0xffffffffu, gmin, off));
    gsum += __shfl_xor_sync(0xffffffffu, gsum, off);
  }
  const ChanInfo ci = chan_info(gmax, gmin, gsum / static_cast<float>(T), b);
  if (part == 0) chan[bh * D + j] = ci;
  const bool lin = ci.linear != 0.f;
  // pass 2, per window of 64 key tiles: the running maximum and the lazy shift are a
  // sequential recurrence, walked by one lane per channel over the window's tile maxima in
  // shared memory; then the four lanes of the channel write their quarter of the tiles'
  // shift, rescale factor, bank coefficients and moved-channel bits in parallel
  const int jl = tid / kParts;
  float cp = -INFINITY, cl = -INFINITY;  // carried across windows by the walking lane
  for (int w0 = 0; w0 < n_kt; w0 += kWin) {
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int kt = w0 + part * kPer + u;
      s_tm[part * kPer + u][jl] = kt < n_kt ? ts[static_cast<size_t>(kt) * D].x : -INFINITY;
    }
    for (int i = tid; i < kWin; i += 128) s_mask[i] = 0u;
    __syncthreads();
    if (part == 0) {
      s_cl[0][jl] = cl;
#pragma unroll 16
      for (int u = 0; u < kWin; ++u) {
        cp = fmaxf(cp, s_tm[u][jl]);
        if (lin) {
          cl = ci.c_lin;
        } else if (cl == -INFINITY || b * (cp - cl) > kShiftLag) {
          cl = cp;
        }
        s_cl[u + 1][jl] = cl;
      }
    }
    __syncthreads();
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int w = part * kPer + u, kt = w0 + w;
      if (kt < n_kt) {
        const float c = s_cl[w + 1][jl], prev = s_cl[w][jl];
        const size_t o = (static_cast<size_t>(bh) * n_kt + kt) * D + j;
        shift[o] = c;
        const bool moved = !lin && kt > 0 && c != prev;
        rfac[o] = moved ? expf(b * (prev - c)) : 1.f;
        if (moved) atomicOr(&s_mask[w], 1u << (j & 31));
        bcoef[o] = bank_coef(lin, b, c);
      }
    }
    __syncthreads();
    for (int i = tid; i < kWin; i += 128) {
      const int kt = w0 + i;
      if (kt < n_kt) {
        unsigned *cm = colmask + (static_cast<size_t>(bh) * n_kt + kt) * 4;
        cm[grp] = s_mask[i];
        if (grp == 0)
          for (int gz = D / 32; gz < 4; ++gz) cm[gz] = 0u;
      }
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// bank: 256 threads.  A slot holds the tile of V as D/64 boxes of 64 channels
// x 128 rows with the 128-byte swizzle (the layout the tensor-core kernel
// reads the bank in) and the tile's BankCoef.  Warp w owns the 16-byte chunks
// (8 channels) w*CPW .. w*CPW + CPW - 1; lane l handles rows l, 32 + l, 64 + l,
// 96 + l of a chunk, so each channel's form (linear or shifted) is uniform
// across the warp.  The bank overwrites V in the slot and leaves with one TMA
// store per box; the column sums of |bank| over the tile's valid rows go to
// colsum[tile][channel].
// ---------------------------------------------------------------------------
template <int D>
struct BankMap {
  static constexpr int kBoxes = D / 64;
  static constexpr int kTileBytes = kBlockK * D * 2;
  static constexpr int kSlotBytes = kTileBytes + D * 16;  // tile, then D BankCoef
  static constexpr int CPW = D / 64;                      // chunks per warp
  static constexpr int kSmem = kStages * kSlotBytes + 1024;
};

template <int D>
__device__ __forceinline__ void bank_issue(const CUtensorMap *tv, const float4 *bcoef, int n_kt, int g, uint32_t slot,
                                           uint32_t bar) {
  using M = BankMap<D>;
  const int bh = g / n_kt, kt = g % n_kt;
  mbar_arrive_expect_tx(bar, static_cast<uint32_t>(M::kSlotBytes));
#pragma unroll
  for (int bx = 0; bx < M::kBoxes; ++bx) tma_load_3d(slot + bx * 16384, tv, bar, bx * 64, kt * kBlockK, bh);
  bulk_load(slot + M::kTileBytes, bcoef + static_cast<size_t>(g) * D, D * 16, bar);
}

// Sum of x[u] over the warp's 32 lanes for u = 0..7 in 9 shuffles: each
// exchange halves the values a lane keeps (lanes keep the half named by the
// exchanged bit), then the last value is summed over the remaining two bits.
// Lane l ends with the sum for u = 4 ((l >> 4) & 1) + 2 ((l >> 3) & 1) +
// ((l >> 2) & 1).
__device__ __forceinline__ float warp_sum8_transposed(const float (&x)[8], int lane) {
  float a[4], b[2];
  const bool h16 = lane & 16, h8 = lane & 8, h4 = lane & 4;
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const float keep = h16 ? x[u + 4] : x[u], send = h16 ? x[u] : x[u + 4];
    a[u] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
  }
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const float keep = h8 ? a[u + 2] : a[u], send = h8 ? a[u] : a[u + 2];
    b[u] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
  }
  float c = (h4 ? b[1] : b[0]) + __shfl_xor_sync(0xffffffffu, h4 ? b[0] : b[1], 4);
  c += __shfl_xor_sync(0xffffffffu, c, 2);
  c += __shfl_xor_sync(0xffffffffu, c, 1);
  return c;
}

// Bank entries of one channel for four values x[0..3] of v, given the tile's
// BankCoef cf (w NaN: the linear bank), before the fp16 rounding.
__device__ __forceinline__ void bank_entries4(const float4 cf, const float (&x)[4], float (&e)[4]) {
  if (cf.w != cf.w) {
    // linear bank: D = expm1(y)/beta, y = beta (v - c) >= -1 (a = 1/beta,
    // b = beta).  For beta >= kBankFastBeta as (e^y - 1)/beta: the
    // absolute error of e^y (about 2^-22) over beta stays below 2^-16,
    // under the fp16 rounding of D.  Smaller beta (and beta = 0): a Taylor
    // series of expm1(y)/y for |y| < 1/2 (truncation < 4e-6 relative),
    // e^y - 1 beyond.  Rows go through the packed fp32x2 pipe in pairs.
    const float2 c2 = make_float2(-cf.z, -cf.z), b2 = make_float2(cf.y, cf.y);
    const float2 l2 = make_float2(cf.y * kLog2e, cf.y * kLog2e);
    if (cf.y >= kBankFastBeta) {
#pragma unroll
      for (int rp = 0; rp < 2; ++rp) {
        const float2 xs = __fadd2_rn(make_float2(x[2 * rp], x[2 * rp + 1]), c2);
        const float2 t = __fmul2_rn(l2, xs);
        const float2 d = __fmul2_rn(__fadd2_rn(make_float2(ex2_approx(t.x), ex2_approx(t.y)),
                                               make_float2(-1.f, -1.f)),
                                    make_float2(cf.x, cf.x));
        e[2 * rp] = d.x;
        e[2 * rp + 1] = d.y;
      }
    } else {
#pragma unroll
      for (int rp = 0; rp < 2; ++rp) {
        const float2 xs = __fadd2_rn(make_float2(x[2 * rp], x[2 * rp + 1]), c2);
        const float2 y = __fmul2_rn(b2, xs);
        float2 poly = __ffma2_rn(y, make_float2(1.f / 720.f, 1.f / 720.f), make_float2(1.f / 120.f, 1.f / 120.f));
        poly = __ffma2_rn(y, poly, make_float2(1.f / 24.f, 1.f / 24.f));
        poly = __ffma2_rn(y, poly, make_float2(1.f / 6.f, 1.f / 6.f));
        poly = __ffma2_rn(y, poly, make_float2(0.5f, 0.5f));
        poly = __ffma2_rn(y, poly, make_float2(1.f, 1.f));
        const float2 lin = __fmul2_rn(xs, poly);
        e[2 * rp] = fabsf(y.x) < 0.5f ? lin.x : (ex2_approx(y.x * kLog2e) - 1.f) * cf.x;
        e[2 * rp + 1] = fabsf(y.y) < 0.5f ? lin.y : (ex2_approx(y.y * kLog2e) - 1.f) * cf.x;
      }
    }
  } else {
    // shifted bank: E = 2^(a v + b)
#pragma unroll
    for (int rp = 0; rp < 2; ++rp) {
      const float2 t = __ffma2_rn(make_float2(cf.x, cf.x), make_float2(x[2 * rp], x[2 * rp + 1]),
                                  make_float2(cf.y, cf.y));
      e[2 * rp] = ex2_approx(t.x);
      e[2 * rp + 1] = ex2_approx(t.y);
    }
  }
}

template <int D>
__global__ void __launch_bounds__(256, 2) bank_kernel(const __grid_constant__ CUtensorMap tv,
                                                       const __grid_constant__ CUtensorMap te,
                                                       const float4 *__restrict__ bcoef, int T, int n_kt,
                                                       int n_tiles, int reverse, float *__restrict__ colsum,
                                                       unsigned *__restrict__ err) {
  using M = BankMap<D>;
  // the read kernel, a programmatic dependent launch, may take the SMs this pass's tail leaves
  grid_dep_launch_dependents();
  extern __shared__ uint8_t bank_smem[];
  __shared__ __align__(8) uint64_t s_full[kStages];
  const uint32_t base_addr = (smem_u32(bank_smem) + 1023u) & ~1023u;  // 128-byte swizzle wants 1024-B alignment
  uint8_t *const ring = bank_smem + (base_addr - smem_u32(bank_smem));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int my_n = tiles_of_block(n_tiles);
  // reverse: the tiles from the end of the list, for a V larger than L2 -- the last tiles the
  // statistics pass read are still in L2 when this pass starts, and the bank tiles written last
  // (the first heads) are the first the read kernel wants
  auto tile_of = [&](int i) {
    const int x = static_cast<int>(blockIdx.x) + i * static_cast<int>(gridDim.x);
    return reverse ? n_tiles - 1 - x : x;
  };
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(smem_u32(&s_full[s]), 1);
    fence_mbar_init();
    for (int i = 0; i < kStages - 1 && i < my_n; ++i)
      bank_issue<D>(&tv, bcoef, n_kt, tile_of(i), base_addr + i * M::kSlotBytes, smem_u32(&s_full[i]));
  }
  __syncthreads();
  for (int i = 0; i < my_n; ++i) {
    const int st = i % kStages, g = tile_of(i);
    const int bh = g / n_kt, kt = g % n_kt, rows = min(kBlockK, T - kt * kBlockK);
    if (!mbar_wait(smem_u32(&s_full[st]), (i / kStages) & 1, err, kErrWaitTma)) {
      if (tid == 0) bulk_wait_group_read0();
      return;
    }
    uint8_t *const tile = ring + st * M::kSlotBytes;
    const float4 *const coef = reinterpret_cast<const float4 *>(tile + M::kTileBytes);
#pragma unroll
    for (int q = 0; q < M::CPW; ++q) {
      const int ch = warp * M::CPW + q;  // chunk: channels 8 ch .. 8 ch + 7
      uint8_t *cell[4];
      uint4 raw[4];
#pragma unroll
      for (int rb = 0; rb < 4; ++rb) {
        const int row = rb * 32 + lane;
        cell[rb] = tile + (ch >> 3) * 16384 + row * 128 + (((ch & 7) ^ (row & 7)) << 4);
        raw[rb] = *reinterpret_cast<const uint4 *>(cell[rb]);
      }
      float res[4][8], csum[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const float4 cf = coef[ch * 8 + u];  // {a, b, c, w}; w NaN: linear bank
        float x[4];
#pragma unroll
        for (int rb = 0; rb < 4; ++rb) {
          const uint32_t w = reinterpret_cast<const uint32_t *>(&raw[rb])[u >> 1];
          x[rb] = __uint_as_float((u & 1) ? (w & 0xffff0000u) : (w << 16));
        }
        float e4[4];
        bank_entries4(cf, x, e4);
#pragma unroll
        for (int rb = 0; rb < 4; ++rb) res[rb][u] = e4[rb];
        // |bank| summed over this lane's valid rows (rows past T are padding)
        float cs = 0.f;
#pragma unroll
        for (int rb = 0; rb < 4; ++rb) cs += rb * 32 + lane < rows ? fabsf(res[rb][u]) : 0.f;
        csum[u] = cs;
      }
#pragma unroll
      for (int rb = 0; rb < 4; ++rb) {
        uint4 o;
        uint32_t *ow = reinterpret_cast<uint32_t *>(&o);
#pragma unroll
        for (int p = 0; p < 4; ++p) {
          const __half2 h2 = __floats2half2_rn(res[rb][2 * p], res[rb][2 * p + 1]);
          ow[p] = *reinterpret_cast<const uint32_t *>(&h2);
        }
        *reinterpret_cast<uint4 *>(cell[rb]) = o;
      }
      const float tot = warp_sum8_transposed(csum, lane);
      if ((lane & 3) == 0)
        colsum[static_cast<size_t>(g) * D + ch * 8 + ((lane >> 4) & 1) * 4 + ((lane >> 3) & 1) * 2 + ((lane >> 2) & 1)] =
            tot;
    }
    fence_proxy_async_smem();
    __syncthreads();
    if (tid == 0) {
#pragma unroll
      for (int bx = 0; bx < M::kBoxes; ++bx) tma_store_3d(&te, base_addr + st * M::kSlotBytes + bx * 16384, bx * 64,
                                                          kt * kBlockK, bh);
      bulk_commit_group();
      // the slot refilled next was last read by the previous tile's store
      bulk_wait_group_read<1>();
      if (i + kStages - 1 < my_n) {
        const int sn = (i + kStages - 1) % kStages;
        bank_issue<D>(&tv, bcoef, n_kt, tile_of(i + kStages - 1), base_addr + sn * M::kSlotBytes,
                      smem_u32(&s_full[sn]));
      }
    }
  }
  if (tid == 0) bulk_wait_group_read<0>();
}

// ---------------------------------------------------------------------------
// prepass: the three passes above in one kernel, for short sequences (up to
// kFusedMaxTiles key tiles), where the three launches' latency rather than the
// bytes set the pre-pass's time.  One 256-thread block per (b, h) and group of
// 32 channels: the statistics of every key tile (the tiles' maxima kept in
// shared memory), the plan of its 32 channels, then the bank and its column
// sums, the tiles taken from the last (the most recently read first).  Warp w
// takes the 16-byte chunk w % 4 (channels 8 (w % 4) .. + 7 of the group) of the
// key tiles w / 4, w / 4 + 2, ...; lane l rows l, l + 32, l + 64, l + 96 of a
// tile, so a channel's bank form is uniform across the warp and all eight warps
// work on sequences of two key tiles.  A warp load touches 32 row segments,
// which costs more than the launches saved from 16 key tiles on; there the
// three kernels run.  The results are those of the three kernels up to the
// summation order of the channel means.
// ---------------------------------------------------------------------------
constexpr int kFusedMaxTiles = 4;
constexpr int kFusedStatsTiles = 4;  // key tiles whose loads a warp keeps in flight (statistics)
constexpr int kFusedBankTiles = 2;   // the same for the bank

// Max (OP 0), min (1) or sum (2) of x[u] over the warp's 32 lanes for u = 0..7,
// transposed like warp_sum8_transposed: lane l ends with the result for
// u = 4 ((l >> 4) & 1) + 2 ((l >> 3) & 1) + ((l >> 2) & 1).
template <int OP>
__device__ __forceinline__ float comb(float a, float b) {
  return OP == 0 ? fmaxf(a, b) : (OP == 1 ? fminf(a, b) : a + b);
}
template <int OP>
__device__ __forceinline__ float warp_reduce8_transposed(const float (&x)[8], int lane) {
  float a[4], b[2];
  const bool h16 = lane & 16, h8 = lane & 8, h4 = lane & 4;
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const float keep = h16 ? x[u + 4] : x[u], send = h16 ? x[u] : x[u + 4];
    a[u] = comb<OP>(keep, __shfl_xor_sync(0xffffffffu, send, 16));
  }
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const float keep = h8 ? a[u + 2] : a[u], send = h8 ? a[u] : a[u + 2];
    b[u] = comb<OP>(keep, __shfl_xor_sync(0xffffffffu, send, 8));
  }
  float c = comb<OP>(h4 ? b[1] : b[0], __shfl_xor_sync(0xffffffffu, h4 ? b[0] : b[1], 4));
  c = comb<OP>(c, __shfl_xor_sync(0xffffffffu, c, 2));
  c = comb<OP>(c, __shfl_xor_sync(0xffffffffu, c, 1));
  return c;
}

template <int D>
__global__ void __launch_bounds__(256, 2) prepass_kernel(const __nv_bfloat16 *__restrict__ v,
                                                          const float *__restrict__ beta, int H, int T, int n_kt,
                                                          ChanInfo *__restrict__ chan, float *__restrict__ shift,
                                                          float *__restrict__ rfac, unsigned *__restrict__ colmask,
                                                          float *__restrict__ colsum, __half *__restrict__ bank) {
  // the read kernel, a programmatic dependent launch, may take the SMs this pass's tail leaves
  grid_dep_launch_dependents();
  extern __shared__ float s_tile[];  // [n_kt][32]: the tiles' maxima, then the shifts
  __shared__ float s_g[2][3][32];     // per tile phase: the channels' max, min and sum
  __shared__ float s_b[32], s_clin[32];
  __shared__ int s_lin[32];
  constexpr int kGroups = D / 32;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int cq = warp & 3, ph = warp >> 2;  // chunk of the group, tile phase
  const int bh = static_cast<int>(blockIdx.x) / kGroups, grp = static_cast<int>(blockIdx.x) % kGroups;
  const int h = bh % H, j0 = grp * 32 + 8 * cq;  // the chunk's first channel
  const int ul = ((lane >> 4) & 1) * 4 + ((lane >> 3) & 1) * 2 + ((lane >> 2) & 1);  // lane's channel after a reduction
  const size_t head = static_cast<size_t>(bh) * T;
  const __nv_bfloat16 *vb = v + head * D + j0;

  // ---- statistics: max, min and sum of every tile's valid keys
  float gmx = -INFINITY, gmn = INFINITY, gsm = 0.f;  // channel j0 + ul over this warp's tiles
  for (int kb = ph; kb < n_kt; kb += 2 * kFusedStatsTiles) {
    uint4 raw[kFusedStatsTiles][4];
#pragma unroll
    for (int i = 0; i < kFusedStatsTiles; ++i) {
      const int kt = kb + 2 * i;
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const int row = kt * kBlockK + r * 32 + lane;
        raw[i][r] = kt < n_kt && row < T ? __ldg(reinterpret_cast<const uint4 *>(vb + static_cast<size_t>(row) * D))
                                         : make_uint4(0u, 0u, 0u, 0u);
      }
    }
#pragma unroll
    for (int i = 0; i < kFusedStatsTiles; ++i) {
      const int kt = kb + 2 * i;
      if (kt >= n_kt) break;
      float mx[8], mn[8], sm[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        mx[u] = -INFINITY;
        mn[u] = INFINITY;
        sm[u] = 0.f;
      }
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        if (kt * kBlockK + r * 32 + lane < T) {
          const __nv_bfloat162 *p2 = reinterpret_cast<const __nv_bfloat162 *>(&raw[i][r]);
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const float2 f = __bfloat1622float2(p2[u]);
            mx[2 * u] = fmaxf(mx[2 * u], f.x);
            mx[2 * u + 1] = fmaxf(mx[2 * u + 1], f.y);
            mn[2 * u] = fminf(mn[2 * u], f.x);
            mn[2 * u + 1] = fminf(mn[2 * u + 1], f.y);
            sm[2 * u] += f.x;
            sm[2 * u + 1] += f.y;
          }
        }
      }
      const float tmx = warp_reduce8_transposed<0>(mx, lane);
      const float tmn = warp_reduce8_transposed<1>(mn, lane);
      const float tsm = warp_reduce8_transposed<2>(sm, lane);
      if ((lane & 3) == 0) s_tile[kt * 32 + 8 * cq + ul] = tmx;
      gmx = fmaxf(gmx, tmx);
      gmn = fminf(gmn, tmn);
      gsm += tsm;
    }
  }
  if ((lane & 3) == 0) {
    s_g[ph][0][8 * cq + ul] = gmx;
    s_g[ph][1][8 * cq + ul] = gmn;
    s_g[ph][2][8 * cq + ul] = gsm;
  }
  __syncthreads();

  // ---- plan: mode and anchor of channel grp*32 + lane, then the lazy shift walked over the tiles
  if (warp == 0) {
    const int j = grp * 32 + lane;
    const float b = beta[h * D + j];
    const ChanInfo ci = chan_info(fmaxf(s_g[0][0][lane], s_g[1][0][lane]), fminf(s_g[0][1][lane], s_g[1][1][lane]),
                                  (s_g[0][2][lane] + s_g[1][2][lane]) / static_cast<float>(T), b);
    chan[bh * D + j] = ci;
    const bool lin = ci.linear != 0.f;
    s_b[lane] = b;
    s_clin[lane] = ci.c_lin;
    s_lin[lane] = lin ? 1 : 0;
    float cp = -INFINITY, cl = -INFINITY;
    for (int kt = 0; kt < n_kt; ++kt) {
      cp = fmaxf(cp, s_tile[kt * 32 + lane]);
      if (lin) {
        cl = ci.c_lin;
      } else if (cl == -INFINITY || b * (cp - cl) > kShiftLag) {
        cl = cp;
      }
      s_tile[kt * 32 + lane] = cl;
    }
  }
  __syncthreads();
  // the schedule: warp w writes tiles w, w + 8, ... (lane = channel)
  {
    const int j = grp * 32 + lane;
    const float b = s_b[lane];
    const bool lin = s_lin[lane] != 0;
    for (int kt = warp; kt < n_kt; kt += 8) {
      const float c = s_tile[kt * 32 + lane], prev = kt > 0 ? s_tile[(kt - 1) * 32 + lane] : -INFINITY;
      const size_t o = (static_cast<size_t>(bh) * n_kt + kt) * D + j;
      shift[o] = c;
      const bool moved = !lin && kt > 0 && c != prev;
      rfac[o] = moved ? expf(b * (prev - c)) : 1.f;
      const unsigned bits = __ballot_sync(0xffffffffu, moved);
      unsigned *cm = colmask + (static_cast<size_t>(bh) * n_kt + kt) * 4;
      if (lane == 0) cm[grp] = bits;
      if (grp == 0 && lane >= kGroups && lane < 4) cm[lane] = 0u;
    }
  }

  // ---- bank: tiles from the last, E = bank(v) in fp16 and the column sums of |E|
  bool lin_u[8];
  float b_u[8], cl_u[8];
#pragma unroll
  for (int u = 0; u < 8; ++u) {
    lin_u[u] = s_lin[8 * cq + u] != 0;
    b_u[u] = s_b[8 * cq + u];
    cl_u[u] = s_clin[8 * cq + u];
  }
  __half *eb = bank + head * D + j0;
  const int n_mine = n_kt > ph ? (n_kt - 1 - ph) / 2 + 1 : 0;  // tiles n_kt - 1 - ph - 2 i
  for (int i0 = 0; i0 < n_mine; i0 += kFusedBankTiles) {
    uint4 raw[kFusedBankTiles][4];
#pragma unroll
    for (int i = 0; i < kFusedBankTiles; ++i) {
      const int kt = n_kt - 1 - ph - 2 * (i0 + i);
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const int row = kt * kBlockK + r * 32 + lane;
        raw[i][r] = i0 + i < n_mine && row < T
                        ? __ldg(reinterpret_cast<const uint4 *>(vb + static_cast<size_t>(row) * D))
                        : make_uint4(0u, 0u, 0u, 0u);
      }
    }
#pragma unroll
    for (int i = 0; i < kFusedBankTiles; ++i) {
      if (i0 + i >= n_mine) break;
      const int kt = n_kt - 1 - ph - 2 * (i0 + i);
      float res[4][8], csum[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const float4 cf = bank_coef(lin_u[u], b_u[u], lin_u[u] ? cl_u[u] : s_tile[kt * 32 + 8 * cq + u]);
        float x[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          const uint32_t w = reinterpret_cast<const uint32_t *>(&raw[i][r])[u >> 1];
          x[r] = __uint_as_float((u & 1) ? (w & 0xffff0000u) : (w << 16));
        }
        float e4[4];
        bank_entries4(cf, x, e4);
        float cs = 0.f;
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          res[r][u] = e4[r];
          cs += kt * kBlockK + r * 32 + lane < T ? fabsf(e4[r]) : 0.f;
        }
        csum[u] = cs;
      }
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const int row = kt * kBlockK + r * 32 + lane;
        if (row < T) {
          uint4 o;
          uint32_t *ow = reinterpret_cast<uint32_t *>(&o);
#pragma unroll
          for (int p = 0; p < 4; ++p) {
            const __half2 h2 = __floats2half2_rn(res[r][2 * p], res[r][2 * p + 1]);
            ow[p] = *reinterpret_cast<const uint32_t *>(&h2);
          }
          *reinterpret_cast<uint4 *>(eb + static_cast<size_t>(row) * D) = o;
        }
      }
      const float tot = warp_sum8_transposed(csum, lane);
      if ((lane & 3) == 0) colsum[(static_cast<size_t>(bh) * n_kt + kt) * D + j0 + ul] = tot;
    }
  }
}

cudaError_t launch_value_bank(const void *v, const CUtensorMap &tv, const CUtensorMap &te, const float *beta, int BH,
                              int H, int T, int d, const BankWorkspace &w, unsigned *err, int num_sms,
                              cudaStream_t stream, bool stats_ready) {
  const int n_kt = (T + kBlockK - 1) / kBlockK, n_tiles = BH * n_kt;
  const __nv_bfloat16 *vb = static_cast<const __nv_bfloat16 *>(v);
  if (n_kt <= kFusedMaxTiles) {
    const size_t smem = static_cast<size_t>(n_kt) * 32 * sizeof(float);
    if (d == 64)
      prepass_kernel<64><<<BH * 2, 256, smem, stream>>>(vb, beta, H, T, n_kt, w.chan, w.shift, w.rfac, w.colmask,
                                                         w.colsum, w.bank);
    else if (d == 128)
      prepass_kernel<128><<<BH * 4, 256, smem, stream>>>(vb, beta, H, T, n_kt, w.chan, w.shift, w.rfac, w.colmask,
                                                          w.colsum, w.bank);
    else
      return cudaErrorInvalidValue;
    return cudaGetLastError();
  }
  const int grid = min(n_tiles, 2 * num_sms);
  // V larger than half of L2: the bank pass walks the tiles backwards (measured at B4 H16 T8192
  // d128: 0.7 % per step; at 25 MB, where V stays in L2, forward was 0.5 % faster)
  const int reverse = static_cast<size_t>(n_tiles) * kBlockK * d * 2 > (size_t{64} << 20) ? 1 : 0;
  cudaError_t e = cudaSuccess;
  if (d == 64) {
    using BM = BankMap<64>;
    e = cudaFuncSetAttribute(bank_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, BM::kSmem);
    if (e != cudaSuccess) return e;
    if (!stats_ready) tile_stats_kernel<64><<<n_tiles, 128, 0, stream>>>(vb, T, n_kt, w.tstat);
    plan_kernel<64><<<dim3(BH, 2), 128, 0, stream>>>(w.tstat, beta, H, T, n_kt, w.chan, w.shift, w.rfac, w.colmask,
                                                     w.bcoef);
    bank_kernel<64><<<grid, 256, BM::kSmem, stream>>>(tv, te, w.bcoef, T, n_kt, n_tiles, reverse, w.colsum, err);
  } else if (d == 128) {
    using BM = BankMap<128>;
    e = cudaFuncSetAttribute(bank_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, BM::kSmem);
    if (e != cudaSuccess) return e;
    if (!stats_ready) tile_stats_kernel<128><<<n_tiles, 128, 0, stream>>>(vb, T, n_kt, w.tstat);
    plan_kernel<128><<<dim3(BH, 4), 128, 0, stream>>>(w.tstat, beta, H, T, n_kt, w.chan, w.shift, w.rfac, w.colmask,
                                                      w.bcoef);
    bank_kernel<128><<<grid, 256, BM::kSmem, stream>>>(tv, te, w.bcoef, T, n_kt, n_tiles, reverse, w.colsum, err);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace fem
