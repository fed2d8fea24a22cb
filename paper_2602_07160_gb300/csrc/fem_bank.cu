// Value-bank pre-pass of the FEM read: statistics, shift schedule and the
// fp16 value bank, written once per key tile for every query tile to share.
//
//   tile_stats  (B*H x key tiles)  max, min and sum of v_.j over each tile of
//                                  128 keys (valid keys only)
//   plan        (B*H)              per channel: bank mode and linear anchor
//                                  from the whole sequence; the running maximum
//                                  cpre[kt] = max over tiles 0..kt; the shifted
//                                  bank's shift c[kt], raised lazily along cpre
//                                  (only when beta*(cpre - c) > kShiftLag);
//                                  a per-tile mask of the channels whose shift moved
//   bank        (B*H x key tiles)  E = bank(v) in fp16 with the tile's shift;
//                                  causal: the (row, 32-channel group) entries
//                                  of the tile's diagonal rows whose visible
//                                  maximum lies more than kHazardTilt/beta below
//                                  the shift, for the exact fix-up
//
// The shift is the per-channel LSE stabilisation of App. E ("Numerical
// stability"), made online over key tiles; only keys < T enter it, and a
// query tile's last key tile is its diagonal tile, so keys beyond a tile's
// last row never raise the shift that tile's rows use.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

// Thread layout shared by tile_stats and bank: 128 threads cover a [128 x D]
// tile with 16-byte chunks; CPR chunks per row, RG row groups of RPG rows.
template <int D>
struct TileMap {
  static constexpr int CPR = D / 8;
  static constexpr int RG = 128 / CPR;
  static constexpr int RPG = 128 / RG;
};

// Both kernels stream the tile's rows (contiguous in V) into shared memory
// with one bulk copy, which keeps the HBM reads in flight independently of the
// threads' own load slots.
template <int D>
__device__ __forceinline__ bool stage_tile(const __nv_bfloat16 *v, int T, int bh, int kt, uint8_t *dst,
                                           uint64_t *bar_word, unsigned *err) {
  const uint32_t bar = smem_u32(bar_word);
  const int rows = min(kBlockK, T - kt * kBlockK);
  if (threadIdx.x == 0) {
    mbar_init(bar, 1);
    fence_mbar_init();
    mbar_arrive_expect_tx(bar, static_cast<uint32_t>(rows * D * 2));
    bulk_load(smem_u32(dst), v + (static_cast<size_t>(bh) * T + static_cast<size_t>(kt) * kBlockK) * D,
              static_cast<uint32_t>(rows * D * 2), bar);
  }
  __syncthreads();
  return mbar_wait(bar, 0, err, kErrWaitTma);
}

template <int D>
__global__ void __launch_bounds__(128) tile_stats_kernel(const __nv_bfloat16 *__restrict__ v, int T,
                                                          float4 *__restrict__ tstat, unsigned *__restrict__ err) {
  using M = TileMap<D>;
  extern __shared__ __align__(16) uint8_t tile_smem[];  // the tile's rows, [128][D] bf16
  __shared__ __align__(8) uint64_t s_bar;
  __shared__ float s_max[M::RG][D], s_min[M::RG][D], s_sum[M::RG][D];
  const int kt = blockIdx.x, bh = blockIdx.y, n_kt = gridDim.x;
  const int cc = threadIdx.x % M::CPR, rg = threadIdx.x / M::CPR;
  if (!stage_tile<D>(v, T, bh, kt, tile_smem, &s_bar, err)) return;
  float mx[8], mn[8], sm[8];
#pragma unroll
  for (int u = 0; u < 8; ++u) {
    mx[u] = -INFINITY;
    mn[u] = INFINITY;
    sm[u] = 0.f;
  }
#pragma unroll
  for (int i = 0; i < M::RPG; ++i) {
    const int row = rg * M::RPG + i;
    if (kt * kBlockK + row < T) {
      const uint4 raw = *reinterpret_cast<const uint4 *>(tile_smem + (row * D + cc * 8) * 2);
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
  for (int u = 0; u < 8; ++u) {
    s_max[rg][cc * 8 + u] = mx[u];
    s_min[rg][cc * 8 + u] = mn[u];
    s_sum[rg][cc * 8 + u] = sm[u];
  }
  __syncthreads();
  for (int j = threadIdx.x; j < D; j += 128) {
    float a = -INFINITY, b = INFINITY, c = 0.f;
    for (int g = 0; g < M::RG; ++g) {
      a = fmaxf(a, s_max[g][j]);
      b = fminf(b, s_min[g][j]);
      c += s_sum[g][j];
    }
    tstat[(static_cast<size_t>(bh) * n_kt + kt) * D + j] = make_float4(a, b, c, 0.f);
  }
}

// Plan of one (b, h) per block: four threads per channel, each holding a
// quarter of a window of 64 key tiles in registers, so every load of a window
// is in flight at once.  The lazy shift is a sequential recurrence over tiles:
// the four quarters run it in turn, handing the running (max, shift) on by
// warp shuffles.
template <int D>
__global__ void __launch_bounds__(4 * D) plan_kernel(const float4 *__restrict__ tstat, const float *__restrict__ beta,
                                                     int H, int T, int n_kt, ChanInfo *__restrict__ chan,
                                                     float *__restrict__ cpre, float *__restrict__ shift,
                                                     float *__restrict__ rfac, unsigned *__restrict__ colmask) {
  constexpr int kParts = 4, kPer = 16, kWin = kParts * kPer;
  __shared__ unsigned s_mask[kWin][4];
  const int tid = threadIdx.x, j = tid / kParts, part = tid % kParts, lane = tid & 31;
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
  const float mean = gsum / static_cast<float>(T);
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
  if (part == 0) chan[bh * D + j] = ci;
  const bool lin = ci.linear != 0.f;
  // pass 2: running maximum, lazy shift, rescale factors, moved-channel masks
  float cp = -INFINITY, cl = -INFINITY;
  for (int w0 = 0; w0 < n_kt; w0 += kWin) {
    float tmx[kPer];
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int kt = w0 + part * kPer + u;
      tmx[u] = kt < n_kt ? ts[static_cast<size_t>(kt) * D].x : -INFINITY;
    }
    for (int i = tid; i < kWin * 4; i += kParts * D) s_mask[i / 4][i % 4] = 0u;
    __syncthreads();
    for (int stage = 0; stage < kParts; ++stage) {
      if (part == stage) {
#pragma unroll
        for (int u = 0; u < kPer; ++u) {
          const int kt = w0 + stage * kPer + u;
          if (kt < n_kt) {
            cp = fmaxf(cp, tmx[u]);
            const float prev = cl;
            if (lin) {
              cl = ci.c_lin;
            } else if (cl == -INFINITY || b * (cp - cl) > kShiftLag) {
              cl = cp;
            }
            const size_t o = (static_cast<size_t>(bh) * n_kt + kt) * D + j;
            cpre[o] = cp;
            shift[o] = cl;
            const bool moved = !lin && kt > 0 && cl != prev;
            rfac[o] = moved ? expf(b * (prev - cl)) : 1.f;
            if (moved) atomicOr(&s_mask[stage * kPer + u][j >> 5], 1u << (j & 31));
          }
        }
      }
      // the quarter that ran hands its state on to the channel's other lanes
      cp = __shfl_sync(0xffffffffu, cp, (lane & ~(kParts - 1)) | stage);
      cl = __shfl_sync(0xffffffffu, cl, (lane & ~(kParts - 1)) | stage);
    }
    __syncthreads();
    for (int i = tid; i < kWin * 4; i += kParts * D) {
      const int kt = w0 + i / 4;
      if (kt < n_kt) colmask[(static_cast<size_t>(bh) * n_kt + kt) * 4 + i % 4] = s_mask[i / 4][i % 4];
    }
    __syncthreads();
  }
}

template <int D>
__global__ void __launch_bounds__(128, 3) bank_kernel(const __nv_bfloat16 *__restrict__ v,
                                                    const float *__restrict__ beta, const ChanInfo *__restrict__ chan,
                                                    const float *__restrict__ cpre, const float *__restrict__ shift,
                                                    int H, int T, int causal, __half *__restrict__ bank,
                                                    FixupEntry *__restrict__ fixups, int *__restrict__ fixup_count,
                                                    int *__restrict__ fixup_rows, int2 *__restrict__ tilefix,
                                                    unsigned *__restrict__ err) {
  using M = TileMap<D>;
  extern __shared__ __align__(16) uint8_t tile_smem[];  // the tile's rows of V, then of the bank, in place
  __shared__ __align__(8) uint64_t s_bar;
  __shared__ float s_a[D], s_b[D], s_c[D], s_lin[D], s_thr[D];
  __shared__ int s_first[D];
  const int kt = blockIdx.x, bh = blockIdx.y, n_kt = gridDim.x, h = bh % H;
  const int tid = threadIdx.x;
  const int cc = tid % M::CPR, rg = tid / M::CPR;
  for (int j = tid; j < D; j += 128) {
    const float b = beta[h * D + j];
    const ChanInfo ci = chan[bh * D + j];
    const size_t o = (static_cast<size_t>(bh) * n_kt + kt) * D + j;
    const float c = shift[o];
    s_lin[j] = ci.linear;
    s_c[j] = c;
    if (ci.linear != 0.f) {
      s_a[j] = b > 0.f ? 1.f / b : 0.f;  // linear bank: 1/beta and beta
      s_b[j] = b;
    } else {
      s_a[j] = b * kLog2e;  // shifted bank: E = ex2(a v + b)
      s_b[j] = (kBankOffset - b * c) * kLog2e;
    }
    // Diagonal hazard of a shifted channel: a row of this tile is safe once its
    // visible maximum reaches c - kHazardTilt/beta, i.e. from the first key at
    // or above that threshold on (row 0 when an earlier tile already reached it).
    const float thr = c - kHazardTilt / b;
    const bool haz = causal && ci.linear == 0.f;
    s_thr[j] = haz ? thr : -INFINITY;
    s_first[j] = (!haz || (kt > 0 && cpre[o - D] >= thr)) ? 0 : kBlockK;
  }
  __syncthreads();

  if (!stage_tile<D>(v, T, bh, kt, tile_smem, &s_bar, err)) return;
  // Thread: the 8 channels of chunk column cc, rows rg*RPG .. rg*RPG+RPG-1,
  // each 16-byte chunk of V replaced by the chunk of the bank.  Both bank
  // forms are evaluated and one is selected, so lanes never diverge.
  const int rows = min(kBlockK, T - kt * kBlockK);
  float pa[8], pb[8], pc[8], pthr[8];
  bool plin[8];
  int first[8];
#pragma unroll
  for (int u = 0; u < 8; ++u) {
    const int j = cc * 8 + u;
    pa[u] = s_a[j];
    pb[u] = s_b[j];
    pc[u] = s_c[j];
    pthr[u] = s_thr[j];
    plin[u] = s_lin[j] != 0.f;
    first[u] = kBlockK;
  }
#pragma unroll 2
  for (int i = 0; i < M::RPG; ++i) {
    {
      const int row = rg * M::RPG + i;
      if (row >= rows) break;
      uint4 *cell = reinterpret_cast<uint4 *>(tile_smem + (row * D + cc * 8) * 2);
      const uint4 raw = *cell;
      const __nv_bfloat16 *vin = reinterpret_cast<const __nv_bfloat16 *>(&raw);
      __align__(16) __half e[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const float x = __bfloat162float(vin[u]);
        if (x >= pthr[u]) first[u] = min(first[u], row);
        // linear bank: D = expm1(y)/beta, y = beta (v - c) >= -1, as a Taylor
        // series of expm1(y)/y for |y| < 1/2 (truncation < 4e-6 relative),
        // e^y - 1 beyond; shifted bank: E = 2^(a v + b)
        const float xs = x - pc[u];
        const float y = pb[u] * xs;
        float poly = fmaf(y, 1.f / 720.f, 1.f / 120.f);
        poly = fmaf(y, poly, 1.f / 24.f);
        poly = fmaf(y, poly, 1.f / 6.f);
        poly = fmaf(y, poly, 0.5f);
        poly = fmaf(y, poly, 1.f);
        const float lin = fabsf(y) < 0.5f ? xs * poly : (ex2_approx(y * kLog2e) - 1.f) * pa[u];
        const float shf = ex2_approx(fmaf(pa[u], x, pb[u]));
        e[u] = __float2half_rn(plin[u] ? lin : shf);
      }
      *cell = *reinterpret_cast<const uint4 *>(e);
    }
  }
  // the tile of the bank leaves with one bulk store
  fence_proxy_async_smem();
  __syncthreads();
  if (tid == 0) {
    bulk_store(bank + (static_cast<size_t>(bh) * T + static_cast<size_t>(kt) * kBlockK) * D, smem_u32(tile_smem),
               static_cast<uint32_t>(rows * D * 2));
    bulk_commit_group();
  }
  if (causal) {
#pragma unroll
    for (int u = 0; u < 8; ++u)
      if (first[u] < kBlockK) atomicMin(&s_first[cc * 8 + u], first[u]);
  }
  if (!causal) {
    if (tid == 0) bulk_wait_group_read0();
    return;
  }
  __syncthreads();
  // rows r < max_j first_j of this tile get one entry with their channel masks
  __shared__ int s_rows;
  if (tid == 0) {
    int hz_max = 0;
    for (int j = 0; j < D; ++j) hz_max = max(hz_max, s_first[j]);
    s_rows = min(hz_max, T - kt * kBlockQ);
  }
  __syncthreads();
  const int n_rows = s_rows;
  int2 *tf = tilefix + static_cast<size_t>(bh) * n_kt + kt;
  if (n_rows <= 0) {
    if (tid == 0) {
      *tf = make_int2(0, 0);
      bulk_wait_group_read0();
    }
    return;
  }
  // the tile's entries take a multiple of 8 slots (padding rows -1), so the
  // fix-up's 8-entry chunks never straddle two tiles
  const int n_slots = (n_rows + 7) & ~7;
  __shared__ int s_base;
  if (tid == 0) {
    s_base = atomicAdd(fixup_count, n_slots);
    atomicAdd(fixup_rows, n_rows);
    *tf = make_int2(s_base, n_rows);
  }
  __syncthreads();
  for (int r = tid; r < n_slots; r += 128) {
    FixupEntry e;
    e.row = r < n_rows ? bh * T + kt * kBlockQ + r : -1;
#pragma unroll
    for (int g = 0; g < 4; ++g) {
      unsigned m = 0;
      for (int c = 0; c < 32; ++c) {
        const int j = 32 * g + c;
        if (j < D && r < n_rows && s_first[j] > r) m |= 1u << c;
      }
      e.mask[g] = m;
    }
    e.m_pre = -INFINITY;
    e.l_pre = 0.f;
    e.pad = 0;
    fixups[s_base + r] = e;
  }
  if (tid == 0) bulk_wait_group_read0();
}

cudaError_t launch_value_bank(const void *v, const float *beta, int BH, int H, int T, int d, int causal,
                              const BankWorkspace &w, unsigned *err, cudaStream_t stream) {
  const int n_kt = (T + kBlockK - 1) / kBlockK;
  const dim3 grid(n_kt, BH);
  const __nv_bfloat16 *vb = static_cast<const __nv_bfloat16 *>(v);
  if (d == 64) {
    tile_stats_kernel<64><<<grid, 128, kBlockK * 64 * 2, stream>>>(vb, T, w.tstat, err);
    plan_kernel<64><<<BH, 4 * 64, 0, stream>>>(w.tstat, beta, H, T, n_kt, w.chan, w.cpre, w.shift, w.rfac, w.colmask);
  } else if (d == 128) {
    tile_stats_kernel<128><<<grid, 128, kBlockK * 128 * 2, stream>>>(vb, T, w.tstat, err);
    plan_kernel<128><<<BH, 4 * 128, 0, stream>>>(w.tstat, beta, H, T, n_kt, w.chan, w.cpre, w.shift, w.rfac,
                                                 w.colmask);
  } else {
    return cudaErrorInvalidValue;
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (d == 64)
    bank_kernel<64><<<grid, 128, kBlockK * 64 * 2, stream>>>(vb, beta, w.chan, w.cpre, w.shift, H, T, causal, w.bank,
                                                             w.fixups, w.fixup_count, w.fixup_rows, w.tilefix, err);
  else
    bank_kernel<128><<<grid, 128, kBlockK * 128 * 2, stream>>>(vb, beta, w.chan, w.cpre, w.shift, H, T, causal,
                                                               w.bank, w.fixups, w.fixup_count, w.fixup_rows,
                                                               w.tilefix, err);
  return cudaGetLastError();
}

}  // namespace fem
