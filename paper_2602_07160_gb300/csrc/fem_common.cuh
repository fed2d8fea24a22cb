// Shared device-side definitions for the FEM read kernels (sm_103a).
//
// Inline-PTX wrappers for mbarriers, TMA tensor copies and the tcgen05
// tensor-core instructions (TMEM allocation, MMA, commit, TMEM loads/stores),
// the numerical constants of the read's value bank, and the bounded waits
// every kernel uses: a wait that does not complete within kWaitLimitNs sets a
// bit in the per-device error word and returns false instead of hanging.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace fem {

// ---------------------------------------------------------------------------
// Constants of the read's numerics.
//
// Value bank.  For each channel j the kernel mixes the prior weights against
// a bank built from v once per key tile.  The "linear" bank
//   D_ij = expm1(beta_j (v_ij - c_j)) / beta_j
// with a fixed anchor c_j read as o = c + log1p(beta * acc / L) / beta
// (o = c + acc/L at beta = 0) keeps the small-beta read free of the
// cancellation in LSE(s + beta v) - LSE(s).  A channel uses it when an anchor
// exists with
//   beta_j (c_j - min v) <= kLinearLowTilt     (1 + beta acc/L >= e^-1: no cancellation)
//   expm1(beta_j (max v - c_j)) / beta_j <= kLinearBankMax   (the bank fits fp16)
// and c_j is the channel mean clamped into that interval, so acc/L stays
// near zero and neither fp16 rounding of D nor a relative error of the fp32
// accumulation is magnified.  Every other channel uses the "shifted" bank
//   E_ij = exp(beta_j (v_ij - c_j) + kBankOffset)
// with a running shift c_j and reads o = c + (log(acc/L) - kBankOffset)/beta.
// Until c_j moves, E <= exp(kShiftLag + kBankOffset) = e^11 < 65504 (fp16);
// a larger lag means fewer tiles on which acc must be rescaled for a moved
// shift.
//
// Underflow guard.  The prior weights P <= 2^kRowMaxLag and the bank are
// rounded to fp16, whose normal range ends at 2^-14; below it values keep an
// absolute error up to 2^-25 (subnormal or flushed).  In the units of the
// final row maximum and shift, with L = sum_i P_i (fp32) and
// Ecol_j = sum_i |bank_ij| over the keys read, the accumulator's error from
// the subnormal range is at most 2^-25 (L + Ecol_j) (shifted bank; the P side
// through Ecol_j, the bank side through L) or 2^-25 Ecol_j in value units
// (linear bank, whose own subnormals are absolute errors in v).  An entry
// whose bound exceeds kGuardTau times what it can cost, i.e.
//   shifted: 2^-25 (L + Ecol_j) > kGuardTau * beta_j * acc_j,
//   linear:  2^-25 Ecol_j       > kGuardTau * (L + beta_j * acc_j),
// would move o_tj by more than kGuardTau and is recomputed exactly (peaked
// priors at large beta, where the read is carried by keys of tiny prior
// weight or a heavy key's value lies far below the shift; the first rows of
// a causal diagonal tile, whose shift includes keys they do not see).
// ---------------------------------------------------------------------------
constexpr float kLinearLowTilt = 1.0f;
constexpr float kLinearBankMax = 30000.f;  // fp16 holds values up to 65504
constexpr float kBankOffset = 4.0f;        // natural-log offset of the shifted bank
constexpr float kShiftLag = 7.0f;          // c_j moves only when beta*(new max - c) > this
constexpr float kRowMaxLag = 8.0f;         // row max moves only when it grows by > 2^this
constexpr float kGuardTau = 0.0078125f;    // 2^-7: largest output error the guard lets through
constexpr float kGuardUlp = 2.98023224e-08f * 1.0078125f;  // 2^-25 (fp16 subnormal half-spacing), with slack
                                                           // for sums taken before the fp16 rounding
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

constexpr int kBlockQ = 128;  // query rows per tile (TMEM lanes)
constexpr int kBlockK = 128;  // keys per tile
constexpr int kFixChunk = 8;  // fix-up entries per chunk: rows scored together, one warp each

// Error bits of the per-device error word.
constexpr unsigned kErrWaitTma = 1u;
constexpr unsigned kErrWaitMma = 2u;
constexpr unsigned kErrTmemAlloc = 4u;
constexpr unsigned kErrWaitProbe = 8u;  // the diagnostic wait probe gave up (fem_probe_wait_timeout)

constexpr unsigned long long kWaitLimitNs = 1000000000ull;  // 1 s per wait

// Per-channel statistics the pre-pass hands to the main kernel.
struct ChanInfo {
  float c_lin;   // anchor of the linear bank (unused by shifted channels)
  float linear;  // 1.0f when the channel uses the linear bank, else 0.0f
};

// One fix-up entry, written by the tensor-core kernel in blocks padded to a
// multiple of kFixChunk: row = (b*H + h)*T + t (-1: padding); channel 32*g + bit is recomputed exactly for every set bit of
// mask[g], over the key tiles kt0 .. the row's last one.  With kt0 > 0 (a
// causal row whose state before its diagonal tile passed the guard) the
// recomputation starts from that state: m_pre and l_pre, the row's running
// maximum (log2 units) and sum of 2^(s log2 e - m_pre) over the key tiles
// before kt0, and, in out[row][j], channel j's accumulator over them (the bank
// of tile kt0 - 1's shift).  With kt0 = 0 every key is taken again, and l_pre
// is 1 when the gated read's mean must be recomputed as well, 0 otherwise.
struct __align__(32) FixupEntry {
  int row;
  unsigned mask[4];
  float m_pre, l_pre;
  int kt0;
};

// A fix-up chunk that recomputes its rows from the first key tile over many
// tiles is split into segments of fix_seg_tiles(n_kt) key tiles that blocks
// take separately; each leaves its partial state in a pool slot and the last
// to finish merges them.  At most kFixPoolSlots chunks are split per read
// (later ones run whole); none when the sequence has fewer than
// kFixSplitMinTiles key tiles (at 8192 keys the longest such chunks cost no
// more than the spread of the last claims, and the claims' extra code cost
// 1 to 2 % of the step).
constexpr int kFixSegMin = 8;       // key tiles per segment, at least
constexpr int kFixMaxSeg = 16;      // segments per chunk, at most
constexpr int kFixPoolSlots = 128;  // chunks split at once
__host__ __device__ inline int fix_seg_tiles(int n_kt) {
  const int s = (n_kt + kFixMaxSeg - 1) / kFixMaxSeg;
  return s > kFixSegMin ? s : kFixSegMin;
}
constexpr int kFixSplitMinTiles = 128;
__host__ __device__ inline bool fix_split_on(int n_kt) { return n_kt >= kFixSplitMinTiles; }
__host__ __device__ inline int fix_max_segs(int n_kt) { return (n_kt + fix_seg_tiles(n_kt) - 1) / fix_seg_tiles(n_kt); }
// One split chunk: the chunk, its segment count, the next unclaimed segment,
// the segments finished, and ready = 1 once the others are written (all zero
// before the fix-up).
struct __align__(32) FixSlot {
  int chunk, n_seg, next, done, ready, pad[3];
};

// ---------------------------------------------------------------------------
// Small helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long global_timer_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ float lg2_approx(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float rcp_approx(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// max(a, max(b, c)) in one instruction (three-operand max.f32, sm_100 and later).
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// ---------------------------------------------------------------------------
// mbarrier
// ---------------------------------------------------------------------------
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

// Programmatic dependent launch: a kernel launched with the programmatic
// stream-serialisation attribute may start while the previous kernel of its
// stream still runs; it waits here, before touching any global memory that
// kernel (or one before it) writes or reads, for that kernel's completion and
// the visibility of its writes.  Without the attribute the wait returns at once.
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
// Lets the next kernel of the stream be scheduled once every block of this one
// has started (or passed here): its blocks then take the SMs this kernel's tail
// leaves idle and run their prologue up to their own wait.
__device__ __forceinline__ void grid_dep_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" :::); }

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(done)
      : "r"(bar), "r"(parity)
      : "memory");
  return done != 0;
}

// try_wait that lets the thread sleep (up to ~hint_ns) until the phase
// completes instead of spinning.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint32_t bar, uint32_t parity, uint32_t hint_ns) {
  uint32_t done;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(done)
      : "r"(bar), "r"(parity), "r"(hint_ns)
      : "memory");
  return done != 0;
}


// Waits for the phase with the given parity to complete.  Gives up after
// limit_ns, records `code` in the error word and returns false.
__device__ __forceinline__ bool mbar_wait_for(uint32_t bar, uint32_t parity, unsigned *err, unsigned code,
                                              unsigned long long limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = global_timer_ns();
  while (true) {
    for (int i = 0; i < 64; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (global_timer_ns() - t0 > limit_ns) {
      atomicOr(err, code);
      return false;
    }
  }
}

// mbar_wait_for with the kernels' limit, kWaitLimitNs.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, unsigned *err, unsigned code) {
  return mbar_wait_for(bar, parity, err, code, kWaitLimitNs);
}

// ---------------------------------------------------------------------------
// Async-proxy fences and TMA
// ---------------------------------------------------------------------------
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// 3-D tiled TMA load into shared memory, completion via mbarrier tx bytes.
// Coordinates are element indices {x (innermost), y, z}.
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *map, uint32_t bar, int x, int y,
                                            int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, %5}], "
      "[%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y), "r"(z)
      : "memory");
}

// Plain bulk copy global -> shared (16-byte aligned addresses, size a multiple
// of 16), completion via mbarrier tx bytes.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar)
               : "memory");
}

// Plain bulk copy shared -> global (16-byte aligned addresses, size a multiple
// of 16), bulk-group completion.
__device__ __forceinline__ void bulk_store(void *dst, uint32_t src, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(reinterpret_cast<uint64_t>(dst)),
               "r"(src), "r"(bytes)
               : "memory");
}

// 3-D tiled TMA store from shared memory (bulk-group completion).  Rows
// outside the tensor's extent are not written.
__device__ __forceinline__ void tma_store_3d(const CUtensorMap *map, uint32_t src, int x, int y, int z) {
  asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.tile.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(src), "r"(x), "r"(y), "r"(z)
               : "memory");
}
__device__ __forceinline__ void bulk_commit_group() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// Waits until every committed bulk store has finished reading shared memory.
__device__ __forceinline__ void bulk_wait_group_read0() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
// Wait until at most N committed bulk groups still read shared memory.
template <int N>
__device__ __forceinline__ void bulk_wait_group_read() {
  asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}

// Named barrier over `nthreads` threads that returns the AND of `v` over them.
__device__ __forceinline__ bool bar_and(int id, int nthreads, bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 q, %1, 0;\n\t"
      "bar.red.and.pred p, %2, %3, q;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(v)), "r"(id), "r"(nthreads)
      : "memory");
  return r != 0;
}
__device__ __forceinline__ void bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap *map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// ---------------------------------------------------------------------------
// tcgen05: TMEM allocation
// ---------------------------------------------------------------------------
// Warp-collective: writes the TMEM base address to shared memory at `dst`.
__device__ __forceinline__ void tmem_alloc(uint32_t dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

__device__ __forceinline__ void tc_fence_before_sync() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after_sync() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// ---------------------------------------------------------------------------
// tcgen05: descriptors and MMA
// ---------------------------------------------------------------------------
// Shared-memory matrix descriptor for a 128-byte-swizzled operand.
//   bits  0-13 : start address >> 4
//   bits 16-29 : leading-dimension byte offset >> 4
//   bits 32-45 : stride-dimension byte offset >> 4
//   bits 46-47 : descriptor version (1 for tcgen05)
//   bits 61-63 : swizzle mode (2 = 128-byte swizzle)
// K-major operand: rows of 128 bytes (64 16-bit elements), 8-row groups
// 1024 bytes apart (SBO); LBO unused.  MN-major operand: K rows of 128
// bytes, 8-row groups SBO apart, 64-element MN blocks LBO apart.
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr, uint32_t lbo_bytes, uint32_t sbo_bytes) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>((lbo_bytes >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>((sbo_bytes >> 4) & 0x3FFFu) << 32;
  d |= 1ull << 46;
  d |= 2ull << 61;
  return d;
}

// Instruction descriptor of tcgen05.mma kind::f16 with fp32 accumulation.
//   bits 4-5 : D format (1 = f32);  bits 7-9 / 10-12 : A / B format (0 = f16,
//   1 = bf16);  bit 15 / 16 : A / B major (0 = K-major, 1 = MN-major);
//   bits 17-22 : N >> 3;  bits 24-28 : M >> 4.
__host__ __device__ constexpr uint32_t idesc_f16(int M, int N, bool ab_bf16, bool b_mn_major) {
  return (1u << 4) | ((ab_bf16 ? 1u : 0u) << 7) | ((ab_bf16 ? 1u : 0u) << 10) | ((b_mn_major ? 1u : 0u) << 16) |
         (static_cast<uint32_t>(N >> 3) << 17) | (static_cast<uint32_t>(M >> 4) << 24);
}

// D[tmem] (+)= A[smem] * B[smem]^T, issued by one thread.
__device__ __forceinline__ void mma_f16_ss(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                           uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// D[tmem] (+)= A[tmem] * B[smem]^T, issued by one thread.
__device__ __forceinline__ void mma_f16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                           uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive on `bar` once every tcgen05 operation this thread issued so far is done.
__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}

// ---------------------------------------------------------------------------
// tcgen05: TMEM <-> registers.  32x32b shape: thread i of the warp accesses
// TMEM lane (warp's lane quarter base + i); .x32 moves 32 consecutive 32-bit
// columns.
// ---------------------------------------------------------------------------
#define FEM_R8(b) "=r"(r[b + 0]), "=r"(r[b + 1]), "=r"(r[b + 2]), "=r"(r[b + 3]), "=r"(r[b + 4]), "=r"(r[b + 5]), \
                  "=r"(r[b + 6]), "=r"(r[b + 7])
#define FEM_W8(b) "r"(r[b + 0]), "r"(r[b + 1]), "r"(r[b + 2]), "r"(r[b + 3]), "r"(r[b + 4]), "r"(r[b + 5]), \
                  "r"(r[b + 6]), "r"(r[b + 7])

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : FEM_R8(0), FEM_R8(8), FEM_R8(16), FEM_R8(24)
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      FEM_W8(0), FEM_W8(8), FEM_W8(16), FEM_W8(24)
      : "memory");
}

__device__ __forceinline__ uint32_t tmem_ld1(uint32_t taddr) {
  uint32_t r;
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];" : "=r"(r) : "r"(taddr));
  return r;
}

__device__ __forceinline__ void tmem_st1(uint32_t taddr, uint32_t r) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x1.b32 [%0], {%1};" ::"r"(taddr), "r"(r) : "memory");
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      FEM_W8(0), FEM_W8(8)
      : "memory");
}

#undef FEM_R8
#undef FEM_W8

__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Byte offset of the 16-byte chunk holding elements [8*chunk, 8*chunk+8) of
// `row` in a 128-byte-swizzled tile of 64-element (128-byte) rows.
__host__ __device__ __forceinline__ uint32_t sw128_offset(uint32_t row, uint32_t chunk) {
  return row * 128u + ((chunk ^ (row & 7u)) << 4);
}

}  // namespace fem
