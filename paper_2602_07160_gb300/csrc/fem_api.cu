// C ABI of libfem.so (declared in include/fem.h): argument checks, workspace
// layout, TMA tensor maps and the launch sequence of the FEM read.
//
// bf16 path, in stream order:
//   1. tile_stats, plan, bank: channel modes, shift schedule, the fp16 value
//      bank (once per key tile) and its column sums
//   2. fem_tc (tcgen05): the read for every row and channel, and the list of
//      entries its underflow guard rejects
//   3. fixup: the listed entries recomputed exactly, from the state fem_tc
//      left before their diagonal tile or over every key tile
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <vector>

#include "fem.h"
#include "fem_chunks.h"
#include "fem_launch.h"

namespace fem {
namespace {

__device__ unsigned g_error_word;
__device__ int g_last_fixup;
__device__ unsigned g_beta_bad;  // FEM_DEBUG: set when a beta entry is negative, NaN or infinite

constexpr int kMaxDevices = 64;

struct DeviceState {
  bool ready = false;
  unsigned *err = nullptr;
  int *last_fixup = nullptr;
  int num_sms = 0;
  // stream-ordered workspaces come from this pool, which keeps freed memory for
  // the next call instead of returning it to the driver at every synchronisation
  cudaMemPool_t pool = nullptr;
  unsigned *beta_bad = nullptr;
  // copy streams of fem_fwd_host, created on its first call
  cudaStream_t copy_in = nullptr, copy_out = nullptr;
};

std::mutex g_mutex;
thread_local cudaEvent_t t_ev_start = nullptr, t_ev_stop = nullptr;
DeviceState g_dev[kMaxDevices];
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

int map_cuda(cudaError_t e) {
  if (e == cudaSuccess) return FEM_OK;
  if (e == cudaErrorMemoryAllocation) return FEM_ERR_NO_MEMORY;
  return FEM_ERR_CUDA;
}

// Per-device addresses of the error word and fix-up counter, SM count and the
// tensor-map encoder, set up once with the device current.  No allocation.
int device_state(DeviceState **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return FEM_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mutex);
  DeviceState &s = g_dev[dev];
  if (!s.ready) {
    if (cudaGetSymbolAddress(reinterpret_cast<void **>(&s.err), g_error_word) != cudaSuccess) return FEM_ERR_CUDA;
    if (cudaGetSymbolAddress(reinterpret_cast<void **>(&s.last_fixup), g_last_fixup) != cudaSuccess)
      return FEM_ERR_CUDA;
    if (cudaDeviceGetAttribute(&s.num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return FEM_ERR_CUDA;
    if (cudaGetSymbolAddress(reinterpret_cast<void **>(&s.beta_bad), g_beta_bad) != cudaSuccess) return FEM_ERR_CUDA;
    if (!g_encode) {
      cudaDriverEntryPointQueryResult q;
      void *fn = nullptr;
      if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
              cudaSuccess ||
          q != cudaDriverEntryPointSuccess || !fn)
        return FEM_ERR_CUDA;
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    s.ready = true;
  }
  *out = &s;
  return FEM_OK;
}

// FEM_DEBUG=1 (read once, at the first check): the entry points that take beta check it (beta >= 0
// and finite) before they enqueue the computation, a synchronisation of the stream each.
bool fem_debug() {
  static const bool on = [] {
    const char *e = std::getenv("FEM_DEBUG");
    return e != nullptr && *e != 0 && std::strcmp(e, "0") != 0;
  }();
  return on;
}

__global__ void beta_check_kernel(const float *__restrict__ beta, int n, unsigned *bad) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
    const float b = beta[i];
    if (!(b >= 0.f) || b == INFINITY) atomicOr(bad, 1u);
  }
}

// FEM_OK unless FEM_DEBUG is on and beta [n] (device) holds a negative, NaN or infinite entry
// (FEM_ERR_INVALID_ARG); a failing CUDA call gives FEM_ERR_CUDA.
int debug_check_beta(const float *beta, long long n, DeviceState *ds, cudaStream_t s) {
  if (!fem_debug()) return FEM_OK;
  if (n <= 0 || n > (1ll << 30)) return FEM_ERR_INVALID_ARG;
  unsigned bad = 0;
  cudaError_t e = cudaMemsetAsync(ds->beta_bad, 0, sizeof(unsigned), s);
  if (e == cudaSuccess) {
    beta_check_kernel<<<static_cast<int>(std::min<long long>((n + 255) / 256, 1024)), 256, 0, s>>>(
        beta, static_cast<int>(n), ds->beta_bad);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaMemcpyAsync(&bad, ds->beta_bad, sizeof(unsigned), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return FEM_ERR_CUDA;
  return bad ? FEM_ERR_INVALID_ARG : FEM_OK;
}

// the same for beta in host memory
int debug_check_beta_host(const float *beta, long long n) {
  if (!fem_debug()) return FEM_OK;
  for (long long i = 0; i < n; ++i)
    if (!(beta[i] >= 0.f) || beta[i] == INFINITY) return FEM_ERR_INVALID_ARG;
  return FEM_OK;
}

// Stream-ordered workspace from the device's library pool (free with
// cudaFreeAsync).  The pool is created by the first entry point that
// allocates on the device.
cudaError_t ws_alloc(DeviceState *ds, void **p, size_t bytes, cudaStream_t s) {
  {
    std::lock_guard<std::mutex> lock(g_mutex);
    if (!ds->pool) {
      int dev = 0;
      cudaError_t e = cudaGetDevice(&dev);
      if (e != cudaSuccess) return e;
      cudaMemPoolProps props = {};
      props.allocType = cudaMemAllocationTypePinned;
      props.location.type = cudaMemLocationTypeDevice;
      props.location.id = dev;
      cudaMemPool_t pool = nullptr;
      if ((e = cudaMemPoolCreate(&pool, &props)) != cudaSuccess) return e;
      uint64_t keep = ~uint64_t(0);
      if ((e = cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &keep)) != cudaSuccess) {
        cudaMemPoolDestroy(pool);
        return e;
      }
      ds->pool = pool;
    }
  }
  return cudaMallocFromPoolAsync(p, bytes, ds->pool, s);
}

// [BH, T, d] row-major tensor; boxes of box_rows rows x 128 bytes (64 16-bit
// or 32 32-bit elements), 128-byte swizzle.
int make_map(CUtensorMap *map, const void *base, int BH, int T, int d,
             CUtensorMapDataType dtype = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, int elem_bytes = 2, int box_rows = 128) {
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(T), static_cast<cuuint64_t>(BH)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(d) * elem_bytes, static_cast<cuuint64_t>(T) * d * elem_bytes};
  cuuint32_t box[3] = {static_cast<cuuint32_t>(128 / elem_bytes), static_cast<cuuint32_t>(box_rows), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_encode(map, dtype, 3, const_cast<void *>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? FEM_OK : FEM_ERR_CUDA;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t round256(size_t x) { return (x + 255) & ~size_t(255); }

// The counters zeroed before every read: four ints, then the fix-up's split slots.
constexpr size_t kCountBytes = 256 + kFixPoolSlots * sizeof(FixSlot);

struct WsLayout {
  size_t tstat, chan, bcoef, shift, rfac, colsum, colmask, bank, fixups, count, fixpart, total;
};

// Head dimensions of the bf16 read that run on CUDA cores (no workspace but the counters).
bool small_d(int d) { return d == 16 || d == 32; }

bool ws_layout(int B, int H, int T, int d, int causal, WsLayout *w) {
  (void)causal;  // the guard's fix-up list serves both forms of the read
  if (B <= 0 || H <= 0 || T <= 0 || d <= 0) return false;
  if (small_d(d)) {
    *w = WsLayout{};
    w->count = 0;
    w->total = 256;
    return true;
  }
  const size_t BH = static_cast<size_t>(B) * H;
  const size_t n_kt = (static_cast<size_t>(T) + kBlockK - 1) / kBlockK;
  size_t off = 0;
  w->bank = off;
  off += round256(BH * static_cast<size_t>(T) * d * 2);
  w->tstat = off;
  off += round256(BH * n_kt * d * sizeof(float4));
  w->chan = off;
  off += round256(BH * d * sizeof(ChanInfo));
  w->bcoef = off;
  off += round256(BH * n_kt * d * sizeof(float4));
  w->shift = off;
  off += round256(BH * n_kt * d * sizeof(float));
  w->rfac = off;
  off += round256(BH * n_kt * d * sizeof(float));
  w->colsum = off;
  off += round256(BH * n_kt * d * sizeof(float));
  w->colmask = off;
  off += round256(BH * n_kt * 4 * sizeof(unsigned));
  w->fixups = off;
  off += round256(fixup_capacity(BH, static_cast<size_t>(T)) * sizeof(FixupEntry));
  w->count = off;  // fix-up slots, fix-up rows, the fix-up's chunk counter, split chunks; then the split slots
  off += kCountBytes;
  w->fixpart = off;
  if (fix_split_on(static_cast<int>(n_kt)))
    off += round256(static_cast<size_t>(kFixPoolSlots) * fix_max_segs(static_cast<int>(n_kt)) * kFixChunk *
                    (2 + 4 * static_cast<size_t>(d)) * sizeof(float));
  w->total = off;
  return true;
}

int check_common(const void *q, const void *k, const void *v, const float *beta, const float *out, const float *lse,
                 int B, int H, int T, int d, int causal) {
  if (!q || !k || !v || !beta || !out) return FEM_ERR_INVALID_ARG;
  if (B <= 0 || H <= 0 || T <= 0 || d <= 0) return FEM_ERR_INVALID_ARG;
  if (causal != 0 && causal != 1) return FEM_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out)) return FEM_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(beta) & 3u) || (lse && (reinterpret_cast<uintptr_t>(lse) & 3u)))
    return FEM_ERR_INVALID_ARG;
  const long long rows = static_cast<long long>(B) * H * T;
  if (rows >= (1ll << 31) || static_cast<long long>(B) * H > 65535) return FEM_ERR_UNSUPPORTED;
  return FEM_OK;
}

// Sizes the tensor-core read takes: d in {64, 128} and T up to kMaxSeqLen.
int check_tc_sizes(int T, int d) {
  if (d != 64 && d != 128) return FEM_ERR_UNSUPPORTED;
  if (T > kMaxSeqLen) return FEM_ERR_UNSUPPORTED;
  return FEM_OK;
}

// Sizes the plain bf16 read takes: the tensor-core sizes, and d in {16, 32} on CUDA cores.
int check_read_sizes(int T, int d) { return small_d(d) ? FEM_OK : check_tc_sizes(T, d); }

// ---------------------------------------------------------------------------
// Fixed scratch for fem_fwd_noalloc.  Some callers may not allocate device
// memory while they run the read (for example a plugin whose execute callback
// must not allocate, or a service that hands out all device memory up front),
// so that entry point uses this file-scope array as its workspace instead of
// cudaMallocAsync.  Every GPU that loads the library holds it until exit.
// Host code must not use the array's name as a device address; the entry
// point looks the address up once per device with cudaGetSymbolAddress.
// ---------------------------------------------------------------------------
constexpr size_t kStaticScratchBytes = size_t(16) << 20;  // 16 MiB
static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

std::mutex g_static_mutex;
void *g_static_addr[kMaxDevices] = {};

// Device address of g_static_scratch on the current device (set up on the
// first call per device, with that device current).
int static_scratch(void **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return FEM_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_static_mutex);
  if (!g_static_addr[dev]) {
    void *ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_static_scratch) != cudaSuccess || !ptr) return FEM_ERR_CUDA;
    g_static_addr[dev] = ptr;
  }
  *out = g_static_addr[dev];
  return FEM_OK;
}

// The error path of the bounded waits, exercised on purpose: one thread waits
// on an mbarrier of its own that nothing arrives on, with the library's wait
// helper and a short limit; the helper gives up, records kErrWaitProbe in the
// error word and the kernel returns.  No copy or tensor-core operation is
// issued, so nothing is left in flight.
__global__ void wait_probe_kernel(unsigned *err, unsigned long long limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  mbar_init(smem_u32(&bar), 1);
  fence_mbar_init();
  mbar_wait_for(smem_u32(&bar), 0, err, kErrWaitProbe, limit_ns);
}

}  // namespace
}  // namespace fem

using namespace fem;

extern "C" {

const char *fem_status_str(int status) {
  switch (status) {
    case FEM_OK: return "FEM_OK";
    case FEM_ERR_INVALID_ARG: return "FEM_ERR_INVALID_ARG";
    case FEM_ERR_UNSUPPORTED: return "FEM_ERR_UNSUPPORTED";
    case FEM_ERR_CUDA: return "FEM_ERR_CUDA";
    case FEM_ERR_TIMEOUT: return "FEM_ERR_TIMEOUT";
    case FEM_ERR_NO_MEMORY: return "FEM_ERR_NO_MEMORY";
    default: return "FEM_ERR_UNKNOWN";
  }
}

size_t fem_fwd_workspace_bytes(int B, int H, int T, int d, int causal) {
  WsLayout w;
  if (!ws_layout(B, H, T, d, causal ? 1 : 0, &w)) return 0;
  return w.total;
}

// The read's workspace arrays at `ws` (layout ws_layout).
static BankWorkspace bank_workspace(uint8_t *ws, const WsLayout &w) {
  BankWorkspace bw;
  bw.tstat = reinterpret_cast<float4 *>(ws + w.tstat);
  bw.chan = reinterpret_cast<ChanInfo *>(ws + w.chan);
  bw.bcoef = reinterpret_cast<float4 *>(ws + w.bcoef);
  bw.shift = reinterpret_cast<float *>(ws + w.shift);
  bw.rfac = reinterpret_cast<float *>(ws + w.rfac);
  bw.colsum = reinterpret_cast<float *>(ws + w.colsum);
  bw.colmask = reinterpret_cast<unsigned *>(ws + w.colmask);
  bw.bank = reinterpret_cast<__half *>(ws + w.bank);
  bw.fixups = reinterpret_cast<FixupEntry *>(ws + w.fixups);
  bw.fixup_count = reinterpret_cast<int *>(ws + w.count);
  bw.fixup_rows = reinterpret_cast<int *>(ws + w.count) + 1;
  bw.fixup_next = reinterpret_cast<int *>(ws + w.count) + 2;
  bw.fix_long = reinterpret_cast<int *>(ws + w.count) + 3;
  bw.fix_slots = reinterpret_cast<FixSlot *>(ws + w.count + 256);
  bw.fix_part = w.total > w.fixpart ? reinterpret_cast<float *>(ws + w.fixpart) : nullptr;
  return bw;
}

// Gated part of a read: the mean's pre-pass workspace (ws_layout, non-causal)
// and its zero beta, the gates, and mu_side (the mean at the fix-up entries).
struct GatedArgs {
  uint8_t *ws0;
  const float *zero_beta, *lam, *g;
  float *mu_side;
};

// The read at beta (the plain read, or with ga the one-pass gated read at
// beta_max = beta) into out and lse, with the arguments already checked.
static int fwd_impl(const void *q, const void *k, const void *v, const float *beta, float *out, float *lse, int B,
                    int H, int T, int d, int causal, uint8_t *ws, const GatedArgs *ga, DeviceState *ds,
                    cudaStream_t s) {
  const int BH = B * H;
  if (small_d(d) && !ga) {
    // CUDA cores, exact to fp32 rounding: no bank, no guard, no fix-up rows
    cudaError_t e = cudaMemsetAsync(ds->last_fixup, 0, sizeof(int), s);
    const cudaEvent_t ev0 = t_ev_start, ev1 = t_ev_stop;
    t_ev_start = t_ev_stop = nullptr;
    if (e == cudaSuccess && ev0) e = cudaEventRecord(ev0, s);
    if (e == cudaSuccess) e = launch_simt_bf16(q, k, v, beta, out, lse, B, H, T, d, causal, s);
    if (e == cudaSuccess && ev1) e = cudaEventRecord(ev1, s);
    return map_cuda(e);
  }
  WsLayout w;
  ws_layout(B, H, T, d, causal, &w);
  BankWorkspace bw = bank_workspace(ws, w);
  CUtensorMap tq, tk, tv, te, te0;
  int rc;
  if ((rc = make_map(&tq, q, BH, T, d)) != FEM_OK) return rc;
  if ((rc = make_map(&tk, k, BH, T, d)) != FEM_OK) return rc;
  if ((rc = make_map(&tv, v, BH, T, d)) != FEM_OK) return rc;
  if ((rc = make_map(&te, bw.bank, BH, T, d, CU_TENSOR_MAP_DATA_TYPE_FLOAT16)) != FEM_OK) return rc;
  BankWorkspace bw0;
  TcGate gate;
  if (ga) {
    WsLayout w0;
    ws_layout(B, H, T, d, 0, &w0);
    bw0 = bank_workspace(ga->ws0, w0);
    if ((rc = make_map(&te0, bw0.bank, BH, T, d, CU_TENSOR_MAP_DATA_TYPE_FLOAT16)) != FEM_OK) return rc;
    gate = TcGate{ga->lam, ga->g, ga->mu_side, bw0.chan, bw0.colsum};
  }

  // the four counters, and the split slots when the fix-up may split
  cudaError_t e = cudaMemsetAsync(bw.fixup_count, 0, bw.fix_part ? kCountBytes : 4 * sizeof(int), s);
  // the mean's bank (every channel linear at beta = 0: v - c with c the channel mean)
  if (e == cudaSuccess && ga)
    e = launch_value_bank(v, tv, te0, ga->zero_beta, BH, H, T, d, bw0, ds->err, ds->num_sms, s);
  if (ga) bw.tstat = bw0.tstat;  // the tiles' statistics do not depend on beta
  if (e == cudaSuccess)
    e = launch_value_bank(v, tv, te, beta, BH, H, T, d, bw, ds->err, ds->num_sms, s, ga != nullptr);
  const cudaEvent_t ev0 = t_ev_start, ev1 = t_ev_stop;
  t_ev_start = t_ev_stop = nullptr;
  // the read and the fix-up are programmatic dependent launches on the kernel before them (their
  // blocks take the SMs of its tail and wait there), unless events bracket the read.  The pre-pass
  // kernels launched that way ran slower (+0.9 % per step at the headline).
  const bool pdl = ev0 == nullptr && ev1 == nullptr;
  if (e == cudaSuccess && ev0) e = cudaEventRecord(ev0, s);
  if (e == cudaSuccess)
    e = launch_tc(d, tq, tk, te, ga ? &te0 : nullptr, out, beta, bw, lse, BH, H, T, causal, ga ? &gate : nullptr,
                  ds->err, s, pdl);
  if (e == cudaSuccess && ev1) e = cudaEventRecord(ev1, s);
  if (e == cudaSuccess)
    e = launch_fixup(q, k, v, beta, bw.chan, bw.shift, out, H, T, d, causal, bw.fixups, bw.fixup_count,
                     bw.fixup_rows, bw.fixup_next, ds->last_fixup, ga ? &gate : nullptr, bw.fix_long, bw.fix_slots,
                     bw.fix_part, ds->num_sms, s, pdl);
  return map_cuda(e);
}

int fem_fwd_ws(const void *q, const void *k, const void *v, const float *beta, float *out, float *lse, int B, int H,
               int T, int d, int causal, void *workspace, size_t workspace_bytes, void *stream) {
  int rc = check_common(q, k, v, beta, out, lse, B, H, T, d, causal);
  if (rc != FEM_OK) return rc;
  if ((rc = check_read_sizes(T, d)) != FEM_OK) return rc;
  WsLayout w;
  ws_layout(B, H, T, d, causal, &w);
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u)) return FEM_ERR_INVALID_ARG;
  if (workspace_bytes < w.total) return FEM_ERR_NO_MEMORY;
  DeviceState *ds = nullptr;
  if ((rc = device_state(&ds)) != FEM_OK) return rc;
  if ((rc = debug_check_beta(beta, static_cast<long long>(H) * d, ds, static_cast<cudaStream_t>(stream))) != FEM_OK)
    return rc;
  return fwd_impl(q, k, v, beta, out, lse, B, H, T, d, causal, static_cast<uint8_t *>(workspace), nullptr, ds,
                  static_cast<cudaStream_t>(stream));
}

int fem_fwd(const void *q, const void *k, const void *v, const float *beta, float *out, float *lse, int B, int H,
            int T, int d, int causal, void *stream) {
  int rc = check_common(q, k, v, beta, out, lse, B, H, T, d, causal);
  if (rc != FEM_OK) return rc;
  if ((rc = check_read_sizes(T, d)) != FEM_OK) return rc;
  DeviceState *ds = nullptr;
  if ((rc = device_state(&ds)) != FEM_OK) return rc;
  if ((rc = debug_check_beta(beta, static_cast<long long>(H) * d, ds, static_cast<cudaStream_t>(stream))) != FEM_OK)
    return rc;
  const size_t bytes = fem_fwd_workspace_bytes(B, H, T, d, causal);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  void *ws = nullptr;
  cudaError_t e = ws_alloc(ds, &ws, bytes, s);
  if (e != cudaSuccess) return map_cuda(e);
  rc = fem_fwd_ws(q, k, v, beta, out, lse, B, H, T, d, causal, ws, bytes, stream);
  e = cudaFreeAsync(ws, s);
  if (rc != FEM_OK) return rc;
  return map_cuda(e);
}

int fem_fwd_gated(const void *q, const void *k, const void *v, const float *beta_max, const float *lam,
                  const float *gate, float *out, float *lse, int B, int H, int T, int d, int causal, void *stream) {
  int rc = check_common(q, k, v, beta_max, out, lse, B, H, T, d, causal);
  if (rc != FEM_OK) return rc;
  if (!lam || !gate || !aligned16(lam) || !aligned16(gate)) return FEM_ERR_INVALID_ARG;
  if ((rc = check_tc_sizes(T, d)) != FEM_OK) return rc;
  DeviceState *ds = nullptr;
  if ((rc = device_state(&ds)) != FEM_OK) return rc;
  if ((rc = debug_check_beta(beta_max, static_cast<long long>(H) * d, ds, static_cast<cudaStream_t>(stream))) != FEM_OK)
    return rc;
  // workspace: the beta_max read's, the mean's pre-pass (non-causal layout),
  // a zero beta [H, d], and mu_side [B, H, T, d] fp32 for the fix-up's entries
  // (the guard can list entries of either mask)
  const size_t n = static_cast<size_t>(B) * H * T * d;
  const size_t ws_bytes = round256(fem_fwd_workspace_bytes(B, H, T, d, causal));
  const size_t ws0_bytes = round256(fem_fwd_workspace_bytes(B, H, T, d, 0));
  const size_t zb_bytes = round256(static_cast<size_t>(H) * d * sizeof(float));
  const size_t mu_bytes = round256(n * sizeof(float));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  void *buf = nullptr;
  cudaError_t e = ws_alloc(ds, &buf, ws_bytes + ws0_bytes + zb_bytes + mu_bytes, s);
  if (e != cudaSuccess) return map_cuda(e);
  uint8_t *p = static_cast<uint8_t *>(buf);
  GatedArgs ga;
  ga.ws0 = p + ws_bytes;
  ga.zero_beta = reinterpret_cast<const float *>(p + ws_bytes + ws0_bytes);
  ga.lam = lam;
  ga.g = gate;
  ga.mu_side = reinterpret_cast<float *>(p + ws_bytes + ws0_bytes + zb_bytes);
  e = cudaMemsetAsync(const_cast<float *>(ga.zero_beta), 0, static_cast<size_t>(H) * d * sizeof(float), s);
  rc = map_cuda(e);
  if (rc == FEM_OK) rc = fwd_impl(q, k, v, beta_max, out, lse, B, H, T, d, causal, p, &ga, ds, s);
  e = cudaFreeAsync(buf, s);
  if (rc != FEM_OK) return rc;
  return map_cuda(e);
}

int fem_bwd_f32(const float *q, const float *k, const float *v, const float *beta, const float *out, const float *lse,
                const float *dout, float *dq, float *dk, float *dv, float *dbeta, int B, int H, int T, int d,
                int causal, void *stream) {
  int rc = check_common(q, k, v, beta, out, lse, B, H, T, d, causal);
  if (rc != FEM_OK) return rc;
  if (!lse || !dout || !dq || !dk || !dv || !dbeta) return FEM_ERR_INVALID_ARG;
  for (const void *p : {static_cast<const void *>(dout), static_cast<const void *>(dq), static_cast<const void *>(dk),
                        static_cast<const void *>(dv)})
    if (!aligned16(p)) return FEM_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(dbeta) & 3u) return FEM_ERR_INVALID_ARG;
  if (d > 256) return FEM_ERR_UNSUPPORTED;
  DeviceState *ds = nullptr;
  if ((rc = device_state(&ds)) != FEM_OK) return rc;
  if ((rc = debug_check_beta(beta, static_cast<long long>(H) * d, ds, static_cast<cudaStream_t>(stream))) != FEM_OK)
    return rc;
  return map_cuda(launch_bwd_f32(q, k, v, beta, out, lse, dout, dq, dk, dv, dbeta, B, H, T, d, causal,
                                 static_cast<cudaStream_t>(stream)));
}

int fem_tdc_conv(const float *s, const float *u, float *h, int B, int T, int Hc, void *stream) {
  if (!s || !u || !h) return FEM_ERR_INVALID_ARG;
  if (B <= 0 || T <= 0 || Hc <= 0) return FEM_ERR_INVALID_ARG;
  for (const void *p : {static_cast<const void *>(s), static_cast<const void *>(u), static_cast<const void *>(h)})
    if (reinterpret_cast<uintptr_t>(p) & 3u) return FEM_ERR_INVALID_ARG;
  if (B > 65535 || static_cast<long long>(B) * T * Hc >= (1ll << 40)) return FEM_ERR_UNSUPPORTED;
  DeviceState *ds = nullptr;
  int rc = device_state(&ds);
  if (rc != FEM_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  void *ws = nullptr;
  const size_t bytes = tdc_workspace_bytes(B, T, Hc);  // 0: the one-launch form, no workspace
  if (bytes == 0) return map_cuda(launch_tdc(s, u, h, B, T, Hc, nullptr, st));
  cudaError_t e = ws_alloc(ds, &ws, bytes, st);
  if (e != cudaSuccess) return map_cuda(e);
  rc = map_cuda(launch_tdc(s, u, h, B, T, Hc, ws, st));
  e = cudaFreeAsync(ws, st);
  if (rc != FEM_OK) return rc;
  return map_cuda(e);
}

int fem_gla_fwd_tc(const float *qf, const float *kf, const float *v, const float *logdecay, const float *beta,
                   float *out, float *logz, int B, int H, int T, int m, int d, void *stream) {
  if (!qf || !kf || !v || !logdecay || !beta || !out) return FEM_ERR_INVALID_ARG;
  if (B <= 0 || H <= 0 || T <= 0 || m <= 0 || d <= 0) return FEM_ERR_INVALID_ARG;
  if (!aligned16(qf) || !aligned16(kf) || !aligned16(v) || !aligned16(out)) return FEM_ERR_INVALID_ARG;
  for (const void *p : {static_cast<const void *>(logdecay), static_cast<const void *>(beta),
                        static_cast<const void *>(logz)})
    if (p && (reinterpret_cast<uintptr_t>(p) & 3u)) return FEM_ERR_INVALID_ARG;
  if (m != 64 || d != 64) return FEM_ERR_UNSUPPORTED;
  if (static_cast<long long>(B) * H > 2147483647ll || static_cast<long long>(B) * H * T * 64 >= (1ll << 40))
    return FEM_ERR_UNSUPPORTED;
  DeviceState *ds = nullptr;
  int rc = device_state(&ds);
  if (rc != FEM_OK) return rc;
  if ((rc = debug_check_beta(beta, static_cast<long long>(H) * d, ds, static_cast<cudaStream_t>(stream))) != FEM_OK)
    return rc;
  return map_cuda(launch_gla_tc(qf, kf, v, logdecay, beta, out, logz, B, H, T, ds->err,
                                static_cast<cudaStream_t>(stream)));
}

int fem_gla_fwd(const float *qf, const float *kf, const float *v, const float *logdecay, const float *beta, float *out,
                float *logz, int B, int H, int T, int m, int d, void *stream) {
  if (!qf || !kf || !v || !logdecay || !beta || !out) return FEM_ERR_INVALID_ARG;
  if (B <= 0 || H <= 0 || T <= 0 || m <= 0 || d <= 0) return FEM_ERR_INVALID_ARG;
  if (!aligned16(qf) || !aligned16(kf)) return FEM_ERR_INVALID_ARG;
  for (const void *p : {static_cast<const void *>(v), static_cast<const void *>(logdecay),
                        static_cast<const void *>(beta), static_cast<const void *>(out),
                        static_cast<const void *>(logz)})
    if (p && (reinterpret_cast<uintptr_t>(p) & 3u)) return FEM_ERR_INVALID_ARG;
  if ((m != 16 && m != 32 && m != 64) || d > 155) return FEM_ERR_UNSUPPORTED;
  if (static_cast<long long>(B) * H > 2147483647ll || static_cast<long long>(B) * H * T * (d > m ? d : m) >= (1ll << 40))
    return FEM_ERR_UNSUPPORTED;
  DeviceState *ds = nullptr;
  int rc = device_state(&ds);
  if (rc != FEM_OK) return rc;
  if ((rc = debug_check_beta(beta, static_cast<long long>(H) * d, ds, static_cast<cudaStream_t>(stream))) != FEM_OK)
    return rc;
  const size_t bytes = gla_workspace_bytes(B * H, T, m, d, ds->num_sms, nullptr, nullptr);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  void *ws = nullptr;
  cudaError_t e = ws_alloc(ds, &ws, bytes, s);
  if (e != cudaSuccess) return map_cuda(e);
  rc = map_cuda(launch_gla(qf, kf, v, logdecay, beta, out, logz, B * H, H, T, m, d, ws, ds->num_sms, s));
  e = cudaFreeAsync(ws, s);
  if (rc != FEM_OK) return rc;
  return map_cuda(e);
}

int fem_decode(const void *q, const void *k, const void *v, const float *beta, float *out, float *lse, int B, int H,
               int T, int d, void *stream) {
  if (!q || !k || !v || !beta || !out) return FEM_ERR_INVALID_ARG;
  if (B <= 0 || H <= 0 || T <= 0 || d <= 0) return FEM_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out)) return FEM_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(beta) & 3u) || (lse && (reinterpret_cast<uintptr_t>(lse) & 3u)))
    return FEM_ERR_INVALID_ARG;
  if (d != 64 && d != 128) return FEM_ERR_UNSUPPORTED;
  if (static_cast<long long>(B) * H > 65535 || static_cast<long long>(B) * H * T >= (1ll << 31))
    return FEM_ERR_UNSUPPORTED;
  DeviceState *ds = nullptr;
  int rc = device_state(&ds);
  if (rc != FEM_OK) return rc;
  if ((rc = debug_check_beta(beta, static_cast<long long>(H) * d, ds, static_cast<cudaStream_t>(stream))) != FEM_OK)
    return rc;
  const int BH = B * H;
  const size_t bytes = decode_workspace_bytes(BH, T, d, ds->num_sms);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  void *ws = nullptr;
  cudaError_t e = ws_alloc(ds, &ws, bytes, s);
  if (e != cudaSuccess) return map_cuda(e);
  CUtensorMap tk;
  if ((rc = make_map(&tk, k, BH, T, d, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, kDecodeKeysPerCta)) != FEM_OK) {
    cudaFreeAsync(ws, s);
    return rc;
  }
  rc = map_cuda(launch_decode(tk, q, v, beta, out, lse, BH, H, T, d, static_cast<float *>(ws), ds->err, s));
  e = cudaFreeAsync(ws, s);
  if (rc != FEM_OK) return rc;
  return map_cuda(e);
}

int fem_fwd_f32(const float *q, const float *k, const float *v, const float *beta, float *out, float *lse, int B,
                int H, int T, int d, int causal, void *stream) {
  int rc = check_common(q, k, v, beta, out, lse, B, H, T, d, causal);
  if (rc != FEM_OK) return rc;
  if (d > 256) return FEM_ERR_UNSUPPORTED;
  DeviceState *ds = nullptr;
  if ((rc = device_state(&ds)) != FEM_OK) return rc;
  if ((rc = debug_check_beta(beta, static_cast<long long>(H) * d, ds, static_cast<cudaStream_t>(stream))) != FEM_OK)
    return rc;
  return map_cuda(launch_f32(q, k, v, beta, out, lse, B, H, T, d, causal, static_cast<cudaStream_t>(stream)));
}

int fem_fwd_host(const void *q, const void *k, const void *v, const float *beta, float *out, float *lse, int B,
                 int H, int T, int d, int causal, void *stream) {
  if (!q || !k || !v || !beta || !out) return FEM_ERR_INVALID_ARG;
  if (B <= 0 || H <= 0 || T <= 0 || d <= 0 || (causal != 0 && causal != 1)) return FEM_ERR_INVALID_ARG;
  if (check_read_sizes(T, d) != FEM_OK) return FEM_ERR_UNSUPPORTED;
  if (debug_check_beta_host(beta, static_cast<long long>(H) * d) != FEM_OK) return FEM_ERR_INVALID_ARG;
  DeviceState *ds = nullptr;
  int rc = device_state(&ds);
  if (rc != FEM_OK) return rc;
  {
    std::lock_guard<std::mutex> lock(g_mutex);
    if (!ds->copy_in && cudaStreamCreateWithFlags(&ds->copy_in, cudaStreamNonBlocking) != cudaSuccess)
      return FEM_ERR_CUDA;
    if (!ds->copy_out && cudaStreamCreateWithFlags(&ds->copy_out, cudaStreamNonBlocking) != cudaSuccess)
      return FEM_ERR_CUDA;
  }
  // chunks of heads whose copies in, reads and copies out overlap (fem_chunks.h)
  const int hc = host_chunk_heads(B, H);  // heads per chunk, at most
  const std::vector<HostChunk> chunks = host_chunks(B, H);
  const int n_chunks = static_cast<int>(chunks.size());
  const size_t n = static_cast<size_t>(B) * H * T * d;
  const size_t rows = static_cast<size_t>(B) * H * T;
  const size_t in_b = round256(n * 2), beta_b = round256(static_cast<size_t>(H) * d * 4), out_b = round256(n * 4),
               lse_b = round256(rows * 4), ws_b = round256(fem_fwd_workspace_bytes(1, hc, T, d, causal));
  const size_t total = 3 * in_b + beta_b + out_b + lse_b + ws_b;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint8_t *buf = nullptr;
  cudaError_t e = ws_alloc(ds, reinterpret_cast<void **>(&buf), total, s);
  if (e != cudaSuccess) return map_cuda(e);
  uint8_t *dq = buf, *dk = dq + in_b, *dv = dk + in_b, *db = dv + in_b, *dout = db + beta_b, *dlse = dout + out_b,
          *dws = dlse + lse_b;
  std::vector<cudaEvent_t> ev(2 * n_chunks + 2, nullptr);
  for (auto &x : ev)
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&x, cudaEventDisableTiming);
  // the copy streams start after the allocation, in the caller's stream order
  if (e == cudaSuccess) e = cudaEventRecord(ev[2 * n_chunks], s);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(ds->copy_in, ev[2 * n_chunks], 0);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(ds->copy_out, ev[2 * n_chunks], 0);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(db, beta, static_cast<size_t>(H) * d * 4, cudaMemcpyHostToDevice, ds->copy_in);
  rc = map_cuda(e);
  for (int c = 0; c < n_chunks && rc == FEM_OK; ++c) {
    const int b = chunks[c].b, h0 = chunks[c].h0, nh = chunks[c].nh;
    const size_t e0 = (static_cast<size_t>(b) * H + h0) * T * d, ne = static_cast<size_t>(nh) * T * d;
    const size_t r0 = (static_cast<size_t>(b) * H + h0) * T, nr = static_cast<size_t>(nh) * T;
    const uint8_t *hq = static_cast<const uint8_t *>(q), *hk = static_cast<const uint8_t *>(k),
                  *hv = static_cast<const uint8_t *>(v);
    e = cudaMemcpyAsync(dq + e0 * 2, hq + e0 * 2, ne * 2, cudaMemcpyHostToDevice, ds->copy_in);
    if (e == cudaSuccess) e = cudaMemcpyAsync(dk + e0 * 2, hk + e0 * 2, ne * 2, cudaMemcpyHostToDevice, ds->copy_in);
    if (e == cudaSuccess) e = cudaMemcpyAsync(dv + e0 * 2, hv + e0 * 2, ne * 2, cudaMemcpyHostToDevice, ds->copy_in);
    if (e == cudaSuccess) e = cudaEventRecord(ev[2 * c], ds->copy_in);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s, ev[2 * c], 0);
    rc = map_cuda(e);
    if (rc == FEM_OK)
      rc = fem_fwd_ws(dq + e0 * 2, dk + e0 * 2, dv + e0 * 2, reinterpret_cast<const float *>(db) + h0 * d,
                      reinterpret_cast<float *>(dout) + e0, lse ? reinterpret_cast<float *>(dlse) + r0 : nullptr, 1,
                      nh, T, d, causal, dws, ws_b, stream);
    if (rc != FEM_OK) break;
    e = cudaEventRecord(ev[2 * c + 1], s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(ds->copy_out, ev[2 * c + 1], 0);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(out + e0, reinterpret_cast<float *>(dout) + e0, ne * 4, cudaMemcpyDeviceToHost,
                          ds->copy_out);
    if (e == cudaSuccess && lse)
      e = cudaMemcpyAsync(lse + r0, reinterpret_cast<float *>(dlse) + r0, nr * 4, cudaMemcpyDeviceToHost,
                          ds->copy_out);
    rc = map_cuda(e);
  }
  // the caller's stream frees the buffers once every copy out has landed
  cudaError_t ej = cudaEventRecord(ev[2 * n_chunks + 1], ds->copy_out);
  if (ej == cudaSuccess) ej = cudaStreamWaitEvent(s, ev[2 * n_chunks + 1], 0);
  cudaError_t ef = cudaFreeAsync(buf, s);
  cudaError_t es = cudaStreamSynchronize(s);
  for (auto &x : ev)
    if (x) cudaEventDestroy(x);
  if (rc != FEM_OK) return rc;
  if (ej != cudaSuccess) return map_cuda(ej);
  if (ef != cudaSuccess) return map_cuda(ef);
  return map_cuda(es);
}

int fem_fwd_noalloc(const void *q, const void *k, const void *v, const float *beta, float *out, float *lse, int B,
                    int H, int T, int d, int causal, void *stream) {
  int rc = check_common(q, k, v, beta, out, lse, B, H, T, d, causal);
  if (rc != FEM_OK) return rc;
  if ((rc = check_read_sizes(T, d)) != FEM_OK) return rc;
  const size_t need = fem_fwd_workspace_bytes(B, H, T, d, causal);
  if (need == 0 || need > kStaticScratchBytes) return FEM_ERR_NO_MEMORY;
  void *scratch = nullptr;
  if ((rc = static_scratch(&scratch)) != FEM_OK) return rc;
  return fem_fwd_ws(q, k, v, beta, out, lse, B, H, T, d, causal, scratch, kStaticScratchBytes, stream);
}

int fem_set_kernel_events(void *start, void *stop) {
  if (start && stop) {
    t_ev_start = static_cast<cudaEvent_t>(start);
    t_ev_stop = static_cast<cudaEvent_t>(stop);
  } else {
    t_ev_start = t_ev_stop = nullptr;
  }
  return FEM_OK;
}

int fem_attn_fwd(const void *q, const void *k, const void *v, float *out, float *lse, int B, int H, int T, int d,
                 int causal, void *stream) {
  int rc = check_common(q, k, v, out, out, lse, B, H, T, d, causal);  // out stands in for beta (unused)
  if (rc != FEM_OK) return rc;
  if ((rc = check_tc_sizes(T, d)) != FEM_OK) return rc;
  DeviceState *ds = nullptr;
  if ((rc = device_state(&ds)) != FEM_OK) return rc;
  const int BH = B * H;
  CUtensorMap tq, tk, tv;
  if ((rc = make_map(&tq, q, BH, T, d)) != FEM_OK) return rc;
  if ((rc = make_map(&tk, k, BH, T, d)) != FEM_OK) return rc;
  if ((rc = make_map(&tv, v, BH, T, d)) != FEM_OK) return rc;
  const cudaEvent_t ev0 = t_ev_start, ev1 = t_ev_stop;
  t_ev_start = t_ev_stop = nullptr;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = ev0 ? cudaEventRecord(ev0, s) : cudaSuccess;
  if (e == cudaSuccess) e = launch_attn(d, tq, tk, tv, out, lse, BH, H, T, causal, ds->err, s);
  if (e == cudaSuccess && ev1) e = cudaEventRecord(ev1, s);
  return map_cuda(e);
}

int fem_probe_wait_timeout(unsigned limit_us, void *stream) {
  if (limit_us == 0 || limit_us > 1000000u) return FEM_ERR_INVALID_ARG;
  DeviceState *ds = nullptr;
  int rc = device_state(&ds);
  if (rc != FEM_OK) return rc;
  wait_probe_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(ds->err, 1000ull * limit_us);
  return map_cuda(cudaGetLastError());
}

int fem_check_device_error(void *stream) {
  DeviceState *ds = nullptr;
  int rc = device_state(&ds);
  if (rc != FEM_OK) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) return FEM_ERR_CUDA;
  unsigned word = 0;
  if (cudaMemcpy(&word, ds->err, sizeof(word), cudaMemcpyDeviceToHost) != cudaSuccess) return FEM_ERR_CUDA;
  if (word) {
    const unsigned zero = 0;
    if (cudaMemcpy(ds->err, &zero, sizeof(zero), cudaMemcpyHostToDevice) != cudaSuccess) return FEM_ERR_CUDA;
    return FEM_ERR_TIMEOUT;
  }
  return FEM_OK;
}

int fem_last_fixup_rows(void *stream) {
  DeviceState *ds = nullptr;
  if (device_state(&ds) != FEM_OK) return -1;
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return -1;
  int n = 0;
  if (cudaMemcpy(&n, ds->last_fixup, sizeof(n), cudaMemcpyDeviceToHost) != cudaSuccess) return -1;
  return n;
}

}  // extern "C"
