// Host-side launchers of the FEM read kernels (internal to libfem.so).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include "fem_common.cuh"

namespace fem {

// Launches kernel<<<grid, block, smem, stream>>>(args...), with `pdl` as a
// programmatic dependent launch on the previous kernel of the stream (the
// kernel then orders itself behind it with grid_dep_wait()).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                                 bool pdl, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// Device workspace of one read (all arrays caller-owned): the value-bank
// pre-pass's arrays and the exact fix-up's entry list.
struct BankWorkspace {
  float4 *tstat;            // [B*H, key tiles, d]: max, min, sum of v per tile
  ChanInfo *chan;           // [B*H, d]
  float4 *bcoef;            // [B*H, key tiles, d]: the bank's coefficients for the tile (BankCoef)
  float *shift;             // [B*H, key tiles, d]: the bank's shift for each tile
  float *rfac;              // [B*H, key tiles, d]: exp(beta (shift[kt-1] - shift[kt])), 1 if unmoved
  unsigned *colmask;        // [B*H, key tiles, 4]: bit j set when channel j's shift moved at the tile
  float *colsum;            // [B*H, key tiles, d]: sum of |bank| over the tile's keys
  __half *bank;             // [B*H, T, d]: the value bank, fp16
  FixupEntry *fixups;       // exact-recompute list, written by the tensor-core kernel
  int *fixup_count;         // its length in slots, a multiple of 8 (zeroed before the pre-pass)
  int *fixup_rows;          // rows listed (zeroed before the pre-pass)
  int *fixup_next;          // the fix-up's next unclaimed chunk (zeroed before the pre-pass)
  int *fix_long;            // chunks registered for splitting (zeroed before the pre-pass)
  FixSlot *fix_slots;       // [kFixPoolSlots] (zeroed before the pre-pass)
  float *fix_part;          // [kFixPoolSlots, fix_max_segs, kFixChunk, 2 + 4 d] partial states; null: no split
};

// Capacity of the fix-up list in entries: every row, plus the padding of each
// query tile's two blocks of entries to multiples of kFixChunk.
inline size_t fixup_capacity(size_t BH, size_t T) {
  const size_t n_qt = (T + kBlockQ - 1) / kBlockQ;
  return BH * n_qt * (kBlockQ + 2 * (kFixChunk - 1));
}

// Statistics, plan and value bank (two reads of V, one write of the bank),
// and the bank's column sums per key tile.  `tv` and `te` map V (bf16) and the
// bank (fp16) like the tensor-core kernel's operands: boxes of 64 channels x
// 128 rows, 128-byte swizzle.
//
// BankCoef, one float4 per (b, h, key tile, channel), written by the plan:
//   linear bank   {1/beta (0 at beta = 0), beta, c_lin, NaN}
//   shifted bank  {beta log2 e, (kBankOffset - beta c) log2 e, c, 0}
// stats_ready: w.tstat already holds the tiles' statistics of this V (they do
// not depend on beta); skip recomputing them.
cudaError_t launch_value_bank(const void *v, const CUtensorMap &tv, const CUtensorMap &te, const float *beta, int BH,
                              int H, int T, int d, const BankWorkspace &w, unsigned *err, int num_sms,
                              cudaStream_t stream, bool stats_ready = false);

// Gates of the one-pass two-level gated read: o = g (mu + lambda (F - mu))
// with mu the mean read (its bank v - c_lin, anchors chan0, column sums
// colsum0) and F the read at beta_max.  lam, g: [B*H, T, d] fp32 inputs;
// mu_side: [B*H, T, d] fp32 scratch, written only at the fix-up entries
// (their mu, for the fix-up).
struct TcGate {
  const float *lam, *g;
  float *mu_side;
  const ChanInfo *chan0;
  const float *colsum0;
};

// Tensor-core read.  Returns cudaErrorInvalidValue for an unsupported d or
// size.  `out` is the fp32 output [B*H, T, d], 16-byte aligned.  Entries the
// underflow guard rejects are listed in w.fixups (w.fixup_count slots,
// w.fixup_rows rows) for the fix-up; for entries that restart from the state
// before their diagonal tile the kernel writes, in place of the listed
// channels' outputs, their accumulator before that tile.  With te0 (the mean's
// bank) and gate both given it runs the one-pass gated read; with neither the
// plain read.
// pdl: a programmatic dependent launch on the bank kernel before it.
cudaError_t launch_tc(int d, const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &te,
                      const CUtensorMap *te0, float *out, const float *beta, const BankWorkspace &w, float *lse,
                      int BH, int H, int T, int causal, const TcGate *gate, unsigned *err, cudaStream_t stream,
                      bool pdl = false);

// The attention-mode comparator on the same kernel: o = softmax(q k^T / sqrt(d)) v
// with bf16 P and V on the tensor cores (tv maps V like the bank).
cudaError_t launch_attn(int d, const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &tv, float *out,
                        float *lse, int BH, int H, int T, int causal, unsigned *err, cudaStream_t stream);

// Largest sequence length launch_tc takes (its shared-memory bitmap of moved key tiles).
constexpr int kMaxSeqLen = 8192 * kBlockK;

// Recomputes the listed (row, channel) outputs exactly in fp32, from the
// entry's kt0 on (see FixupEntry), for the read at beta with channel modes
// `chan` and shifts `shift` (those of the bank the tensor-core kernel used).
// gate: nullptr, or the one-pass gated read's gates (an entry restarting
// from its diagonal tile is then gated with the mu the tensor-core kernel
// left in gate->mu_side; a full recomputation computes mu as well).
// next_chunk: a zeroed counter from which the blocks claim chunks of entries.
cudaError_t launch_fixup(const void *q, const void *k, const void *v, const float *beta, const ChanInfo *chan,
                         const float *shift, float *out, int H, int T, int d, int causal, const FixupEntry *entries,
                         const int *count, const int *rows, int *next_chunk, int *last_rows, const TcGate *gate,
                         int *fix_long, FixSlot *fix_slots, float *fix_part, int num_sms, cudaStream_t stream,
                         bool pdl = false);


// Decode read of one query per (b, h) against T cached keys: per-CTA key-chunk
// partials into `part` (decode_workspace_bytes), then their log-add-exp merge.
// tk maps K as [BH, T, d] bf16 in boxes of kDecodeKeysPerCta rows x 64
// channels with the 128-byte swizzle.
constexpr int kDecodeKeysPerCta = 64;
size_t decode_workspace_bytes(int BH, int T, int d, int num_sms);
cudaError_t launch_decode(const CUtensorMap &tk, const void *q, const void *v, const float *beta, float *out,
                          float *lse, int BH, int H, int T, int d, float *part, unsigned *err, cudaStream_t stream);

// FEM read over a GLA prior (fp32, segmented recurrent scan); m in {16, 32, 64},
// d <= 155; `ws` holds gla_workspace_bytes() bytes (segment states).
size_t gla_workspace_bytes(int BH, int T, int m, int d, int num_sms, int *seg_len, int *n_seg);
cudaError_t launch_gla(const float *qf, const float *kf, const float *v, const float *logdecay, const float *beta,
                       float *out, float *logz, int BH, int H, int T, int m, int d, void *ws, int num_sms,
                       cudaStream_t stream);

// The GLA-prior read chunked on the tensor cores (m = d = 64), one CTA per (b, h).
cudaError_t launch_gla_tc(const float *qf, const float *kf, const float *v, const float *logdecay, const float *beta,
                          float *out, float *logz, int B, int H, int T, unsigned *err, cudaStream_t stream);

// Time-decay conditioner convolution h_t = exp(-s_t) h_{t-1} + u_t over [B, T, Hc]
// (segmented scan: one launch of 8-CTA clusters up to T = 16384, no workspace, then
// tdc_workspace_bytes() is 0; three launches beyond); `ws` holds tdc_workspace_bytes() bytes.
size_t tdc_workspace_bytes(int B, int T, int Hc);
cudaError_t launch_tdc(const float *s, const float *u, float *h, int B, int T, int Hc, void *ws, cudaStream_t stream);

// Backward of the fp32 read (dq, dk, dv, and dbeta summed over batch and time).
cudaError_t launch_bwd_f32(const float *q, const float *k, const float *v, const float *beta, const float *out,
                           const float *lse, const float *dout, float *dq, float *dk, float *dv, float *dbeta, int B,
                           int H, int T, int d, int causal, cudaStream_t stream);

// fp32-input read on CUDA cores.
cudaError_t launch_f32(const float *q, const float *k, const float *v, const float *beta, float *out, float *lse,
                       int B, int H, int T, int d, int causal, cudaStream_t stream);
// bf16 inputs of head dimension 16 or 32 on the same CUDA-core kernel (fp32 arithmetic).
cudaError_t launch_simt_bf16(const void *q, const void *k, const void *v, const float *beta, float *out, float *lse,
                             int B, int H, int T, int d, int causal, cudaStream_t stream);

}  // namespace fem
