/*
 * fem.h -- C ABI of libfem.so: the forward free-energy read of the Free
 * Energy Mixer (arXiv 2602.07160) with a softmax prior, on sm_103a GPUs.
 *
 * The read (Sec. 2.3, Eq. "fem-free-energy-main"; softmax prior of App. C,
 * Eq. "softmax-prior"; masked scaled scores of Sec. 1):
 *
 *   s_{t,i} = q_t . k_i / sqrt(d),  i in M_t = {0..t} (causal) or {0..T-1}
 *   o_{t,j} = (1/beta_j) ( LSE_i(s_{t,i} + beta_j v_{i,j}) - LSE_i s_{t,i} )
 *           = (1/beta_j) log sum_{i in M_t} softmax(s_t)_i exp(beta_j v_{i,j})
 *   lse_t   = LSE_i s_{t,i}   (natural log; LSE_i(s + beta v) = lse + beta o)
 *
 * beta_j = 0 is the continuous beta -> 0 limit, the prior mean
 * sum_i p_t(i) v_{i,j} (Prop. "app-baseline").  beta_j < 0 is outside the
 * method and a precondition violation: device memory is not inspected unless
 * the environment variable FEM_DEBUG is set (to anything but "0") when the
 * library first checks it.  Then every entry point that takes beta checks it
 * first (one small kernel and a synchronisation of `stream`) and returns
 * FEM_ERR_INVALID_ARG, with nothing of the computation enqueued, when an entry
 * is negative, NaN or infinite.  Debug mode is not for stream capture.
 *
 * Conventions for every entry point:
 *  - Layout: q, k, v are [B, H, T, d] contiguous, d fastest; beta is [H, d]
 *    float32 (per head, per channel, shared over batch and time); out is
 *    [B, H, T, d] float32; lse is [B, H, T] float32 or NULL.
 *  - Ownership: the caller owns every buffer.  Device pointers must be
 *    16-byte aligned.  The library keeps no pointer after a call returns.
 *  - Streams: `stream` is a cudaStream_t (NULL = legacy default stream).
 *    Device work is enqueued asynchronously on it; outputs are valid once the
 *    stream reaches the end of the call's work.
 *  - Errors: argument errors are reported synchronously and nothing is
 *    enqueued.  A CUDA launch or allocation failure returns FEM_ERR_CUDA or
 *    FEM_ERR_NO_MEMORY.  A kernel that gives up on a bounded wait records
 *    the fact in a per-device error word and exits cleanly; read it with
 *    fem_check_device_error().  No exception crosses the ABI.
 *  - Threads: entry points may be called from several host threads; calls
 *    share only the per-device error word and fix-up counter.
 */
#ifndef FEM_H
#define FEM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    FEM_OK = 0,
    FEM_ERR_INVALID_ARG = 1,  /* null pointer, non-positive size, misalignment */
    FEM_ERR_UNSUPPORTED = 2,  /* a head dimension the path does not implement */
    FEM_ERR_CUDA = 3,         /* a CUDA runtime/driver call failed */
    FEM_ERR_TIMEOUT = 4,      /* a kernel gave up on a bounded wait */
    FEM_ERR_NO_MEMORY = 5     /* workspace allocation failed / too small */
} fem_status;

/*
 * fem_fwd -- the read for bf16 inputs (the tensor-core path).
 *   q, k, v : device, bf16 [B, H, T, d]
 *   beta    : device, float32 [H, d], beta >= 0
 *   out     : device, float32 [B, H, T, d]
 *   lse     : device, float32 [B, H, T], or NULL
 *   B, H, T : >= 1;  d in {16, 32, 64, 128};  causal: 0 (full prior) or 1
 * d = 64 and 128 run on the tensor cores as below.  d = 16 and 32, too narrow
 * for 64-channel tiles to pay, run on CUDA cores (fem_fwd_f32's kernel reading
 * bf16): every product and sum in fp32, no workspace beyond 256 bytes, no
 * fix-up rows.  Any other d is FEM_ERR_UNSUPPORTED.
 * Allocates its workspace stream-ordered on `stream` from a memory pool the
 * library keeps per device (freed memory stays in the pool for the next
 * call; the entry points that allocate all use it).  Accuracy: the score contraction takes bf16 q, k; the second
 * contraction takes the prior weights and the per-channel value bank in fp16
 * (11-bit significand); both accumulate in fp32.  Every output whose 16-bit
 * operands could have lost more than 2^-7 to underflow is recomputed
 * exactly in fp32, so the result holds for any prior (peaked or flat).
 */
int fem_fwd(const void *q, const void *k, const void *v, const float *beta,
            float *out, float *lse, int B, int H, int T, int d, int causal,
            void *stream);

/*
 * fem_fwd_workspace_bytes -- bytes of device workspace fem_fwd_ws needs for
 * these sizes (0 on invalid sizes).
 */
size_t fem_fwd_workspace_bytes(int B, int H, int T, int d, int causal);

/*
 * fem_fwd_ws -- fem_fwd with a caller-owned device workspace of at least
 * fem_fwd_workspace_bytes() bytes, 256-byte aligned.  Performs no allocation.
 * The workspace must not be used by another call that overlaps on the GPU.
 */
int fem_fwd_ws(const void *q, const void *k, const void *v, const float *beta,
               float *out, float *lse, int B, int H, int T, int d, int causal,
               void *workspace, size_t workspace_bytes, void *stream);

/*
 * fem_fwd_f32 -- the read for float32 inputs on CUDA cores (exact fp32
 * arithmetic with a per-row, per-channel shift).  Same layout and rules as
 * fem_fwd with q, k, v float32; 1 <= d <= 256.  No workspace.
 */
int fem_fwd_f32(const float *q, const float *k, const float *v,
                const float *beta, float *out, float *lse, int B, int H, int T,
                int d, int causal, void *stream);

/*
 * fem_fwd_host -- fem_fwd on HOST buffers: copies q, k, v, beta to the
 * device, runs the read and copies out (and lse, if non-NULL) back, then
 * synchronises `stream`.  The work is split into chunks of consecutive heads
 * (about eight in all): the copies in of one chunk, the read of the previous
 * one (on `stream`) and the copies out of the one before overlap, on two copy
 * streams the library creates once per device.  Host buffers should be pinned
 * for full copy bandwidth.  Device buffers come stream-ordered from the
 * library's pool and are freed before return.  Returns after the results are
 * in host memory; fem_last_fixup_rows then reports the last chunk's count.
 */
int fem_fwd_host(const void *q, const void *k, const void *v, const float *beta,
                 float *out, float *lse, int B, int H, int T, int d, int causal,
                 void *stream);

/*
 * fem_fwd_noalloc -- fem_fwd for callers that may not allocate device memory
 * during the call (for example a plugin whose execute callback is not
 * allowed to allocate, or a service that reserves all device memory up
 * front).  The paper has no counterpart; this is an interface convenience.
 * Same arguments, layout and results as fem_fwd; the caller still passes
 * every input and output.  Instead of a stream-ordered allocation it uses a fixed
 * 16 MiB scratch array compiled into the library, which every GPU that
 * loads the library holds until the process exits.  Problems needing more
 * workspace than that (fem_fwd_workspace_bytes() > 16 MiB, about 2*d + 80
 * bytes per row (b, h, t)) return FEM_ERR_NO_MEMORY before anything is
 * enqueued.  It calls no allocation routine and creates no memory pool.  The
 * first call on a device looks up the scratch address and the library's
 * per-device error word on that device (cudaGetSymbolAddress), so make that
 * first call outside any stream capture.  All calls share the one array and
 * it keeps the previous call's contents (the call clears what must start at
 * zero): calls that overlap on the GPU, from any stream or thread, race and
 * must be serialised by the caller.
 */
int fem_fwd_noalloc(const void *q, const void *k, const void *v,
                    const float *beta, float *out, float *lse, int B, int H,
                    int T, int d, int causal, void *stream);

/*
 * fem_fwd_gated -- the two-level gated read (Sec. 3, "Two-Level Gated FEM":
 * inner gate by linearised temperature learning, Eq. "inner-gate-main", and
 * outer gate, Eq. "fem-two-gates-main"):
 *
 *   mu_{t,j}   = sum_{i in M_t} p_t(i) v_{i,j}                   (the beta = 0 read)
 *   Fmax_{t,j} = (1/bmax_j) log sum_{i in M_t} p_t(i) exp(bmax_j v_{i,j})
 *   out_{t,j}  = g_{t,j} ((1 - lambda_{t,j}) mu_{t,j} + lambda_{t,j} Fmax_{t,j})
 *
 *   q, k, v   : device, bf16 [B, H, T, d]
 *   beta_max  : device, float32 [H, d], > 0 (the global maximum inverse temperature)
 *   lam, gate : device, float32 [B, H, T, d]: the inner gate lambda in [0, 1]
 *               and the outer gate g (> 0), already activated by the caller
 *   out, lse  : as fem_fwd; lse does not depend on the gates
 *   d in {64, 128}
 * One tensor-core pass (the one-pass form of App. "One-pass implementation"):
 * the same prior weights mix two value banks, the mean's and beta_max's,
 * into two accumulators, and the epilogue applies the gates.  Allocates its
 * workspace stream-ordered on `stream`: fem_fwd's workspace twice (one per
 * bank) and 4 B*H*T*d bytes written only at the fix-up's entries.
 * Errors as fem_fwd; a null or misaligned lam or gate is
 * FEM_ERR_INVALID_ARG.
 */
int fem_fwd_gated(const void *q, const void *k, const void *v, const float *beta_max,
                  const float *lam, const float *gate, float *out, float *lse, int B,
                  int H, int T, int d, int causal, void *stream);

/*
 * fem_decode -- the decode read: one new query per (b, h) against a cache of
 * T keys and values that already holds the query's own key and value (the
 * last row of a causal read; Sec. 2.3 read with the softmax prior of App. C):
 *
 *   s_i = q . k_i / sqrt(d),  o_j = (1/beta_j) log sum_i softmax(s)_i exp(beta_j v_{i,j}),
 *   lse = LSE_i s_i,  i = 0 .. T-1
 *
 *   q        : device, bf16 [B, H, d]
 *   k, v     : device, bf16 [B, H, T, d] (the cache)
 *   beta     : device, float32 [H, d], beta >= 0 (0 = the prior mean)
 *   out      : device, float32 [B, H, d];  lse: device, float32 [B, H] or NULL
 *   d in {64, 128}
 * Each CTA reads a chunk of 64 keys; the chunks' partials are merged with
 * log-add-exp in two levels, all in fp32 arithmetic.  Allocates a small
 * workspace (3d + 2 floats per chunk) stream-ordered on `stream`.
 */
int fem_decode(const void *q, const void *k, const void *v, const float *beta, float *out,
               float *lse, int B, int H, int T, int d, void *stream);

/*
 * fem_gla_fwd -- the read over a gated-linear-attention prior (App. "Gated
 * Linear Attention (GLA) Prior", Eqs. "gla-score-appendix" and "gla-assoc"):
 *
 *   s_t(i) = K_{t,i} <qf_t, kf_i> (i <= t),  K_{t,i} = exp(g_{i+1} + ... + g_t),
 *   p_t = s_t / Z_t,  o_{t,j} = (1/beta_j) log sum_i p_t(i) exp(beta_j v_{i,j}),
 *   logz_t = log Z_t
 *
 *   qf, kf   : device, float32 [B, H, T, m], nonnegative (the caller's
 *              feature map, e.g. ReLU(RoPE(.)) + eps); m in {16, 32, 64}
 *   v        : device, float32 [B, H, T, d], 1 <= d <= 155
 *   logdecay : device, float32 [B, H, T], g_t <= 0
 *   beta     : device, float32 [H, d], beta >= 0 (0 = the prior mean)
 *   out      : device, float32 [B, H, T, d];  logz: device, float32 [B, H, T] or NULL
 * An O(T) recurrent scan in fp32 on CUDA cores, split into time segments
 * (segment end states, a combine over segments, then the outputs).  Allocates
 * its workspace (the segments' start states) stream-ordered on `stream`.
 */
int fem_gla_fwd(const float *qf, const float *kf, const float *v, const float *logdecay,
                const float *beta, float *out, float *logz, int B, int H, int T, int m, int d,
                void *stream);

/*
 * fem_gla_fwd_tc -- the same read (fem_gla_fwd's definition and arguments)
 * chunked on the tensor cores, for m = d = 64 (FEM_ERR_UNSUPPORTED
 * otherwise).  One CTA per (b, h) walks 128-step chunks: the decay-masked
 * qf kf^T of the chunk against the chunk's value bank, qf against the state
 * of the earlier chunks, and the state's update, as bf16 contractions with
 * fp32 accumulation (tcgen05); the state itself is kept in fp32.  Channels
 * with beta < 1/4 use the bank expm1(beta (v - c)) / beta anchored at the
 * smallest value so far, the others exp(beta v - lambda) with a log-scaled
 * state.  Accuracy is the bf16 read's for values of unit spread (max abs 2e-2,
 * mean abs 2e-3 against the float64 definition); per entry the bound is about
 * 2^-8 |v - c| (linear) or 2^-8 / beta (shifted), so it scales with the
 * values' spread.  Entries whose in-chunk part could be carried by terms
 * under fp32's range are recomputed exactly.  No workspace; qf, kf, v, out
 * 16-byte aligned.
 */
int fem_gla_fwd_tc(const float *qf, const float *kf, const float *v, const float *logdecay,
                   const float *beta, float *out, float *logz, int B, int H, int T, int m, int d,
                   void *stream);

/*
 * fem_tdc_conv -- the time-decay conditioner's convolution (App. "Low-rank
 * Convolution: Time-Decay Conditioner (TDC)", Eq. "tdc-conv", streaming form
 * of Prop. "tdc-lowrank"):
 *
 *   h_t = sum_{i<=t} exp(-(s_{i+1} + ... + s_t)) u_i = exp(-s_t) h_{t-1} + u_t
 *
 *   s, u : device, float32 [B, T, Hc]; s >= 0 (the softplus rates)
 *   h    : device, float32 [B, T, Hc]
 * A segmented scan in fp32 (segment end states, a combine over segments, then
 * the outputs).  Up to T = 16384 one launch of 8-CTA clusters that combine
 * through distributed shared memory and allocates nothing; beyond, three
 * launches with a workspace allocated stream-ordered on `stream`.
 */
int fem_tdc_conv(const float *s, const float *u, float *h, int B, int T, int Hc, void *stream);

/*
 * fem_bwd_f32 -- gradients of the fp32 read (fem_fwd_f32) from its saved
 * outputs, recomputing the scores:
 *
 *   dF/dv_{i,j}   = q_{t,i,j}, the posterior prop. to p_t(i) exp(beta_j v_{i,j})  (Prop. "app-geom")
 *   dF/ds_{t,i}   = (q_{t,i,j} - p_t(i)) / beta_j                            (Prop. "app-bounds" (iv))
 *   dF/dbeta_j    = KL(q || p) / beta_j^2                                     (Eq. "app-beta-deriv")
 *
 * chained through s = q k / sqrt(d).
 *   q, k, v, out, dout : device, float32 [B, H, T, d]; out the forward's output
 *   lse                : device, float32 [B, H, T], the forward's lse
 *   beta               : device, float32 [H, d]
 *   dq, dk, dv         : device, float32 [B, H, T, d]
 *   dbeta              : device, float32 [H, d], summed over batch and time
 *   1 <= d <= 256
 * fp32 on CUDA cores, O(T^2 d) like the forward; no workspace.
 */
int fem_bwd_f32(const float *q, const float *k, const float *v, const float *beta, const float *out,
                const float *lse, const float *dout, float *dq, float *dk, float *dv, float *dbeta,
                int B, int H, int T, int d, int causal, void *stream);

/*
 * fem_check_device_error -- synchronises `stream`, then returns FEM_OK, or
 * FEM_ERR_TIMEOUT if any kernel of this library on the current device gave up
 * on a bounded wait since the last check (the word is cleared), or
 * FEM_ERR_CUDA if the synchronisation failed.
 */
int fem_check_device_error(void *stream);

/*
 * fem_attn_fwd -- diagnostic comparator: plain softmax attention on the same
 * tensor-core kernel, o_t = sum_i softmax(s_t)_i v_i (the read's beta -> 0
 * limit, Prop. "app-baseline", and the prior mean of the two-level gated read,
 * Sec. 3), with V itself (bf16) in place of the value bank: no pre-pass, no
 * shifts, no underflow guard, P rounded to bf16 for the second contraction.
 * It measures the cost of the free-energy read over attention at the same
 * shapes.  Layout and rules as fem_fwd (no beta); lse as fem_fwd.  No
 * workspace.
 */
int fem_attn_fwd(const void *q, const void *k, const void *v, float *out, float *lse, int B,
                 int H, int T, int d, int causal, void *stream);

/*
 * fem_probe_wait_timeout -- diagnostic of the failure path; the paper has no
 * counterpart.  Enqueues on `stream` one kernel whose single thread waits,
 * with the same bounded-wait helper every kernel of the library uses, on a
 * shared-memory mbarrier that nothing completes.  After limit_us
 * microseconds (1 .. 1,000,000) the wait gives up, records the fact in the
 * per-device error word and the kernel returns; fem_check_device_error()
 * then reports FEM_ERR_TIMEOUT (and clears the word).  The kernel issues no
 * copy and no tensor-core operation, so the context stays usable.  A
 * limit_us of 0 or above 1,000,000 is FEM_ERR_INVALID_ARG.
 */
int fem_probe_wait_timeout(unsigned limit_us, void *stream);

/*
 * fem_last_fixup_rows -- synchronises `stream` and returns the number of rows
 * the last bf16 read on the current device recomputed exactly for some of
 * their channels: the entries whose 16-bit operands could have lost more
 * than 2^-7 of the output to underflow (peaked priors at large beta, and the
 * first rows of causal diagonal tiles whose value-bank shift includes keys
 * they do not see).  Diagnostic; -1 on error.
 */
int fem_last_fixup_rows(void *stream);

/*
 * fem_set_kernel_events -- diagnostic timing hook.  With both arguments
 * non-NULL (caller-owned cudaEvent_t handles), the next bf16 read issued by
 * the calling host thread records `start` on its stream immediately before
 * its tensor-core kernel and `stop` immediately after it, then forgets the
 * events.  Passing NULL clears a pending request.  Always FEM_OK.
 */
int fem_set_kernel_events(void *start, void *stop);

/* fem_status_str -- a static string naming a status code. */
const char *fem_status_str(int status);

#ifdef __cplusplus
}
#endif

#endif /* FEM_H */
