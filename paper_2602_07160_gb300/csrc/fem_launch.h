// Host-side launchers of the FEM read kernels (internal to libfem.so).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include "fem_common.cuh"

namespace fem {

// Value statistics, shift schedule and exact-recompute list (one read of V).
cudaError_t launch_value_stats(const void *v, const float *beta, int BH, int H, int T, int d, int causal,
                               ChanInfo *chan, float *cpre, FixupEntry *fixups, int *fixup_count,
                               cudaStream_t stream);

// Tensor-core read.  Returns cudaErrorInvalidValue for an unsupported d.
cudaError_t launch_tc(int d, const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &tv, const float *beta,
                      const ChanInfo *chan, const float *cpre, float *out, float *lse, int BH, int H, int T,
                      int causal, unsigned *err, cudaStream_t stream);

// Exact recompute of the listed (row, channel group) entries.
cudaError_t launch_fixup(const void *q, const void *k, const void *v, const float *beta, float *out, int H, int T,
                         int d, const FixupEntry *entries, const int *count, int *last_count, int num_sms,
                         cudaStream_t stream);

// fp32-input read on CUDA cores.
cudaError_t launch_f32(const float *q, const float *k, const float *v, const float *beta, float *out, float *lse,
                       int B, int H, int T, int d, int causal, cudaStream_t stream);

}  // namespace fem
