// Outer and inner gates of the two-level gated read (Sec. 3, "Two-Level
// Gated FEM", Eqs. "inner-gate-main" and "fem-two-gates-main"):
//
//   out = g (x) ((1 - lambda) (x) mu + lambda (x) Fmax)
//
// elementwise over [B, H, T, d], with mu the beta = 0 read and Fmax the read
// at beta_max.  HBM-bound: 16 bytes read and 4 written per element, float4
// loads and stores over a grid sized to the SM count.
#include "fem_common.cuh"
#include "fem_launch.h"

namespace fem {

__global__ void __launch_bounds__(256) gate_kernel(const float4 *__restrict__ mu, const float4 *__restrict__ lam,
                                                   const float4 *__restrict__ g, float4 *__restrict__ out,
                                                   size_t n4) {
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n4;
       i += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const float4 m = mu[i], l = lam[i], s = g[i], f = out[i];
    // (1 - l) m + l f = m + l (f - m)
    out[i] = make_float4(s.x * fmaf(l.x, f.x - m.x, m.x), s.y * fmaf(l.y, f.y - m.y, m.y),
                         s.z * fmaf(l.z, f.z - m.z, m.z), s.w * fmaf(l.w, f.w - m.w, m.w));
  }
}

cudaError_t launch_gate(const float *mu, const float *lam, const float *g, float *out, size_t n, int num_sms,
                        cudaStream_t stream) {
  if (n % 4) return cudaErrorInvalidValue;
  const size_t n4 = n / 4;
  const size_t want = (n4 + 255) / 256;
  const int grid = static_cast<int>(want < static_cast<size_t>(num_sms) * 8 ? want : static_cast<size_t>(num_sms) * 8);
  if (grid == 0) return cudaSuccess;
  gate_kernel<<<grid, 256, 0, stream>>>(reinterpret_cast<const float4 *>(mu), reinterpret_cast<const float4 *>(lam),
                                        reinterpret_cast<const float4 *>(g), reinterpret_cast<float4 *>(out), n4);
  return cudaGetLastError();
}

}  // namespace fem
