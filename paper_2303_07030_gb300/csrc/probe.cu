// probe.cu -- measurement aid: the FP32 FMA throughput of the device.
//
// The loss kernels of matrix factorisation, CP and the graph's H^T G are
// bound by FP32 arithmetic or by L2 gathers rather than by HBM; their
// fraction of peak needs a measured FP32 FMA rate, taken in the same run.
// Each thread runs kChains independent FMA chains (enough to cover the FMA
// pipe's latency), `iters` steps long; the result is stored so the compiler
// keeps the work.
#include <cuda_runtime.h>

#include "internal.h"
#include "sdad.h"

namespace sdad {

constexpr int kChains = 16;

__global__ void __launch_bounds__(256) fma_probe_kernel(float* __restrict__ out, int iters,
                                                        float a, float b) {
  float x[kChains];
#pragma unroll
  for (int c = 0; c < kChains; ++c) x[c] = (float)(threadIdx.x + c);
  for (int it = 0; it < iters; ++it) {
#pragma unroll
    for (int c = 0; c < kChains; ++c) x[c] = fmaf(x[c], a, b);
  }
  float s = 0.f;
#pragma unroll
  for (int c = 0; c < kChains; ++c) s += x[c];
  out[blockIdx.x * blockDim.x + threadIdx.x] = s;
}

}  // namespace sdad

using namespace sdad;

extern "C" sdad_status sdad_probe_fma(float* out, int32_t blocks, int32_t iters, double* flops,
                                      void* stream) {
  if (!out || !flops) return SDAD_ERR_NULL;
  if (blocks <= 0 || iters <= 0) return SDAD_ERR_SHAPE;
  sdad_status s = check_device();
  if (s) return s;
  // a = 1 - 2^-20, b = 2^-20: the chains stay bounded and never denormal
  const float a = 1.f - 9.5367431640625e-7f, b = 9.5367431640625e-7f;
  fma_probe_kernel<<<blocks, 256, 0, (cudaStream_t)stream>>>(out, iters, a, b);
  *flops = 2.0 * kChains * (double)iters * 256.0 * (double)blocks;
  return map_cuda(cudaGetLastError());
}
