// fma_probe.cu — FP32 fused multiply-add rate of the GPU, the denominator of the FP32
// roofline fractions that the benchmark reports for the ALU-bound kernels.  Not part of
// the method: every thread runs kChains independent FMA chains (enough independent work
// to keep each SM sub-partition's FMA pipe busy) and stores their sum so nothing is
// eliminated.
#include <cstdint>

#include "kernels.h"

namespace simx {

constexpr int kProbeChains = 16;
constexpr int kProbeThreads = 256;
constexpr int kProbeBlocksPerSM = 4;

__global__ void __launch_bounds__(kProbeThreads) k_fma_probe(int64_t iters, float* __restrict__ sink) {
  float a[kProbeChains];
  const float x = 1.0f + 1e-7f * (float)threadIdx.x, y = 0.999999f;
#pragma unroll
  for (int c = 0; c < kProbeChains; ++c) a[c] = (float)(c + blockIdx.x);
  for (int64_t i = 0; i < iters; ++i) {
#pragma unroll
    for (int c = 0; c < kProbeChains; ++c) a[c] = __fmaf_rn(a[c], y, x);
  }
  float s = 0.0f;
#pragma unroll
  for (int c = 0; c < kProbeChains; ++c) s += a[c];
  sink[(size_t)blockIdx.x * blockDim.x + threadIdx.x] = s;
}

int fma_probe_blocks() {
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return sms * kProbeBlocksPerSM;
}

cudaError_t launch_fma_probe(int64_t iters, float* sink, double* flops, cudaStream_t s) {
  const int blocks = fma_probe_blocks();
  k_fma_probe<<<blocks, kProbeThreads, 0, s>>>(iters, sink);
  count_launches(1);
  *flops = 2.0 * kProbeChains * (double)iters * blocks * kProbeThreads;
  return cudaGetLastError();
}

size_t fma_probe_sink_floats() { return (size_t)fma_probe_blocks() * kProbeThreads; }

}  // namespace simx
