// Adam (Kingma & Ba 2015), the optimiser step of the policy-gradient training loop
// (Sec. 4.3), on a flat parameter vector.  One elementwise kernel; with gradient
// clipping a fixed-grid sum of squares (fp64 partials, reduced in a fixed order, so the
// scale is the same bits on every run) and a one-block finish run first.
#include "kernels.h"

namespace simx {

namespace {

constexpr int kAdamThreads = 256;
constexpr int kNormBlocks = 304;  // two per SM

__global__ void __launch_bounds__(kAdamThreads) k_sumsq(const float* __restrict__ g,
                                                        const uint8_t* __restrict__ mask,
                                                        int64_t n, double* part) {
  __shared__ double red[kAdamThreads];
  double acc = 0.0;
  for (int64_t i = (int64_t)blockIdx.x * kAdamThreads + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * kAdamThreads) {
    if (mask && !mask[i]) continue;
    const double x = (double)g[i];
    acc += x * x;
  }
  red[threadIdx.x] = acc;
  __syncthreads();
  for (int w = kAdamThreads / 2; w > 0; w /= 2) {
    if ((int)threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) part[blockIdx.x] = red[0];
}

// scale = min(1, max_norm / ||g||), 1 for a zero gradient.
__global__ void k_clip_scale(const double* part, int nb, float max_norm, float* scale) {
  if (threadIdx.x != 0) return;
  double s = 0.0;
  for (int b = 0; b < nb; ++b) s += part[b];
  const double norm = sqrt(s);
  *scale = (norm > (double)max_norm) ? (float)((double)max_norm / norm) : 1.0f;
}

__global__ void __launch_bounds__(kAdamThreads) k_adam(float* __restrict__ p,
                                                       const float* __restrict__ g,
                                                       float* __restrict__ m, float* __restrict__ v,
                                                       const uint8_t* __restrict__ mask, int64_t n,
                                                       const float* scale, float step_size,
                                                       float inv_sqrt_c2, float b1, float b2,
                                                       float eps) {
  const float s = scale ? *scale : 1.0f;
  for (int64_t i = (int64_t)blockIdx.x * kAdamThreads + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * kAdamThreads) {
    if (mask && !mask[i]) continue;
    const float gs = g[i] * s;
    const float mi = b1 * m[i] + (1.0f - b1) * gs;
    const float vi = b2 * v[i] + (1.0f - b2) * (gs * gs);
    m[i] = mi;
    v[i] = vi;
    const float denom = sqrtf(vi) * inv_sqrt_c2 + eps;
    p[i] = p[i] - step_size * (mi / denom);
  }
}

}  // namespace

size_t adam_workspace_bytes(int64_t) { return (size_t)kNormBlocks * sizeof(double) + 16; }

cudaError_t launch_adam(float* p, const float* g, float* m, float* v, const uint8_t* mask,
                        int64_t n, int64_t t, float lr, float b1, float b2, float eps,
                        float max_norm, void* ws, cudaStream_t s) {
  const double c1 = 1.0 - pow((double)b1, (double)t);
  const double c2 = 1.0 - pow((double)b2, (double)t);
  const float step_size = (float)((double)lr / c1);
  const float inv_sqrt_c2 = (float)(1.0 / sqrt(c2));
  float* scale = nullptr;
  if (max_norm > 0.0f) {
    double* part = static_cast<double*>(ws);
    scale = reinterpret_cast<float*>(static_cast<char*>(ws) + (size_t)kNormBlocks * sizeof(double));
    k_sumsq<<<kNormBlocks, kAdamThreads, 0, s>>>(g, mask, n, part);
    k_clip_scale<<<1, 32, 0, s>>>(part, kNormBlocks, max_norm, scale);
    count_launches(2);
  }
  int64_t blocks = (n + kAdamThreads - 1) / kAdamThreads;
  if (blocks > 152 * 8) blocks = 152 * 8;
  k_adam<<<(unsigned)blocks, kAdamThreads, 0, s>>>(p, g, m, v, mask, n, scale, step_size,
                                                   inv_sqrt_c2, b1, b2, eps);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace simx
