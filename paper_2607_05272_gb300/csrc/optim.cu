// Adam (Kingma & Ba 2015), the optimiser step of the policy-gradient training loop
// (Sec. 4.3), on a flat parameter vector.  One elementwise kernel; with gradient
// clipping a fixed-grid sum of squares (fp64 partials) runs first, and every block of the
// update finishes that sum in the same fixed order (so the scale is the same bits on
// every run and in every block).  A device step counter advances in the sum-of-squares
// kernel (or, without clipping, in a one-warp scalar kernel), so that a captured CUDA
// graph of training steps needs no host argument per step.
#include "kernels.h"

namespace simx {

namespace {

constexpr int kAdamThreads = 256;
// Blocks of the sum of squares: fixed, so the sum order is the same on any device; few, so
// that every block of the update finishes their partials in two loads per lane (policy
// vectors are 10^3-10^5 parameters).
constexpr int kNormBlocks = 64;

__global__ void __launch_bounds__(kAdamThreads) k_sumsq(const float* __restrict__ g,
                                                        const uint8_t* __restrict__ mask,
                                                        int64_t n, double* part, int64_t* d_t) {
  // the device step counter advances here, one kernel before the update reads it
  if (d_t && blockIdx.x == 0 && threadIdx.x == 0) *d_t = *d_t + 1;
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

// b^t for t >= 1 by binary powering in fp64 (a few dependent multiplies: a general pow
// is a long fp64 chain, and fp64 is slow on this GPU).
__device__ double pow_int(double b, int64_t t) {
  double r = 1.0;
  while (t > 0) {
    if (t & 1) r *= b;
    b *= b;
    t >>= 1;
  }
  return r;
}

// scal[0] = min(1, max_norm / ||g||) (1 for a zero gradient, or without clipping);
// with a device step counter also t = ++*d_t, scal[1] = lr / (1 - b1^t) and
// scal[2] = 1 / sqrt(1 - b2^t), the bias corrections the host computes otherwise.
__global__ void k_adam_scalars(const double* part, int nb, float max_norm, int64_t* d_t,
                               float lr, float b1, float b2, float* scal) {
  double s = 0.0;  // lane l sums partials l, l + 32, ...; a fixed butterfly combines lanes
  if (part)
    for (int b = (int)threadIdx.x; b < nb; b += 32) s += part[b];
  for (int d = 16; d > 0; d /= 2) s += __shfl_xor_sync(0xffffffffu, s, d);
  if (threadIdx.x != 0) return;
  float sc = 1.0f;
  if (part) {
    const double norm = sqrt(s);
    if (norm > (double)max_norm) sc = (float)((double)max_norm / norm);
  }
  scal[0] = sc;
  if (d_t) {
    const int64_t t = *d_t + 1;
    *d_t = t;
    scal[1] = (float)((double)lr / (1.0 - pow_int((double)b1, t)));
    scal[2] = (float)(1.0 / sqrt(1.0 - pow_int((double)b2, t)));
  }
}

// With `part` (clipping), every block derives the scale (and, with a device counter, the
// bias corrections from the already advanced *d_t) from the sum-of-squares partials itself,
// in the fixed order of k_adam_scalars, so no separate scalar kernel runs; otherwise the
// scalars come from `scal` (k_adam_scalars) or the host.
__global__ void __launch_bounds__(kAdamThreads) k_adam(float* __restrict__ p,
                                                       const float* __restrict__ g,
                                                       float* __restrict__ m, float* __restrict__ v,
                                                       const uint8_t* __restrict__ mask, int64_t n,
                                                       const float* scal, bool dev_t,
                                                       float step_size, float inv_sqrt_c2,
                                                       float b1, float b2, float eps,
                                                       const double* part, int nb, float max_norm,
                                                       const int64_t* d_t, float lr) {
  __shared__ float sh[3];
  float s;
  if (part) {
    if (threadIdx.x < 32) {
      double acc = 0.0;
      for (int b = (int)threadIdx.x; b < nb; b += 32) acc += part[b];
      for (int d = 16; d > 0; d /= 2) acc += __shfl_xor_sync(0xffffffffu, acc, d);
      if (threadIdx.x == 0) {
        float sc = 1.0f;
        const double norm = sqrt(acc);
        if (norm > (double)max_norm) sc = (float)((double)max_norm / norm);
        sh[0] = sc;
        if (dev_t) {
          const int64_t t = *d_t;
          sh[1] = (float)((double)lr / (1.0 - pow_int((double)b1, t)));
          sh[2] = (float)(1.0 / sqrt(1.0 - pow_int((double)b2, t)));
        }
      }
    }
    __syncthreads();
    s = sh[0];
    if (dev_t) {
      step_size = sh[1];
      inv_sqrt_c2 = sh[2];
    }
  } else {
    s = scal ? scal[0] : 1.0f;
    if (dev_t) {
      step_size = scal[1];
      inv_sqrt_c2 = scal[2];
    }
  }
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

// t >= 1: the step number from the host; d_t: a device counter incremented by the step
// (then t is ignored and the workspace is always used).
cudaError_t launch_adam(float* p, const float* g, float* m, float* v, const uint8_t* mask,
                        int64_t n, int64_t t, int64_t* d_t, float lr, float b1, float b2,
                        float eps, float max_norm, void* ws, cudaStream_t s) {
  float step_size = 0.0f, inv_sqrt_c2 = 0.0f;
  if (!d_t) {
    const double c1 = 1.0 - pow((double)b1, (double)t);
    const double c2 = 1.0 - pow((double)b2, (double)t);
    step_size = (float)((double)lr / c1);
    inv_sqrt_c2 = (float)(1.0 / sqrt(c2));
  }
  float* scal = nullptr;
  double* part = nullptr;
  if (max_norm > 0.0f) {
    // clipping: the sum of squares (which also advances a device counter), then the update
    part = static_cast<double*>(ws);
    k_sumsq<<<kNormBlocks, kAdamThreads, 0, s>>>(g, mask, n, part, d_t);
    count_launches(1);
  } else if (d_t) {
    scal = reinterpret_cast<float*>(static_cast<char*>(ws) + (size_t)kNormBlocks * sizeof(double));
    k_adam_scalars<<<1, 32, 0, s>>>(nullptr, kNormBlocks, max_norm, d_t, lr, b1, b2, scal);
    count_launches(1);
  }
  int64_t blocks = (n + kAdamThreads - 1) / kAdamThreads;
  if (blocks > (int64_t)sm_count() * 8) blocks = (int64_t)sm_count() * 8;
  k_adam<<<(unsigned)blocks, kAdamThreads, 0, s>>>(p, g, m, v, mask, n, scal, d_t != nullptr,
                                                   step_size, inv_sqrt_c2, b1, b2, eps, part,
                                                   kNormBlocks, max_norm, d_t, lr);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace simx
