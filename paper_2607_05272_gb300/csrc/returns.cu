// returns.cu — REINFORCE returns and GAE advantages over the [T][E] rollout
// buffer (Sec. 4.3; GAE after Schulman et al. 2016), and the mean-return baseline.
//
// Both recurrences are first-order affine maps run backwards in time,
//   x_t = delta_t + c_t x_{t+1},
// REINFORCE: x = G, delta_t = r_t, c_t = gamma (1 - d_t), x_T = last_value;
// GAE:       x = A, delta_t = r_t + gamma (1 - d_t) V_{t+1} - V_t,
//            c_t = gamma lambda (1 - d_t), x_T = 0.
// Large env counts with 16-byte aligned rows take k_returns_wide: one thread owns four
// adjacent envs for the whole horizon (one pass: every input read once, every output
// written once, 17 bytes per sample for GAE), loading 8 time steps ahead with 16-byte
// loads, so a block reads 1 KB of each row per step.  Otherwise:
// a block owns 32 envs (threadIdx.x) and splits time into S chunks (threadIdx.y).
// Each thread composes its chunk's map x_{t0} = a x_{t1} + b, one thread per env
// chains the S maps in shared memory, then every thread replays its chunk from the
// right carry.  Loads are coalesced across envs; no global scratch is needed.
#include <cstdint>

#include "kernels.h"

namespace simx {

constexpr int kRetMaxChunks = 32;

__global__ void __launch_bounds__(1024)
k_returns_gae(const float* __restrict__ rew, const float* __restrict__ val,
              const uint8_t* __restrict__ done, const float* __restrict__ last_val, int64_t T,
              int64_t E, int64_t ld, float gamma, float lam, float* __restrict__ ret,
              float* __restrict__ adv) {
  __shared__ float sa[kRetMaxChunks][32], sb[kRetMaxChunks][32], scarry[kRetMaxChunks][32];
  const int64_t e = (int64_t)blockIdx.x * 32 + threadIdx.x;
  const int S = blockDim.y, j = threadIdx.y;
  const bool gae_mode = lam >= 0.0f;
  const float cmul = gae_mode ? gamma * lam : gamma;
  const int64_t L = (T + S - 1) / S;
  const int64_t t0 = (int64_t)j * L;
  const int64_t t1 = t0 + L < T ? t0 + L : T;
  const bool live = e < E;
  float last = 0.0f;
  if (live && last_val) last = last_val[e];
  // pass 1: this chunk's map with a zero carry
  float a = 1.0f, b = 0.0f;
  if (live) {
    float vnext = 0.0f;
    if (gae_mode) vnext = (t1 < T) ? val[t1 * ld + e] : last;
    for (int64_t t = t1 - 1; t >= t0; --t) {
      const int64_t o = t * ld + e;
      const float mask = done[o] ? 0.0f : 1.0f;
      float delta = rew[o];
      if (gae_mode) {
        const float v = val[o];
        delta = delta + gamma * mask * vnext - v;
        vnext = v;
      }
      const float c = cmul * mask;
      b = delta + c * b;
      a = c * a;
    }
  }
  sa[j][threadIdx.x] = a;
  sb[j][threadIdx.x] = b;
  __syncthreads();
  if (j == 0) {
    float carry = gae_mode ? 0.0f : last;
    for (int q = S - 1; q >= 0; --q) {
      scarry[q][threadIdx.x] = carry;
      carry = sb[q][threadIdx.x] + sa[q][threadIdx.x] * carry;
    }
  }
  __syncthreads();
  if (!live) return;
  // pass 2: replay with the carry that enters the chunk from the right
  float x = scarry[j][threadIdx.x];
  float vnext = 0.0f;
  if (gae_mode) vnext = (t1 < T) ? val[t1 * ld + e] : last;
  for (int64_t t = t1 - 1; t >= t0; --t) {
    const int64_t o = t * ld + e;
    const float mask = done[o] ? 0.0f : 1.0f;
    float delta = rew[o];
    float v = 0.0f;
    if (gae_mode) {
      v = val[o];
      delta = delta + gamma * mask * vnext - v;
      vnext = v;
    }
    x = delta + cmul * mask * x;
    if (gae_mode) {
      adv[o] = x;
      ret[o] = x + v;
    } else {
      ret[o] = x;
      if (adv) adv[o] = x;
    }
  }
}

constexpr int kWideU = 8;                 // time steps loaded ahead
constexpr int kWideThreads = 64;          // 256 envs per block: every SM gets blocks from 65,536 envs
constexpr int64_t kWideMinEnvs = 65536;

__device__ __forceinline__ float4 ld4(const float* p) { return *reinterpret_cast<const float4*>(p); }
__device__ __forceinline__ void st4(float* p, float4 v) { *reinterpret_cast<float4*>(p) = v; }

template <bool GAE>
__global__ void __launch_bounds__(kWideThreads, 8)
k_returns_wide(const float* __restrict__ rew, const float* __restrict__ val,
               const uint8_t* __restrict__ done, const float* __restrict__ last_val, int64_t T,
               int64_t E, int64_t ld, float gamma, float lam, float* __restrict__ ret,
               float* __restrict__ adv) {
  const int64_t e = ((int64_t)blockIdx.x * kWideThreads + threadIdx.x) * 4;
  if (e >= E) return;
  const float cmul = GAE ? gamma * lam : gamma;
  float4 last = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
  if (last_val) last = ld4(last_val + e);
  float x[4] = {GAE ? 0.0f : last.x, GAE ? 0.0f : last.y, GAE ? 0.0f : last.z, GAE ? 0.0f : last.w};
  float vn[4] = {last.x, last.y, last.z, last.w};
  for (int64_t tb = T; tb > 0; tb -= kWideU) {
    const int n = tb < kWideU ? (int)tb : kWideU;
    float4 r[kWideU], v[kWideU];
    uint32_t d[kWideU];
#pragma unroll
    for (int i = 0; i < kWideU; ++i) {
      if (i < n) {
        const int64_t o = (tb - 1 - i) * ld + e;
        r[i] = ld4(rew + o);
        d[i] = *reinterpret_cast<const uint32_t*>(done + o);
        if (GAE) v[i] = ld4(val + o);
      }
    }
#pragma unroll
    for (int i = 0; i < kWideU; ++i) {
      if (i < n) {
        const int64_t o = (tb - 1 - i) * ld + e;
        const float rv[4] = {r[i].x, r[i].y, r[i].z, r[i].w};
        float vv[4] = {0.0f, 0.0f, 0.0f, 0.0f};
        if (GAE) {
          vv[0] = v[i].x;
          vv[1] = v[i].y;
          vv[2] = v[i].z;
          vv[3] = v[i].w;
        }
        float o4[4], g4[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float mask = ((d[i] >> (8 * k)) & 0xFFu) ? 0.0f : 1.0f;
          float delta = rv[k];
          if (GAE) {
            delta = delta + gamma * mask * vn[k] - vv[k];
            vn[k] = vv[k];
          }
          x[k] = delta + cmul * mask * x[k];
          o4[k] = x[k];
          g4[k] = x[k] + vv[k];
        }
        if (GAE) {
          st4(adv + o, make_float4(o4[0], o4[1], o4[2], o4[3]));
          st4(ret + o, make_float4(g4[0], g4[1], g4[2], g4[3]));
        } else {
          st4(ret + o, make_float4(o4[0], o4[1], o4[2], o4[3]));
          if (adv) st4(adv + o, make_float4(o4[0], o4[1], o4[2], o4[3]));
        }
      }
    }
  }
}

static bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

cudaError_t launch_returns_gae(const float* rew, const float* val, const uint8_t* done,
                               const float* last_val, int64_t T, int64_t E, int64_t ld,
                               float gamma, float lam, float* ret, float* adv, cudaStream_t s) {
  if (T <= 0 || E <= 0) return cudaSuccess;
  const bool gae = lam >= 0.0f;
  if (E >= kWideMinEnvs && E % 4 == 0 && ld % 4 == 0 && aligned16(rew) && aligned16(ret) &&
      ((uintptr_t)done & 3u) == 0 && (!gae || aligned16(val)) && (!adv || aligned16(adv)) &&
      (!last_val || aligned16(last_val))) {
    const unsigned grid = (unsigned)((E / 4 + kWideThreads - 1) / kWideThreads);
    if (gae)
      k_returns_wide<true><<<grid, kWideThreads, 0, s>>>(rew, val, done, last_val, T, E, ld, gamma, lam, ret, adv);
    else
      k_returns_wide<false><<<grid, kWideThreads, 0, s>>>(rew, val, done, last_val, T, E, ld, gamma, lam, ret, adv);
    count_launches(1);
    return cudaGetLastError();
  }
  // Enough (env, chunk) threads to fill the GPU: ~300k threads, chunks of >= 16 steps.
  int S = 1;
  while (S < kRetMaxChunks && E * S * 2 <= 311296 && T / (S * 2) >= 16) S *= 2;
  const dim3 block(32, S);
  const dim3 grid((unsigned)((E + 31) / 32));
  k_returns_gae<<<grid, block, 0, s>>>(rew, val, done, last_val, T, E, ld, gamma, lam, ret, adv);
  count_launches(1);
  return cudaGetLastError();
}

// Mean-return baseline: per-block fp64 partial sums, then every block of the second
// kernel reduces the partials in block order (same mean everywhere) and centres.
constexpr int kBaseThreads = 256;

int baseline_blocks(int64_t n) {
  int64_t b = (n + kBaseThreads * 8 - 1) / (kBaseThreads * 8);
  if (b > 1024) b = 1024;
  if (b < 1) b = 1;
  return (int)b;
}

__global__ void __launch_bounds__(kBaseThreads)
k_base_partial(const float* __restrict__ x, int64_t n, double* __restrict__ part) {
  __shared__ double sh[kBaseThreads];
  double acc = 0.0;
  for (int64_t i = (int64_t)blockIdx.x * kBaseThreads + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * kBaseThreads)
    acc += (double)x[i];
  sh[threadIdx.x] = acc;
  __syncthreads();
  for (int d = kBaseThreads / 2; d > 0; d >>= 1) {
    if ((int)threadIdx.x < d) sh[threadIdx.x] += sh[threadIdx.x + d];
    __syncthreads();
  }
  if (threadIdx.x == 0) part[blockIdx.x] = sh[0];
}

__global__ void __launch_bounds__(kBaseThreads)
k_base_center(const float* __restrict__ x, int64_t n, const double* __restrict__ part, int nparts,
              float* __restrict__ adv, float* __restrict__ mean_out) {
  __shared__ double sh[kBaseThreads];
  double acc = 0.0;
  for (int i = threadIdx.x; i < nparts; i += kBaseThreads) acc += part[i];
  sh[threadIdx.x] = acc;
  __syncthreads();
  for (int d = kBaseThreads / 2; d > 0; d >>= 1) {
    if ((int)threadIdx.x < d) sh[threadIdx.x] += sh[threadIdx.x + d];
    __syncthreads();
  }
  const double mean = sh[0] / (double)n;
  if (blockIdx.x == 0 && threadIdx.x == 0 && mean_out) mean_out[0] = (float)mean;
  if (!adv) return;
  for (int64_t i = (int64_t)blockIdx.x * kBaseThreads + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * kBaseThreads)
    adv[i] = (float)((double)x[i] - mean);
}

cudaError_t launch_baseline(const float* x, int64_t n, float* adv, float* mean_out, double* ws,
                            int nblocks, cudaStream_t s) {
  k_base_partial<<<nblocks, kBaseThreads, 0, s>>>(x, n, ws);
  k_base_center<<<nblocks, kBaseThreads, 0, s>>>(x, n, ws, nblocks, adv, mean_out);
  count_launches(2);
  return cudaGetLastError();
}

}  // namespace simx
