// sim.cuh — device-side environment state, lane-group helpers and the fused
// policy MLP used by the rollout, step and policy-forward kernels.
//
// Execution model: each environment is owned by a group of G consecutive lanes of
// a warp (G = 8: four environments per warp).  Scalar environment state is held
// replicated in the group's registers and updated identically by every lane;
// per-server state (ROUTE mode) lives in lane k for server k; arrival candidates
// are generated G at a time, one per lane, and combined with group ballots and
// shuffle scans.  Rings (the per-(server, type) FIFO queues of Sec. 3.1) live in
// global memory, one contiguous block per environment.
#pragma once
#include <cstdint>

#include "../../include/simx.h"
#include "devmath.cuh"

namespace simx {

// Header fields of the SoA state ([field][env]); the same order as the canonical
// state image.
enum : int {
  F_NOW = 0, F_TG, F_CJ, F_CT, F_SWI, F_SWT, F_MST, F_EP, F_EPO, F_PT, F_PTY, F_PC,
  F_NARR, F_NDROP, F_NDISP, F_NBAT, F_SWLO, F_SWHI, F_TLD, F_PREV, F_NLAST, F_TLAST,
  F_LMW, F_RATE, F_NA0, F_NA1, F_ND0, F_ND1, F_STATUS, F_COUNT
};

struct DevState {
  uint32_t* hdr;   // [F_COUNT][E]
  uint32_t* srv;   // [2][K][E]: busy_until, batch size
  uint32_t* qh;    // [K][T][E] ring head
  uint32_t* qc;    // [K][T][E] queue length
  uint32_t* ring;  // [E][K][T][cap] arrival times
  uint32_t* cost;  // [E][K][cap] per-request costs of the cost type (or null)
  uint32_t E, K, T, cap;
};

// Policy parameters repacked for the device: Wt[l] is [K_l][Npad_l] (transposed,
// columns padded to a multiple of 4G with zeros), bias[l] is [Npad_l].
struct DevMlp {
  const float* Wt[SIMX_MAX_LAYERS];
  const float* bias[SIMX_MAX_LAYERS];
  int dims[SIMX_MAX_LAYERS + 1];
  int npad[SIMX_MAX_LAYERS + 1];
  int n_layers, has_value, n_actions;
};

template <int G>
struct Grp {
  uint32_t lane, gl, gi, mask;
  __device__ __forceinline__ Grp() {
    lane = threadIdx.x & 31u;
    gl = lane % G;
    gi = lane / G;
    mask = (G == 32) ? 0xFFFFFFFFu : (((1u << G) - 1u) << (gi * G));
  }
  __device__ __forceinline__ uint32_t ballot(bool p) const {
    const uint32_t b = __ballot_sync(mask, p);
    return (G == 32) ? b : ((b >> (gi * G)) & ((1u << G) - 1u));
  }
  __device__ __forceinline__ uint32_t shfl(uint32_t v, int src) const {
    return __shfl_sync(mask, v, src, G);
  }
  __device__ __forceinline__ float shflf(float v, int src) const {
    return __shfl_sync(mask, v, src, G);
  }
  __device__ __forceinline__ uint32_t sum(uint32_t v) const {
#pragma unroll
    for (int d = G / 2; d > 0; d >>= 1) v += __shfl_xor_sync(mask, v, d, G);
    return v;
  }
  __device__ __forceinline__ uint64_t sum64(uint64_t v) const {
#pragma unroll
    for (int d = G / 2; d > 0; d >>= 1) {
      const uint32_t lo = __shfl_xor_sync(mask, (uint32_t)v, d, G);
      const uint32_t hi = __shfl_xor_sync(mask, (uint32_t)(v >> 32), d, G);
      v += ((uint64_t)hi << 32) | lo;
    }
    return v;
  }
  __device__ __forceinline__ uint32_t bor(uint32_t v) const {
#pragma unroll
    for (int d = G / 2; d > 0; d >>= 1) v |= __shfl_xor_sync(mask, v, d, G);
    return v;
  }
  __device__ __forceinline__ uint32_t scan_incl(uint32_t v) const {
#pragma unroll
    for (int d = 1; d < G; d <<= 1) {
      const uint32_t y = __shfl_up_sync(mask, v, d, G);
      if (gl >= (uint32_t)d) v += y;
    }
    return v;
  }
  __device__ __forceinline__ void sync() const { __syncwarp(mask); }
};

// One tanh MLP layer for one environment, computed by its G lanes from the
// shared-memory activation vector x[0..K) into y[0..N) (a second buffer).
// Lane gl owns outputs 4 gl + 4 G b + c, taken in passes of at most kPass column
// blocks (16 accumulators); every output is the fp32 fused multiply-add chain over
// k = 0..K-1 in order from 0, then + bias (Sec. 4.2).  The k loop is unrolled by
// four (one float4 of activations, four weight rows) with the per-output order
// unchanged.  tanh is applied afterwards, one output per lane at a time.
constexpr int kPass = 4;

template <int G>
__device__ __forceinline__ void mlp_layer(const float* __restrict__ Wt,
                                          const float* __restrict__ bias, int K, int N,
                                          int Npad, const float* x, float* y, bool do_tanh,
                                          const Grp<G>& g) {
  const int nb = Npad / (4 * G);
  const float* wp = Wt + 4 * g.gl;
  for (int p0 = 0; p0 < nb; p0 += kPass) {
    float acc[4 * kPass];
#pragma unroll
    for (int q = 0; q < 4 * kPass; ++q) acc[q] = 0.0f;
    int k = 0;
    for (; k + 4 <= K; k += 4) {
      const float4 xv = *reinterpret_cast<const float4*>(x + k);
      const float* wr = wp + (size_t)k * Npad + 4 * G * p0;
#pragma unroll
      for (int b = 0; b < kPass; ++b) {
        if (p0 + b < nb) {
          const float4 w0 = __ldg(reinterpret_cast<const float4*>(wr + 4 * G * b));
          const float4 w1 = __ldg(reinterpret_cast<const float4*>(wr + Npad + 4 * G * b));
          const float4 w2 = __ldg(reinterpret_cast<const float4*>(wr + 2 * Npad + 4 * G * b));
          const float4 w3 = __ldg(reinterpret_cast<const float4*>(wr + 3 * Npad + 4 * G * b));
          float* a4 = acc + 4 * b;
          a4[0] = __fmaf_rn(w3.x, xv.w, __fmaf_rn(w2.x, xv.z, __fmaf_rn(w1.x, xv.y, __fmaf_rn(w0.x, xv.x, a4[0]))));
          a4[1] = __fmaf_rn(w3.y, xv.w, __fmaf_rn(w2.y, xv.z, __fmaf_rn(w1.y, xv.y, __fmaf_rn(w0.y, xv.x, a4[1]))));
          a4[2] = __fmaf_rn(w3.z, xv.w, __fmaf_rn(w2.z, xv.z, __fmaf_rn(w1.z, xv.y, __fmaf_rn(w0.z, xv.x, a4[2]))));
          a4[3] = __fmaf_rn(w3.w, xv.w, __fmaf_rn(w2.w, xv.z, __fmaf_rn(w1.w, xv.y, __fmaf_rn(w0.w, xv.x, a4[3]))));
        }
      }
    }
    for (; k < K; ++k) {
      const float xk = x[k];
      const float* wr = wp + (size_t)k * Npad + 4 * G * p0;
#pragma unroll
      for (int b = 0; b < kPass; ++b) {
        if (p0 + b < nb) {
          const float4 w4 = __ldg(reinterpret_cast<const float4*>(wr + 4 * G * b));
          acc[4 * b + 0] = __fmaf_rn(w4.x, xk, acc[4 * b + 0]);
          acc[4 * b + 1] = __fmaf_rn(w4.y, xk, acc[4 * b + 1]);
          acc[4 * b + 2] = __fmaf_rn(w4.z, xk, acc[4 * b + 2]);
          acc[4 * b + 3] = __fmaf_rn(w4.w, xk, acc[4 * b + 3]);
        }
      }
    }
#pragma unroll
    for (int b = 0; b < kPass; ++b) {
      if (p0 + b < nb) {
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) {
          const int j = 4 * (int)g.gl + 4 * G * (p0 + b) + cc;
          if (j < N) y[j] = __fadd_rn(acc[4 * b + cc], __ldg(bias + j));
        }
      }
    }
  }
  g.sync();
  if (do_tanh) {
    for (int j = (int)g.gl; j < N; j += G) y[j] = det_tanh(y[j]);
    g.sync();
  }
}

// Policy head (Sec. 4.2) on the observation in bufA: forward through all layers
// (alternating bufA / bufB), then (mode SAMPLE) categorical sampling by inversion of
// the cumulative softmax with a POLICY-stream uniform, or (ARGMAX) the first
// largest logit.  p_i = e^{z_i - max} are computed by the lanes in parallel and summed
// by lane 0 in index order.  Returns the action; logp/value valid in every lane;
// *zout (if given) points at the logits.  scratch holds n_actions floats.
template <int G>
__device__ __forceinline__ int policy_eval(const DevMlp& m, float* bufA, float* bufB,
                                           float* scratch, int mode, uint32_t key0,
                                           uint32_t key1, uint32_t step, uint32_t env,
                                           float& logp, float& value, const Grp<G>& g,
                                           float** zout = nullptr) {
  float* in = bufA;
  float* out = bufB;
  for (int l = 0; l < m.n_layers; ++l) {
    mlp_layer<G>(m.Wt[l], m.bias[l], m.dims[l], m.dims[l + 1], m.npad[l + 1], in, out,
                 l + 1 < m.n_layers, g);
    float* t = in;
    in = out;
    out = t;
  }
  const float* z = in;
  if (zout) *zout = in;
  const int A = m.n_actions;
  // group argmax (first index of the largest logit)
  float mx = -__uint_as_float(0x7F800000u);
  int ai = 0x7FFFFFFF;
  for (int i = (int)g.gl; i < A; i += G) {
    const float v = z[i];
    if (v > mx) {
      mx = v;
      ai = i;
    }
  }
#pragma unroll
  for (int d = G / 2; d > 0; d >>= 1) {
    const float om = __shfl_xor_sync(g.mask, mx, d, G);
    const int oi = __shfl_xor_sync(g.mask, ai, d, G);
    if (om > mx || (om == mx && oi < ai)) {
      mx = om;
      ai = oi;
    }
  }
  for (int i = (int)g.gl; i < A; i += G) scratch[i] = det_exp(__fsub_rn(z[i], mx));
  g.sync();
  int a = 0;
  float lp = 0.0f;
  if (g.gl == 0) {
    float S = 0.0f;
    for (int i = 0; i < A; ++i) S = __fadd_rn(S, scratch[i]);
    if (mode == SIMX_POLICY_ARGMAX) {
      a = ai;
    } else {
      const U4 w = philox(step, env, kStreamPolicy, 0u, key0, key1);
      const float thr = __fmul_rn(u_open1(w.x), S);
      float cum = 0.0f;
      a = A - 1;
      for (int i = 0; i < A; ++i) {
        cum = __fadd_rn(cum, scratch[i]);
        if (cum > thr) {
          a = i;
          break;
        }
      }
    }
    lp = __fsub_rn(__fsub_rn(z[a], mx), det_log(S));
  }
  a = (int)g.shfl((uint32_t)a, 0);
  logp = g.shflf(lp, 0);
  value = m.has_value ? z[A] : 0.0f;
  g.sync();
  return a;
}

}  // namespace simx
