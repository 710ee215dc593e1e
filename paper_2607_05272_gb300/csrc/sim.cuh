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
#include "tc_common.cuh"

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
// columns padded to a multiple of 4 with zeros), bias[l] is [Npad_l].
struct DevMlp {
  const float* Wt[SIMX_MAX_LAYERS];
  const float* bias[SIMX_MAX_LAYERS];
  int dims[SIMX_MAX_LAYERS + 1];
  int npad[SIMX_MAX_LAYERS + 1];
  int n_layers, has_value, n_actions;
  int act[SIMX_MAX_LAYERS];  // simx_act after layer l, -1 for the output layer
  int grid;                  // grid policy: layer l's input on the grid 2^-gx[l]
  int gx[SIMX_MAX_LAYERS];
};

// The FP32 block-wide forward with its weights staged in shared memory (fp32 policies
// whose weights L1 does not hold): one thread streams each layer's rows, in chunks of
// rpc[l] rows, into S stages of cb bytes with bulk copies; every thread reads its
// register tile's weights (te[l] envs x to[l] outputs) from the stage.  The chunk
// sequence of one forward (layer 0's, then layer 1's, ...) repeats every step, so the
// next step's first chunks load during the simulator's phases.  Byte offsets are inside
// the kernel's dynamic shared memory.
struct StagePlan {
  int on;                      // 1: this launch stages the weights
  int S;                       // stages
  int n;                       // chunks per forward
  uint32_t cb;                 // bytes per stage
  uint32_t off;                // first stage
  uint32_t bar_off;            // S mbarriers (8 B each), then the timeout flag (4 B)
  int rpc[SIMX_MAX_LAYERS];    // weight rows per chunk
  int cnt[SIMX_MAX_LAYERS];    // chunks of each layer
  int te[SIMX_MAX_LAYERS], to[SIMX_MAX_LAYERS];   // register tile: envs x outputs
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

// Two fp32 fused multiply-adds in one instruction (fma.rn.f32x2, sm_100 and later): each
// half of the 64-bit operands is one fp32 value (the low half first) and each half of the
// result is the IEEE fma of its own halves, rounded to nearest: the bits of two
// __fmaf_rn.  The tiles below pair adjacent outputs of one env, whose weights arrive as
// adjacent floats of a 16-byte load.
__device__ __forceinline__ uint64_t f2_pack(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f2_unpack(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}

// ---------------------------------------------------------------------------
// Policy network (Sec. 4.2) evaluated for all envs of a block at once.
//
// Activations live in shared memory feature-major, X[k * ld + e] for the block's B
// envs (row stride ld = B + 4 spreads an env's features over the banks), so one
// layer is the small GEMM Y = X^T W^T.  Each thread owns tiles of TE
// envs x 4 outputs; per k it loads one float4 of weights (row k of the transposed,
// padded Wt) and TE activations and issues 2 TE paired fused multiply-adds (f2_fma).
// Every output is still the fp32 chain acc = fma(W[j][k], x[k], acc) over k = 0..K-1 in
// order from acc = 0, then + bias: the same bits as evaluating one env at a time.
// ---------------------------------------------------------------------------
// GELU over rows j0 .. min(j0 + 4, N) - 1, columns 0 .. te - 1 of Y.  Out of line: inlined,
// its code inside the rollout kernel's loop slowed the tanh policies that never run it.
static __device__ __noinline__ void gelu_tile(float* Y, int ld, int j0, int N, int te) {
  for (int j = j0; j < j0 + 4 && j < N; ++j)
    for (int e = 0; e < te; ++e) Y[j * ld + e] = det_gelu(Y[j * ld + e]);
}

// Grid rounding of the grid policy (the exact policy forward): Q(v, e) = clamp(rint(v 2^e),
// -255, 255) 2^-e with ties to even, 0 <= e <= 24.  Both scalings are by exact powers of
// two, so the only rounding is rintf's.
__device__ __forceinline__ float grid_q(float v, int e) {
  const float up = __int_as_float((127 + e) << 23), down = __int_as_float((127 - e) << 23);
  const float r = fminf(fmaxf(rintf(__fmul_rn(v, up)), -255.0f), 255.0f);
  return __fmul_rn(r, down);
}

// Grid rounding of rows j0 .. min(j0 + 4, N) - 1, columns 0 .. te - 1 of Y (after the
// activation).  Out of line, like gelu_tile, so the other policies' loop stays small.
static __device__ __noinline__ void grid_tile(float* Y, int ld, int j0, int N, int te, int e) {
  for (int j = j0; j < j0 + 4 && j < N; ++j)
    for (int c = 0; c < te; ++c) Y[j * ld + c] = grid_q(Y[j * ld + c], e);
}

// The observation of a grid policy on its input grid: rows 0 .. D-1, columns 0 .. B-1 of
// X (row stride ld), split over threads tid, tid + nthr, ...
static __device__ __noinline__ void grid_rows(float* X, int D, int B, int ld, int e, int tid,
                                              int nthr) {
  for (int i = tid; i < D * B; i += nthr) {
    float* x = X + (i / B) * ld + i % B;
    *x = grid_q(*x, e);
  }
}

// act: the activation after this layer: -1 none (output layer), 0 tanh, 1 identity,
// 2 GELU (det_gelu); GRID and gq >= 0: the grid policy's rounding of the activated
// output.  GRID is a template parameter so that the fp32 policies' instantiations carry
// no trace of it (an untaken runtime check here slowed the narrow rollout by about 5 %).
// Threads tid, tid + nthr, ... of the cooperating group take the tiles.
template <int TE, bool GRID>
__device__ __forceinline__ void mlp_tiles(const float* __restrict__ Wt,
                                          const float* __restrict__ bias, int K, int N, int Npad,
                                          const float* X, float* Y, int B, int ld, int act,
                                          int gq, int tid, int nthr) {
  const int neb = B / TE, nob = (N + 3) / 4;
  const int ntiles = neb * nob;
  for (int tile = tid; tile < ntiles; tile += nthr) {
    const int eb = tile % neb, ob = tile / neb;
    uint64_t acc2[TE][2];   // outputs (0, 1) and (2, 3) of each env
#pragma unroll
    for (int e = 0; e < TE; ++e) acc2[e][0] = acc2[e][1] = 0ull;
    const float* wc = Wt + 4 * ob;
    const float* xc = X + TE * eb;
#pragma unroll 4
    for (int k = 0; k < K; ++k) {
      const ulonglong2 w = __ldg(reinterpret_cast<const ulonglong2*>(wc + (size_t)k * Npad));
      float xv[TE];
      if (TE == 4) {
        const float4 x4 = *reinterpret_cast<const float4*>(xc + k * ld);
        xv[0] = x4.x;
        xv[1 % TE] = x4.y;
        xv[2 % TE] = x4.z;
        xv[3 % TE] = x4.w;
      } else {
        xv[0] = xc[k * ld];
      }
#pragma unroll
      for (int e = 0; e < TE; ++e) {
        const uint64_t xx = f2_pack(xv[e], xv[e]);
        acc2[e][0] = f2_fma(w.x, xx, acc2[e][0]);
        acc2[e][1] = f2_fma(w.y, xx, acc2[e][1]);
      }
    }
    float acc[TE][4];
#pragma unroll
    for (int e = 0; e < TE; ++e) {
      f2_unpack(acc2[e][0], acc[e][0], acc[e][1]);
      f2_unpack(acc2[e][1], acc[e][2], acc[e][3]);
    }
#pragma unroll
    for (int o = 0; o < 4; ++o) {
      const int j = 4 * ob + o;
      if (j < N) {
        const float bj = __ldg(bias + j);
#pragma unroll
        for (int e = 0; e < TE; ++e) Y[j * ld + TE * eb + e] = __fadd_rn(acc[e][o], bj);
      }
    }
    // one activation per output, over this thread's own tile
    if (act == 0) {
#pragma unroll 1
      for (int q = 0; q < 4 * TE; ++q) {
        const int j = 4 * ob + q / TE;
        if (j < N) {
          float* y = Y + j * ld + TE * eb + q % TE;
          *y = det_tanh(*y);
        }
      }
    } else if (act == 2) {
      gelu_tile(Y + TE * eb, ld, 4 * ob, N, TE);
    }
    if (GRID && gq >= 0) grid_tile(Y + TE * eb, ld, 4 * ob, N, TE, gq);
  }
}

// Forward through every layer for the block's envs: the observation is in X0,
// layers alternate X0 -> X1 -> X0 ...; returns the buffer holding the last layer
// (logits rows 0..A-1, value row A).  Contains the block barriers.  GRID: the grid
// policy (m.grid set), whose inputs and hidden outputs are rounded to their grids.
template <bool GRID>
__device__ __forceinline__ float* mlp_forward_block(const DevMlp& m, float* X0, float* X1, int B,
                                                   int ld) {
  float* in = X0;
  float* out = X1;
  __syncthreads();
  if (GRID) {
    grid_rows(X0, m.dims[0], B, ld, m.gx[0], threadIdx.x, blockDim.x);
    __syncthreads();
  }
  for (int l = 0; l < m.n_layers; ++l) {
    const int K = m.dims[l], N = m.dims[l + 1], Np = m.npad[l + 1];
    const int th = m.act[l];
    const int gq = (GRID && l + 1 < m.n_layers) ? m.gx[l + 1] : -1;
    // 4-env tiles when they keep every thread busy, otherwise 1-env tiles
    if ((B / 4) * ((N + 3) / 4) >= (int)blockDim.x)
      mlp_tiles<4, GRID>(m.Wt[l], m.bias[l], K, N, Np, in, out, B, ld, th, gq, threadIdx.x, blockDim.x);
    else
      mlp_tiles<1, GRID>(m.Wt[l], m.bias[l], K, N, Np, in, out, B, ld, th, gq, threadIdx.x, blockDim.x);
    __syncthreads();
    float* t = in;
    in = out;
    out = t;
  }
  return in;
}

// The same forward for the Bw envs (columns col0 .. col0 + Bw - 1) whose lanes form this
// warp: only the warp's own lanes take its tiles, so warp barriers replace block
// barriers.  Every output is still the K-ordered fma chain.  Returns the buffer (not
// offset by col0) holding the last layer.
template <bool GRID>
__device__ __forceinline__ float* mlp_forward_warp(const DevMlp& m, float* X0, float* X1, int Bw,
                                                  int ld, int col0) {
  float* in = X0;
  float* out = X1;
  const int lane = (int)(threadIdx.x & 31u);
  __syncwarp();
  if (GRID) {
    grid_rows(X0 + col0, m.dims[0], Bw, ld, m.gx[0], lane, 32);
    __syncwarp();
  }
  for (int l = 0; l < m.n_layers; ++l) {
    const int K = m.dims[l], N = m.dims[l + 1], Np = m.npad[l + 1];
    const int th = m.act[l];
    const int gq = (GRID && l + 1 < m.n_layers) ? m.gx[l + 1] : -1;
    if ((Bw / 4) * ((N + 3) / 4) >= 32)
      mlp_tiles<4, GRID>(m.Wt[l], m.bias[l], K, N, Np, in + col0, out + col0, Bw, ld, th, gq, lane, 32);
    else
      mlp_tiles<1, GRID>(m.Wt[l], m.bias[l], K, N, Np, in + col0, out + col0, Bw, ld, th, gq, lane, 32);
    __syncwarp();
    float* t = in;
    in = out;
    out = t;
  }
  return in;
}

// ---------------------------------------------------------------------------
// The block-wide forward with the weights staged in shared memory (StagePlan).  Thread 0
// keeps S chunks of weight rows in flight (bulk copies completing on one mbarrier per
// stage); every thread owns one register tile of TE envs x TO outputs of the layer and,
// per chunk, waits for its stage, runs its rows k in order (paired fmas, f2_fma) and
// meets the block at a barrier, after which thread 0 refills the stage with the chunk S
// ahead.  Every output is the same K-ordered fma chain from 0 as in mlp_tiles, then +
// bias, the activation and the grid rounding: the same bits.  A wait that times out sets the block's flag; from
// then on nothing is issued or waited for and the step's outputs are garbage, which the
// caller reports as SIMX_DEV_COPY_TIMEOUT.
// ---------------------------------------------------------------------------
struct StagePipe {
  float* stages;
  uint64_t* full;
  volatile int* flag;
  uint32_t cc;      // chunks consumed so far in the launch
  uint32_t total;   // chunks the launch consumes (steps x chunks per forward)
};

// Thread 0: chunk g of the launch's sequence into stage g mod S (nothing past the last).
__device__ __forceinline__ void stage_issue(const DevMlp& m, const StagePlan& P,
                                            const StagePipe& p, uint32_t g) {
  if (g >= p.total || *p.flag) return;
  uint32_t c = g % (uint32_t)P.n;
  int l = 0;
  while (c >= (uint32_t)P.cnt[l]) {
    c -= (uint32_t)P.cnt[l];
    ++l;
  }
  const int Np = m.npad[l + 1];
  const int row0 = (int)c * P.rpc[l];
  const int rows = m.dims[l] - row0 < P.rpc[l] ? m.dims[l] - row0 : P.rpc[l];
  const uint32_t bytes = (uint32_t)(rows * Np) * 4u;
  const uint32_t st = g % (uint32_t)P.S;
  tcx::mbar_arrive_expect_tx(&p.full[st], bytes);
  tcx::bulk_g2s(p.stages + (size_t)st * (P.cb / 4u), m.Wt[l] + (size_t)row0 * Np, bytes,
                &p.full[st]);
}

// Thread 0 at launch start: the barriers, then the first S chunks.
__device__ __forceinline__ void stage_start(const DevMlp& m, const StagePlan& P, const StagePipe& p) {
  for (int i = 0; i < P.S; ++i) tcx::mbar_init(&p.full[i], 1);
  *p.flag = 0;
  tcx::mbar_fence_init();
  for (int i = 0; i < P.S; ++i) stage_issue(m, P, p, (uint32_t)i);
}

// Thread 0 at launch end, after a timeout only: a bounded wait for every stage's copy
// still in flight, so that none lands after the block has exited.
__device__ __forceinline__ void stage_drain(const StagePlan& P, const StagePipe& p) {
  for (uint32_t g = p.cc; g < p.cc + (uint32_t)P.S && g < p.total; ++g)
    tcx::mbar_wait(&p.full[g % (uint32_t)P.S], (g / (uint32_t)P.S) & 1u, 200000000ll);
}

// One layer of the staged forward; returns the chunks consumed so far.
template <int TE, int TO, bool GRID>
__device__ __forceinline__ uint32_t layer_staged(const DevMlp& m, const StagePlan& P,
                                                     StagePipe p, int l, const float* X, float* Y,
                                                     int B, int ld, int gq) {
  const int K = m.dims[l], N = m.dims[l + 1], Np = m.npad[l + 1];
  const int neb = B / TE, nob = (N + TO - 1) / TO;
  const int tid = (int)threadIdx.x;
  const bool active = tid < neb * nob;
  const int eb = tid % neb, ob = tid / neb;
  uint64_t acc2[TE][TO / 2];   // adjacent output pairs of each env
#pragma unroll
  for (int e = 0; e < TE; ++e)
#pragma unroll
    for (int o = 0; o < TO / 2; ++o) acc2[e][o] = 0ull;
  const int rpc = P.rpc[l];
  for (int j = 0; j < P.cnt[l]; ++j) {
    const uint32_t st = p.cc % (uint32_t)P.S;
    if (!*p.flag && !tcx::mbar_wait(&p.full[st], (p.cc / (uint32_t)P.S) & 1u, 2000000000ll))
      *p.flag = 1;
    const float* w = p.stages + (size_t)st * (P.cb / 4u) + TO * ob;
    const float* xc = X + (size_t)(j * rpc) * ld + TE * eb;
    const int rows = K - j * rpc < rpc ? K - j * rpc : rpc;
    if (active) {
#pragma unroll 8
      for (int k = 0; k < rows; ++k) {
        uint64_t wv[TO / 2];
#pragma unroll
        for (int q = 0; q < TO / 4; ++q) {
          const ulonglong2 w4 = *reinterpret_cast<const ulonglong2*>(w + k * Np + 4 * q);
          wv[2 * q] = w4.x;
          wv[2 * q + 1] = w4.y;
        }
        float xv[TE];
        if (TE == 4) {
          const float4 x4 = *reinterpret_cast<const float4*>(xc + k * ld);
          xv[0] = x4.x;
          xv[1 % TE] = x4.y;
          xv[2 % TE] = x4.z;
          xv[3 % TE] = x4.w;
        } else if (TE == 2) {
          const float2 x2 = *reinterpret_cast<const float2*>(xc + k * ld);
          xv[0] = x2.x;
          xv[1 % TE] = x2.y;
        } else {
          xv[0] = xc[k * ld];
        }
#pragma unroll
        for (int e = 0; e < TE; ++e) {
          const uint64_t xx = f2_pack(xv[e], xv[e]);
#pragma unroll
          for (int o = 0; o < TO / 2; ++o) acc2[e][o] = f2_fma(wv[o], xx, acc2[e][o]);
        }
      }
    }
    __syncthreads();
    if (tid == 0) {
      tcx::fence_async_smem();
      stage_issue(m, P, p, p.cc + (uint32_t)P.S);
    }
    ++p.cc;
  }
  if (active) {
    float acc[TE][TO];
#pragma unroll
    for (int e = 0; e < TE; ++e)
#pragma unroll
      for (int o = 0; o < TO / 2; ++o) f2_unpack(acc2[e][o], acc[e][2 * o], acc[e][2 * o + 1]);
    const int act = m.act[l];
#pragma unroll
    for (int o = 0; o < TO; ++o) {
      const int jj = TO * ob + o;
      if (jj < N) {
        const float bj = __ldg(m.bias[l] + jj);
#pragma unroll
        for (int e = 0; e < TE; ++e) {
          float v = __fadd_rn(acc[e][o], bj);
          if (act == 0) v = det_tanh(v);
          Y[jj * ld + TE * eb + e] = v;
        }
      }
    }
    if (act == 2)
      for (int o4 = 0; o4 < TO; o4 += 4) gelu_tile(Y + TE * eb, ld, TO * ob + o4, N, TE);
    if (GRID && gq >= 0)
      for (int o4 = 0; o4 < TO; o4 += 4) grid_tile(Y + TE * eb, ld, TO * ob + o4, N, TE, gq);
  }
  return p.cc;
}

// Forward through every layer with staged weights (the same buffers and result as
// mlp_forward_block).  Contains the block barriers.  Inlined: as an out-of-line call it
// ran the c4 policy 26 % slower inside the rollout.
template <bool GRID>
__device__ __forceinline__ float* mlp_forward_staged(const DevMlp& m, const StagePlan& P,
                                                    StagePipe& p, float* X0, float* X1, int B,
                                                    int ld) {
  float* in = X0;
  float* out = X1;
  __syncthreads();
  if (GRID) {
    grid_rows(X0, m.dims[0], B, ld, m.gx[0], threadIdx.x, blockDim.x);
    __syncthreads();
  }
  for (int l = 0; l < m.n_layers; ++l) {
    const int gq = (GRID && l + 1 < m.n_layers) ? m.gx[l + 1] : -1;
    switch (P.te[l] * 16 + P.to[l]) {
      case 4 * 16 + 8: p.cc = layer_staged<4, 8, GRID>(m, P, p, l, in, out, B, ld, gq); break;
      case 2 * 16 + 8: p.cc = layer_staged<2, 8, GRID>(m, P, p, l, in, out, B, ld, gq); break;
      case 4 * 16 + 4: p.cc = layer_staged<4, 4, GRID>(m, P, p, l, in, out, B, ld, gq); break;
      case 2 * 16 + 4: p.cc = layer_staged<2, 4, GRID>(m, P, p, l, in, out, B, ld, gq); break;
      case 1 * 16 + 8: p.cc = layer_staged<1, 8, GRID>(m, P, p, l, in, out, B, ld, gq); break;
      default: p.cc = layer_staged<1, 4, GRID>(m, P, p, l, in, out, B, ld, gq); break;
    }
    __syncthreads();
    float* t = in;
    in = out;
    out = t;
  }
  return in;
}

// Action from the logits column z[i * B] of one env (Sec. 4.2): SAMPLE draws by
// inversion of the cumulative softmax with a POLICY-stream uniform, ARGMAX takes the
// first largest logit.  p_i = e^{z_i - max} are computed by the env's lanes in
// parallel and summed by lane 0 in index order.  logp/value valid in every lane.
template <int G>
__device__ __forceinline__ int sample_action(const DevMlp& m, const float* z, int B,
                                             float* scratch, int mode, uint32_t key0,
                                             uint32_t key1, uint32_t step, uint32_t env,
                                             float& logp, float& value, const Grp<G>& g) {
  const int A = m.n_actions;
  float mx = -__uint_as_float(0x7F800000u);
  int ai = 0x7FFFFFFF;
  for (int i = (int)g.gl; i < A; i += G) {
    const float v = z[i * B];
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
  for (int i = (int)g.gl; i < A; i += G) scratch[i] = det_exp(__fsub_rn(z[i * B], mx));
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
    lp = __fsub_rn(__fsub_rn(z[a * B], mx), det_log(S));
  }
  a = (int)g.shfl((uint32_t)a, 0);
  logp = g.shflf(lp, 0);
  value = m.has_value ? z[A * B] : 0.0f;
  g.sync();
  return a;
}

}  // namespace simx
