// loss_fused.cu — REINFORCE / PPO loss gradient (Sec. 4.3) in one persistent kernel
// for policies whose parameters fit in shared memory.
//
// Each block walks row tiles of R minibatch rows (64 when two blocks of that size fit
// in one SM's shared memory, else 32).  Per tile: gather the rows' observations, run
// the forward pass keeping every activation in shared memory (feature-major,
// [feature][row]), evaluate the loss head per row (log-softmax,
// rho, clipped surrogate, entropy, value residual -> dL/dZ), then the backward pass:
//   dW_l += dZ_l^T H_l   (each thread owns 4 x 4 blocks of dW_l, accumulated in
//                         shared memory across all of the block's tiles),
//   db_l += column sums of dZ_l,
//   dZ_{l-1} = (dZ_l W_l) * (1 - H_l^2).
// Every GEMM is a register-tiled shared-memory product (4 rows x 4 columns per thread,
// one float4 of each operand per step).  At the end each block writes its dW/db and
// fp64 loss statistics; a second kernel sums the blocks in block order, so the result
// is deterministic for a given launch configuration.  Nothing touches HBM but the
// gathered observations and the per-block partials.
//
// Grid policies (the exact policy forward) run here only: the gathered observations and
// every hidden output are rounded to their grids exactly as the rollout rounds them, so
// the forward reproduces the rollout's logits; the backward passes the gradient through
// each rounding unchanged (the straight-through estimator): the activation's derivative
// at the pre-activation is stored beside the rounded output, and dW uses the rounded
// layer inputs.
#include <cstdint>

#include "devmath.cuh"
#include "kernels.h"

namespace simx {

constexpr int kLThreads = 256;         // threads per block
// Rows per tile R (64 when the shared-memory plan allows, else 32); activation
// buffers have row stride R + 4.

// Y[j][r] = sum_k Wt[k][j] X[k][r] (+ epilogue) for rows r < R, outputs j < N.
// Wt is row-major with row stride ldw (a multiple of 4, 16-byte aligned).  Each
// thread owns TE rows x 4 outputs: 4-row tiles when they give every thread a tile,
// else 1-row tiles (thin layers such as the logits).
// epi 0: + bias, then the activation `act` (-1 none, 0 tanh, 1 identity, 2 GELU; for
// GELU its derivative is written to D as well); with gq >= 0 (a grid policy's hidden
// layer) the activation a is written to Y rounded to its grid, Q(a, gq), and its
// derivative at the pre-activation (1 - a^2, 1 or GELU's) to D: the gradient passes the
// rounding unchanged (straight through).  epi 1: times the derivative of the activation
// `act` of H's layer: 1 - H^2 (tanh, H = the activations), 1 (identity), or H itself
// (GELU and grid layers: H = the stored derivative).
__device__ __forceinline__ void grid_act(float& y, float& d, int act, int gq) {
  float a = y, g = 1.0f;
  if (act == 0) {
    a = det_tanh(y);
    g = 1.0f - a * a;
  } else if (act == 2) {
    det_gelu_grad(y, a, g);
  }
  d = g;
  y = grid_q(a, gq);
}

template <int R, int TE>
__device__ __forceinline__ void tile_gemm_t(const float* __restrict__ Wt, int ldw, int K, int N,
                                            const float* X, float* Y, int epi,
                                            const float* __restrict__ bias, int act,
                                            const float* H, float* D, int gq) {
  constexpr int kLld = R + 4;
  const int neb = R / TE, nob = (N + 3) / 4;
  for (int tile = threadIdx.x; tile < neb * nob; tile += blockDim.x) {
    const int eb = tile % neb, ob = tile / neb;
    float acc[TE][4];
#pragma unroll
    for (int e = 0; e < TE; ++e)
#pragma unroll
      for (int o = 0; o < 4; ++o) acc[e][o] = 0.0f;
    const float* wc = Wt + 4 * ob;
    const float* xc = X + TE * eb;
#pragma unroll 4
    for (int k = 0; k < K; ++k) {
      const float4 w = *reinterpret_cast<const float4*>(wc + (size_t)k * ldw);
      float xv[TE];
      if (TE == 4) {
        const float4 x = *reinterpret_cast<const float4*>(xc + k * kLld);
        xv[0] = x.x;
        xv[1 % TE] = x.y;
        xv[2 % TE] = x.z;
        xv[3 % TE] = x.w;
      } else {
        xv[0] = xc[k * kLld];
      }
#pragma unroll
      for (int e = 0; e < TE; ++e) {
        acc[e][0] = __fmaf_rn(w.x, xv[e], acc[e][0]);
        acc[e][1] = __fmaf_rn(w.y, xv[e], acc[e][1]);
        acc[e][2] = __fmaf_rn(w.z, xv[e], acc[e][2]);
        acc[e][3] = __fmaf_rn(w.w, xv[e], acc[e][3]);
      }
    }
    if (TE == 4) {
      // the tile's 4 rows of output j are one 16-byte store (conflict-free across
      // the warp's consecutive row blocks)
#pragma unroll
      for (int o = 0; o < 4; ++o) {
        const int j = 4 * ob + o;
        if (j >= N) continue;
        float4 v = make_float4(acc[0][o], acc[1 % TE][o], acc[2 % TE][o], acc[3 % TE][o]);
        if (epi == 0) {
          const float bj = bias[j];
          v.x = __fadd_rn(v.x, bj);
          v.y = __fadd_rn(v.y, bj);
          v.z = __fadd_rn(v.z, bj);
          v.w = __fadd_rn(v.w, bj);
        } else if (act == 0) {
          const float4 h = *reinterpret_cast<const float4*>(H + j * kLld + 4 * eb);
          v.x = v.x * (1.0f - h.x * h.x);
          v.y = v.y * (1.0f - h.y * h.y);
          v.z = v.z * (1.0f - h.z * h.z);
          v.w = v.w * (1.0f - h.w * h.w);
        } else if (act == 2) {
          const float4 dd = *reinterpret_cast<const float4*>(H + j * kLld + 4 * eb);
          v.x = v.x * dd.x;
          v.y = v.y * dd.y;
          v.z = v.z * dd.z;
          v.w = v.w * dd.w;
        }
        *reinterpret_cast<float4*>(Y + j * kLld + 4 * eb) = v;
      }
      if (epi == 0 && gq >= 0) {  // grid policy: activation, derivative, rounding
#pragma unroll 1
        for (int q = 0; q < 16; ++q) {
          const int j = 4 * ob + q / 4;
          if (j < N) grid_act(Y[j * kLld + 4 * eb + q % 4], D[j * kLld + 4 * eb + q % 4], act, gq);
        }
      } else if (epi == 0 && act == 0) {  // one det_tanh per output, four rows at a time
#pragma unroll 1
        for (int o = 0; o < 4; ++o) {
          const int j = 4 * ob + o;
          if (j < N) {
            float4* y = reinterpret_cast<float4*>(Y + j * kLld + 4 * eb);
            float4 v = *y;
            v.x = det_tanh(v.x);
            v.y = det_tanh(v.y);
            v.z = det_tanh(v.z);
            v.w = det_tanh(v.w);
            *y = v;
          }
        }
      } else if (epi == 0 && act == 2) {  // GELU and its derivative, four rows at a time
#pragma unroll 1
        for (int q = 0; q < 16; ++q) {
          const int j = 4 * ob + q / 4;
          if (j < N) {
            float* y = Y + j * kLld + 4 * eb + q % 4;
            det_gelu_grad(*y, *y, D[j * kLld + 4 * eb + q % 4]);
          }
        }
      }
    } else {
#pragma unroll
      for (int o = 0; o < 4; ++o) {
        const int j = 4 * ob + o;
        if (j >= N) continue;
        float v = acc[0][o];
        if (epi == 0) {
          v = __fadd_rn(v, bias[j]);
        } else if (act == 0) {
          const float h = H[j * kLld + eb];
          v = v * (1.0f - h * h);
        } else if (act == 2) {
          v = v * H[j * kLld + eb];
        }
        Y[j * kLld + eb] = v;
      }
      if (epi == 0 && gq >= 0) {
#pragma unroll 1
        for (int o = 0; o < 4; ++o) {
          const int j = 4 * ob + o;
          if (j < N) grid_act(Y[j * kLld + eb], D[j * kLld + eb], act, gq);
        }
      } else if (epi == 0 && (act == 0 || act == 2)) {
#pragma unroll 1
        for (int o = 0; o < 4; ++o) {
          const int j = 4 * ob + o;
          if (j < N) {
            if (act == 0) Y[j * kLld + eb] = det_tanh(Y[j * kLld + eb]);
            else det_gelu_grad(Y[j * kLld + eb], Y[j * kLld + eb], D[j * kLld + eb]);
          }
        }
      }
    }
  }
}

template <int R>
__device__ __forceinline__ void tile_gemm(const float* __restrict__ Wt, int ldw, int K, int N,
                                          const float* X, float* Y, int epi,
                                          const float* __restrict__ bias, int act,
                                          const float* H, float* D, int gq = -1) {
  if ((R / 4) * ((N + 3) / 4) >= kLThreads)
    tile_gemm_t<R, 4>(Wt, ldw, K, N, X, Y, epi, bias, act, H, D, gq);
  else
    tile_gemm_t<R, 1>(Wt, ldw, K, N, X, Y, epi, bias, act, H, D, gq);
}

// Row splits for a reduction over the R rows of a tile shared by `items`
// independent outputs: the largest power of two S <= min(32, R / 4) with
// items * S <= the block size (at least 1).
template <int R>
__device__ __forceinline__ int row_splits(int items) {
  int S = 1;
  while (S * 2 <= 32 && S * 2 <= R / 4 && items * S * 2 <= kLThreads) S *= 2;
  return S;
}

// Lane mask of the S adjacent lanes (S a power of two dividing 32) that share an
// output; their partial sums are combined by a fixed xor butterfly, so the order
// is the same on every run.
__device__ __forceinline__ unsigned split_mask(int S) {
  const unsigned lane = threadIdx.x & 31u;
  return (S == 32) ? 0xFFFFFFFFu : (((1u << S) - 1u) << (lane & ~(unsigned)(S - 1)));
}

// dW[j][k] += sum_r dZ[j][r] H[k][r] for one layer and one tile.  Thread block
// (jb, kb) owns j = jb + p nj4, k = kb + q nk4 (p, q < 4; nj4 = ceil(N/4),
// nk4 = ceil(K/4)): neighbouring lanes read neighbouring features, whose rows sit
// R + 4 floats apart, so a warp's 16-byte row loads are free of bank conflicts.
// Each block is handled by S adjacent lanes, lane sp summing rows
// [sp R / S, (sp + 1) R / S); the S partial sums are combined by a fixed xor
// butterfly, so the order is the same on every run.
template <int R, int S>
__device__ __forceinline__ void dw_blocks(const float* dz, const float* Hl, int N, int K,
                                          float* gW) {
  constexpr int kLld = R + 4, rs = R / S;
  static_assert(rs % 4 == 0 && 32 % S == 0, "row split");
  const int nj4 = (N + 3) / 4, nk4 = (K + 3) / 4, nblk = nj4 * nk4;
  for (int qd = threadIdx.x; qd < nblk * S; qd += blockDim.x) {
    const int blk = qd / S, sp = qd % S;
    const int jb = blk / nk4, kb = blk % nk4;
    float acc[4][4];
#pragma unroll
    for (int p = 0; p < 4; ++p)
#pragma unroll
      for (int q = 0; q < 4; ++q) acc[p][q] = 0.0f;
#pragma unroll 2
    for (int r = sp * rs; r < (sp + 1) * rs; r += 4) {
      float4 dv[4], hv[4];
#pragma unroll
      for (int p = 0; p < 4; ++p) {
        const int j = jb + p * nj4, k = kb + p * nk4;
        dv[p] = j < N ? *reinterpret_cast<const float4*>(dz + j * kLld + r) : make_float4(0, 0, 0, 0);
        hv[p] = k < K ? *reinterpret_cast<const float4*>(Hl + k * kLld + r) : make_float4(0, 0, 0, 0);
      }
#pragma unroll
      for (int p = 0; p < 4; ++p)
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          acc[p][q] = __fmaf_rn(dv[p].x, hv[q].x, acc[p][q]);
          acc[p][q] = __fmaf_rn(dv[p].y, hv[q].y, acc[p][q]);
          acc[p][q] = __fmaf_rn(dv[p].z, hv[q].z, acc[p][q]);
          acc[p][q] = __fmaf_rn(dv[p].w, hv[q].w, acc[p][q]);
        }
    }
    if (S > 1) {
      const unsigned gm = split_mask(S);
#pragma unroll
      for (int d = S / 2; d > 0; d >>= 1)
#pragma unroll
        for (int p = 0; p < 4; ++p)
#pragma unroll
          for (int q = 0; q < 4; ++q) acc[p][q] += __shfl_xor_sync(gm, acc[p][q], d, 32);
    }
    if (sp == 0) {
#pragma unroll
      for (int p = 0; p < 4; ++p) {
        const int j = jb + p * nj4;
        if (j >= N) continue;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int k = kb + q * nk4;
          if (k < K) gW[(size_t)j * K + k] += acc[p][q];
        }
      }
    }
  }
}

struct FusedLossArgs {
  LossArgs a;
  const float* Wt[SIMX_MAX_LAYERS];  // [K][Npad] transposed (forward)
  const float* Wn[SIMX_MAX_LAYERS];  // [N][Kpad] row-major copy (backward), Kpad % 4 == 0
  int npad[SIMX_MAX_LAYERS + 1];     // Npad per layer output (index l + 1)
  int kpad[SIMX_MAX_LAYERS + 1];     // Kpad per layer input (index l)
  int act_off[SIMX_MAX_LAYERS + 2];  // row offset of each layer's activation buffer
  int dact_off[SIMX_MAX_LAYERS + 1]; // row offset of the derivative of layer l's input's activation
                                     // (GELU layers, every hidden layer of a grid policy; -1: none)
  int dz_rows;                       // rows of each dZ buffer
  int poff[SIMX_MAX_LAYERS];         // offset of layer l's dW in the flat gradient
  int n_params;
  int wst_off;                       // float offset of the weight staging buffer (WS kernels)
  float* part;                       // [gridDim.x][n_params]
  double* spart;                     // [gridDim.x][4]
  int64_t ntiles;
};

// One layer's packed weights (n floats, n % 4 == 0, both ends 16-byte aligned) copied
// into shared memory by asynchronous 16-byte copies, all in flight at once; the caller
// runs stage_wait() and a block barrier before reading them.
__device__ __forceinline__ void stage_weights(float* dst, const float* __restrict__ src, int n) {
  for (int i = threadIdx.x; i < n / 4; i += blockDim.x) {
    const unsigned d = static_cast<unsigned>(__cvta_generic_to_shared(dst + 4 * i));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(d), "l"(src + 4 * i)
                 : "memory");
  }
  asm volatile("cp.async.commit_group;\n" ::: "memory");
}

__device__ __forceinline__ void stage_wait() { asm volatile("cp.async.wait_all;\n" ::: "memory"); }

// WS: each layer's weights are staged in shared memory before its product (policies
// whose weights do not stay in L1 beside one block's shared memory); the products read
// the same values in the same order either way.
template <int R, bool WS>
__global__ void __launch_bounds__(kLThreads) k_loss_fused(const __grid_constant__ FusedLossArgs F) {
  constexpr int kLR = R, kLld = R + 4, kLanes = kLThreads / R;  // lanes per row in the head
  extern __shared__ float sm[];
  const LossArgs& a = F.a;
  const int L = a.n_layers;
  float* acts = sm;                                        // all layers' activations
  float* dzA = acts + (size_t)F.act_off[L + 1] * kLld;     // two dZ buffers
  float* dzB = dzA + (size_t)F.dz_rows * kLld;
  float* gacc = dzB + (size_t)F.dz_rows * kLld;            // dW/db accumulators [n_params]
  float* wst = sm + F.wst_off;                             // WS: one layer's weights
  for (int i = threadIdx.x; i < F.n_params; i += blockDim.x) gacc[i] = 0.0f;
  double st_pg = 0.0, st_v = 0.0, st_h = 0.0, st_cf = 0.0;
  const int D = a.dims[0];
  const int A = a.n_actions;
  const int NL = a.dims[L];
  const float inv_n = 1.0f / (float)a.n;
  for (int64_t tile = blockIdx.x; tile < F.ntiles; tile += gridDim.x) {
    const int64_t r0 = tile * kLR;
    __syncthreads();
    if (WS) stage_weights(wst, F.Wt[0], a.dims[0] * F.npad[1]);  // lands during the gather
    // gather X [D][R]: thread (r, dq) reads features dq, dq + kLanes, ... of row r
    // (rows past n are zero and have zero dZ); consecutive threads take consecutive
    // rows, so for a fixed feature the reads are coalesced along the env axis
    float* X = acts + (size_t)F.act_off[0] * kLld;
    {
      const int r = threadIdx.x % kLR, dq = threadIdx.x / kLR;
      const int64_t rr = r0 + r;
      if (rr < a.n) {
        const int64_t row = a.idx ? a.idx[rr] : rr;
        const int64_t t = row / a.E, e = row % a.E;
        const float* src = a.obs + t * D * a.E + e;
        if (a.grid)   // a grid policy's input on its grid
          for (int d = dq; d < D; d += kLanes) X[d * kLld + r] = grid_q(src[(int64_t)d * a.E], a.gx[0]);
        else
          for (int d = dq; d < D; d += kLanes) X[d * kLld + r] = src[(int64_t)d * a.E];
      } else {
        for (int d = dq; d < D; d += kLanes) X[d * kLld + r] = 0.0f;
      }
    }
    __syncthreads();
    for (int l = 0; l < L; ++l) {
      const float* Wf = F.Wt[l];
      if (WS) {
        if (l > 0) stage_weights(wst, F.Wt[l], a.dims[l] * F.npad[l + 1]);
        stage_wait();
        __syncthreads();
        Wf = wst;
      }
      tile_gemm<R>(Wf, F.npad[l + 1], a.dims[l], a.dims[l + 1],
                   acts + (size_t)F.act_off[l] * kLld, acts + (size_t)F.act_off[l + 1] * kLld, 0,
                   a.b[l], a.act[l], nullptr,
                   F.dact_off[l + 1] >= 0 ? acts + (size_t)F.dact_off[l + 1] * kLld : nullptr,
                   (a.grid && l + 1 < L) ? a.gx[l + 1] : -1);
      __syncthreads();
    }
    // loss head: kLanes lanes per row (R rows x kLanes = 256 threads); lane q takes
    // logits i = q, q + kLanes, ... and the row's max / sums are reduced across them.
    // e_i = exp(z_i - max) is kept in the dZ buffer between the passes; p_i = e_i / S.
    const float* Z = acts + (size_t)F.act_off[L] * kLld;
    float* dz = dzA;
    {
      const int r = threadIdx.x / kLanes, q = threadIdx.x % kLanes;
      const unsigned gm = (kLanes == 32 ? 0xFFFFFFFFu : ((1u << kLanes) - 1u)) << (threadIdx.x & (32 - kLanes));
      const int64_t rr = r0 + r;
      if (rr < a.n) {
        const int64_t row = a.idx ? a.idx[rr] : rr;
        const int ac = a.action[row];
        const float ad = a.adv[row];
        float m = -__uint_as_float(0x7F800000u);
        for (int i = q; i < A; i += kLanes) m = fmaxf(m, Z[i * kLld + r]);
#pragma unroll
        for (int d = kLanes / 2; d > 0; d >>= 1) m = fmaxf(m, __shfl_xor_sync(gm, m, d, kLanes));
        float S = 0.0f;
        for (int i = q; i < A; i += kLanes) {
          const float e = det_exp(Z[i * kLld + r] - m);
          dz[i * kLld + r] = e;
          S += e;
        }
#pragma unroll
        for (int d = kLanes / 2; d > 0; d >>= 1) S += __shfl_xor_sync(gm, S, d, kLanes);
        const float lse = m + det_log(S);
        const float invS = 1.0f / S;
        float H = 0.0f;
        for (int i = q; i < A; i += kLanes) {
          const float lp = Z[i * kLld + r] - lse;
          H -= dz[i * kLld + r] * invS * lp;
        }
#pragma unroll
        for (int d = kLanes / 2; d > 0; d >>= 1) H += __shfl_xor_sync(gm, H, d, kLanes);
        const float lpa = Z[ac * kLld + r] - lse;
        float coef, pg;
        if (a.algo == SIMX_ALGO_REINFORCE) {
          coef = ad;
          pg = -ad * lpa;
        } else {
          const float rho = det_exp(lpa - a.logp_old[row]);
          const float s1 = rho * ad;
          const float s2 = fminf(fmaxf(rho, 1.0f - a.clip_eps), 1.0f + a.clip_eps) * ad;
          pg = -fminf(s1, s2);
          coef = (s1 <= s2 ? ad : 0.0f) * rho;
          if (q == 0) st_cf += fabsf(rho - 1.0f) > a.clip_eps ? 1.0 : 0.0;
        }
        for (int i = q; i < A; i += kLanes) {
          const float lp = Z[i * kLld + r] - lse;
          const float p = dz[i * kLld + r] * invS;
          const float onehot = (i == ac) ? 1.0f : 0.0f;
          dz[i * kLld + r] = (-coef * (onehot - p) + a.c_entropy * p * (lp + H)) * inv_n;
        }
        if (q == 0) {
          if (a.has_value) {
            const float dv = Z[A * kLld + r] - a.ret[row];
            st_v += (double)dv * (double)dv;
            dz[A * kLld + r] = 2.0f * a.c_value * dv * inv_n;
          }
          st_pg += pg;
          st_h += H;
        }
      } else {
        for (int i = q; i < NL; i += kLanes) dz[i * kLld + r] = 0.0f;
      }
    }
    __syncthreads();
    // backward
    for (int l = L - 1; l >= 0; --l) {
      const int K = a.dims[l], N = a.dims[l + 1];
      const float* Hl = acts + (size_t)F.act_off[l] * kLld;
      float* gW = gacc + F.poff[l];
      float* gb = gW + (size_t)N * K;
      if (WS && l > 0) stage_weights(wst, F.Wn[l], N * F.kpad[l]);  // lands during dW, db
      // dW += dZ^T H: 4 x 4 blocks of (j, k); the tile's rows are split over S
      // adjacent lanes (S > 1 for thin layers) whose partial sums are combined before
      // the block's accumulator is updated
      {
        const int nblk = ((N + 3) / 4) * ((K + 3) / 4);
        switch (row_splits<R>(nblk)) {
          case 1: dw_blocks<R, 1>(dz, Hl, N, K, gW); break;
          case 2: dw_blocks<R, 2>(dz, Hl, N, K, gW); break;
          case 4: dw_blocks<R, 4>(dz, Hl, N, K, gW); break;
          case 8: dw_blocks<R, 8>(dz, Hl, N, K, gW); break;
          default: dw_blocks<R, (R / 4 < 16 ? R / 4 : 16)>(dz, Hl, N, K, gW); break;  // S <= R / 4
        }
      }
      // db += column sums of dZ, rows split the same way
      {
        const int S = row_splits<R>(N), lg = __ffs(S) - 1, rs = kLR >> lg;
        for (int qd = threadIdx.x; qd < N * S; qd += blockDim.x) {
          const int j = qd >> lg, sp = qd & (S - 1);
          float sacc = 0.0f;
          for (int r = sp * rs; r < (sp + 1) * rs; r += 4) {
            const float4 v = *reinterpret_cast<const float4*>(dz + j * kLld + r);
            sacc += (v.x + v.y) + (v.z + v.w);
          }
          const unsigned gm = split_mask(S);
          for (int d = S / 2; d > 0; d >>= 1) sacc += __shfl_xor_sync(gm, sacc, d, 32);
          if (sp == 0) gb[j] += sacc;
        }
      }
      if (l > 0) {
        float* dzn = (dz == dzA) ? dzB : dzA;
        // dZ_{l-1}[k][r] = sum_j W_l[j][k] dZ_l[j][r] * (1 - H_l[k][r]^2); grid policies
        // (and GELU layers) multiply by the stored derivative instead
        const int pa = a.grid ? 2 : a.act[l - 1];  // activation whose derivative applies
        if (WS) {
          stage_wait();
          __syncthreads();
        }
        tile_gemm<R>(WS ? wst : F.Wn[l], F.kpad[l], N, K, dz, dzn, 1, nullptr, pa,
                     pa == 2 ? acts + (size_t)F.dact_off[l] * kLld : Hl, nullptr);
        __syncthreads();
        dz = dzn;
      } else {
        __syncthreads();
      }
    }
  }
  __syncthreads();
  float* out = F.part + (size_t)blockIdx.x * F.n_params;
  for (int i = threadIdx.x; i < F.n_params; i += blockDim.x) out[i] = gacc[i];
  // fp64 statistics of the rows this block owned (lane 0 of each row group holds them)
  __shared__ double sh[4][kLR];
  if (threadIdx.x % kLanes == 0) {
    sh[0][threadIdx.x / kLanes] = st_pg;
    sh[1][threadIdx.x / kLanes] = st_v;
    sh[2][threadIdx.x / kLanes] = st_h;
    sh[3][threadIdx.x / kLanes] = st_cf;
  }
  __syncthreads();
  if (threadIdx.x < 4) {
    double sum = 0.0;
    for (int r = 0; r < kLR; ++r) sum += sh[threadIdx.x][r];
    F.spart[(size_t)blockIdx.x * 4 + threadIdx.x] = sum;
  }
}

// Transposed (forward) and row-major padded (backward) copies of each W_l; blockIdx.y
// is the layer, so one launch packs them all.
struct PackArgs {
  const float* W[SIMX_MAX_LAYERS];
  float* Wt[SIMX_MAX_LAYERS];
  float* Wn[SIMX_MAX_LAYERS];
  int N[SIMX_MAX_LAYERS], K[SIMX_MAX_LAYERS], npad[SIMX_MAX_LAYERS], kpad[SIMX_MAX_LAYERS];
};

__global__ void k_pack_loss_w(const __grid_constant__ PackArgs P) {
  const int l = blockIdx.y;
  const float* __restrict__ W = P.W[l];
  float* __restrict__ Wt = P.Wt[l];
  float* __restrict__ Wn = P.Wn[l];
  const int N = P.N[l], K = P.K[l], npad = P.npad[l], kpad = P.kpad[l];
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < K * npad) {
    const int k = i / npad, j = i % npad;
    Wt[i] = j < N ? W[(size_t)j * K + k] : 0.0f;
  }
  if (i < N * kpad) {
    const int j = i / kpad, k = i % kpad;
    Wn[i] = k < K ? W[(size_t)j * K + k] : 0.0f;
  }
}

namespace {
struct FusedPlan {
  bool ok;
  int R;
  int npad[SIMX_MAX_LAYERS + 1], kpad[SIMX_MAX_LAYERS + 1], act_off[SIMX_MAX_LAYERS + 2];
  int dact_off[SIMX_MAX_LAYERS + 1];
  int dz_rows, poff[SIMX_MAX_LAYERS], n_params, grid;
  bool stage;
  int wst_off;
  size_t smem, w_off[SIMX_MAX_LAYERS][2], part_off, spart_off, total;
};

int r4(int x) { return (x + 3) / 4 * 4; }

FusedPlan plan_r(const LossArgs& a, int R) {
  FusedPlan p{};
  p.R = R;
  const int ld = R + 4;
  const int L = a.n_layers;
  int rows = 0, maxd = 0;
  for (int l = 0; l <= L; ++l) {
    p.act_off[l] = rows;
    rows += r4(a.dims[l]);
    if (l > 0 && a.dims[l] > maxd) maxd = a.dims[l];
  }
  for (int l = 0; l <= L; ++l) {  // derivative of layer l's input (output of l - 1)
    p.dact_off[l] = -1;
    if (l >= 1 && l < L && (a.act[l - 1] == 2 || a.grid)) {
      p.dact_off[l] = rows;
      rows += r4(a.dims[l]);
    }
  }
  p.act_off[L + 1] = rows;
  p.dz_rows = r4(maxd);
  int P = 0;
  for (int l = 0; l < L; ++l) {
    p.npad[l + 1] = r4(a.dims[l + 1]);
    p.kpad[l] = r4(a.dims[l]);
    p.poff[l] = P;
    P += a.dims[l + 1] * a.dims[l] + a.dims[l + 1];
  }
  p.n_params = P;
  p.smem = ((size_t)rows * ld + (size_t)2 * p.dz_rows * ld + (size_t)P) * sizeof(float);
  p.ok = p.smem <= 200 * 1024;
  const int64_t ntiles = (a.n + R - 1) / R;
  // resident blocks per SM: 128 registers x 256 threads allow two; shared memory may allow fewer
  const int per_sm = p.smem <= 110 * 1024 ? 2 : 1;
  int64_t grid = (int64_t)sm_count() * per_sm;
  if (grid > ntiles) grid = ntiles;
  p.grid = (int)(grid < 1 ? 1 : grid);
  size_t off = 0;
  auto take = [&](size_t b) {
    const size_t o = off;
    off += (b + 255) & ~(size_t)255;
    return o;
  };
  for (int l = 0; l < L; ++l) {
    p.w_off[l][0] = take((size_t)a.dims[l] * p.npad[l + 1] * sizeof(float));
    p.w_off[l][1] = take((size_t)a.dims[l + 1] * p.kpad[l] * sizeof(float));
  }
  p.part_off = take((size_t)p.grid * P * sizeof(float));
  p.spart_off = take((size_t)p.grid * 4 * sizeof(double));
  p.total = off;
  return p;
}

// 64-row tiles when two blocks of them fit in shared memory, else 32-row tiles.  A
// plan with one block per SM stages each layer's weights in shared memory when the
// largest layer fits beside it (then the weights no longer compete with the block's
// shared memory for L1, where they missed on 128-wide layers).
FusedPlan plan(const LossArgs& a) {
  const FusedPlan p64 = plan_r(a, 64);
  if (p64.ok && p64.smem <= 110 * 1024) return p64;
  FusedPlan p = plan_r(a, 32);
  if (!p.ok || p.smem <= 110 * 1024) return p;
  int wmax = 0;
  for (int l = 0; l < a.n_layers; ++l) {
    const int f = a.dims[l] * p.npad[l + 1];
    const int b = a.dims[l + 1] * p.kpad[l];
    wmax = f > wmax ? f : wmax;
    if (l > 0) wmax = b > wmax ? b : wmax;
  }
  const size_t off = (p.smem / 16) * 16 + (p.smem % 16 ? 16 : 0);  // 16-byte aligned
  const size_t with = off + (size_t)wmax * sizeof(float);
  if (with + 2 * 1024 <= 227 * 1024) {  // + the static statistics buffer and a margin
    p.stage = true;
    p.wst_off = (int)(off / sizeof(float));
    p.smem = with;
  }
  return p;
}
}  // namespace

bool loss_fused_fits(const LossArgs& a) { return plan(a).ok; }
size_t loss_fused_workspace(const LossArgs& a) { return plan(a).total; }

cudaError_t launch_loss_fused(const LossArgs& a, void* ws, size_t ws_bytes, cudaStream_t s) {
  const FusedPlan p = plan(a);
  if (!p.ok || ws_bytes < p.total) return cudaErrorInvalidValue;
  char* base = static_cast<char*>(ws);
  FusedLossArgs F{};
  F.a = a;
  PackArgs pk{};
  int nmax = 0;
  for (int l = 0; l < a.n_layers; ++l) {
    float* Wt = reinterpret_cast<float*>(base + p.w_off[l][0]);
    float* Wn = reinterpret_cast<float*>(base + p.w_off[l][1]);
    const int n = a.dims[l] * p.npad[l + 1] > a.dims[l + 1] * p.kpad[l] ? a.dims[l] * p.npad[l + 1]
                                                                         : a.dims[l + 1] * p.kpad[l];
    nmax = n > nmax ? n : nmax;
    pk.W[l] = a.W[l];
    pk.Wt[l] = Wt;
    pk.Wn[l] = Wn;
    pk.N[l] = a.dims[l + 1];
    pk.K[l] = a.dims[l];
    pk.npad[l] = p.npad[l + 1];
    pk.kpad[l] = p.kpad[l];
    F.Wt[l] = Wt;
    F.Wn[l] = Wn;
  }
  k_pack_loss_w<<<dim3((unsigned)((nmax + 255) / 256), (unsigned)a.n_layers), 256, 0, s>>>(pk);
  for (int l = 0; l <= a.n_layers; ++l) {
    F.npad[l] = p.npad[l];
    F.kpad[l] = p.kpad[l];
    F.act_off[l] = p.act_off[l];
  }
  F.act_off[a.n_layers + 1] = p.act_off[a.n_layers + 1];
  for (int l = 0; l <= a.n_layers; ++l) F.dact_off[l] = p.dact_off[l];
  F.dz_rows = p.dz_rows;
  for (int l = 0; l < a.n_layers; ++l) F.poff[l] = p.poff[l];
  F.n_params = p.n_params;
  F.wst_off = p.wst_off;
  F.part = reinterpret_cast<float*>(base + p.part_off);
  F.spart = reinterpret_cast<double*>(base + p.spart_off);
  F.ntiles = (a.n + p.R - 1) / p.R;
  auto k = p.R == 64 ? k_loss_fused<64, false>
                     : (p.stage ? k_loss_fused<32, true> : k_loss_fused<32, false>);
  cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem);
  k<<<p.grid, kLThreads, p.smem, s>>>(F);
  launch_loss_reduce(F.part, p.grid, p.n_params, F.spart, a, s);
  count_launches(2);
  return cudaGetLastError();
}

// Sums the per-block partial gradients (in block order) into a.grad and the per-block
// fp64 statistics into a.stats.
void launch_loss_reduce(const float* part, int nb, int n_params, const double* spart,
                        const LossArgs& a, cudaStream_t s) {
  launch_loss_reduce_n(part, nb, n_params, spart, nb, a, s);
}

// The block reduction and the statistics in one launch.  Blocks 0 .. nr - 1 sum the
// gradient partials, element i over blocks 0, 1, ... in order.  The last block sums the
// statistics, one warp per statistic: lane l takes blocks l, l + 32, ... in order, then a
// fixed butterfly combines the lanes (the same order on every run).  Launched with
// programmatic stream serialization: it waits for the kernel before it
// (griddepcontrol.wait) before reading the partials, so its launch overlaps that kernel's
// tail.
__global__ void __launch_bounds__(256) k_reduce_all(const float* __restrict__ part, int nb, int P,
                                                    float* __restrict__ out, const double* __restrict__ sp,
                                                    int nbs, int64_t n, int has_value, float cv,
                                                    float ce, float* __restrict__ stats) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  if ((int)blockIdx.x + 1 < (int)gridDim.x) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= P) return;
    float s = 0.0f;
    for (int b = 0; b < nb; ++b) s += part[(size_t)b * P + i];
    out[i] = s;
    return;
  }
  __shared__ double sh[4];
  if (threadIdx.x >= 128) return;
  const int q = threadIdx.x / 32, lane = threadIdx.x % 32;
  double acc = 0.0;
  for (int b = lane; b < nbs; b += 32) acc += sp[(size_t)b * 4 + q];
  for (int d = 16; d > 0; d /= 2) acc += __shfl_xor_sync(0xffffffffu, acc, d);
  if (lane == 0) sh[q] = acc;
  asm volatile("bar.sync 1, 128;" ::: "memory");
  if (threadIdx.x != 0) return;
  const double s4[4] = {sh[0], sh[1], sh[2], sh[3]};
  const double pg = s4[0] / (double)n, v = s4[1] / (double)n, H = s4[2] / (double)n;
  stats[0] = (float)(pg + (has_value ? (double)cv * v : 0.0) - (double)ce * H);
  stats[1] = (float)pg;
  stats[2] = (float)v;
  stats[3] = (float)H;
  stats[4] = (float)(s4[3] / (double)n);
}

void launch_loss_reduce_n(const float* part, int nb, int n_params, const double* spart, int nbs,
                          const LossArgs& a, cudaStream_t s) {
  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3((unsigned)((n_params + 255) / 256 + 1));
  lc.blockDim = dim3(256);
  lc.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  lc.attrs = at;
  lc.numAttrs = 1;
  cudaLaunchKernelEx(&lc, k_reduce_all, part, nb, n_params, a.grad, spart, nbs, a.n, a.has_value,
                     a.c_value, a.c_entropy, a.stats);
  count_launches(1);
}

}  // namespace simx
