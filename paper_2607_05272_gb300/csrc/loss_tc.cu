// loss_tc.cu — REINFORCE / PPO loss gradient (Sec. 4.3) on the tensor cores
// (tcgen05.mma kind::tf32: TF32 inputs rounded to nearest, FP32 accumulation in
// tensor memory), for policies whose per-tile operands fit in one SM's shared memory.
//
// One persistent CTA of 512 threads per SM walks tiles of 128 minibatch rows.  Every
// matrix product of the forward and backward pass is one MMA chain with M = 128:
//   forward   Z_l  = [H_l, 1] [W_l, b_l]^T          (rows x outputs; the bias rides on a
//                                                   ones column of the activations)
//   weights   dW_l += G_l^T H_l                      (outputs x inputs, K = the tile's rows)
//   biases    db_l += G_l^T 1                        (FP32 sums on the CUDA cores, beside
//                                                   the weight products)
//   inputs    dH_l  = G_l W_l                        (rows x inputs)
// where G_l is dL/d(pre-activation of layer l).  dW_l and db_l stay in tensor memory for
// all of the CTA's tiles and are read out once at the end.  Threads do the elementwise
// work between the products: tanh, the loss head (log-softmax, rho, clipped surrogate,
// entropy, value residual), and G_{l-1} = dH_l * (1 - H_l^2), reading accumulators with
// tcgen05.ld (thread = TMEM lane = row; the 4 warps that share a lane quarter split the
// columns) and writing the next operands to shared memory.
//
// The first layer's product is split TF32 ("3-pass": x = x_hi + x_lo, each part TF32,
// x_hi w_hi + x_hi w_lo + x_lo w_hi), because raw observations reach magnitudes in the
// hundreds: a TF32 error there moves saturated tanh units' derivatives by percents.
// Later layers see tanh outputs and take one TF32 pass.  Activations kept for the
// backward pass are stored in FP32 (the derivative 1 - h^2 is taken from them).
//
// TF32 operands require both MMA operands K-major, so an operand used with K = rows
// (H_l and G_l in the weight products) is also kept row-contiguous ("transposed" below).
// Operands use the no-swizzle canonical layout: 8 x 16-byte core matrices.  In the
// transposed buffers consecutive 4-row core matrices are 144 bytes apart (16 bytes of
// padding) so that a warp's per-row scalar stores and loads hit 32 distinct banks.
//
// Results are per-CTA partial gradients and fp64 statistics, summed in CTA order by the
// same reduction kernels as the FP32 path: deterministic for a given launch.  Accuracy
// is that of TF32 inputs (about 1e-3 relative per product); the FP32 SIMT path
// (loss_fused.cu) is the exact alternative.
#include <cstdint>

#include "devmath.cuh"
#include "kernels.h"

namespace simx {
namespace tcl {

constexpr int kR = 128;                // rows per tile (MMA M)
constexpr int kThreads = 512;          // 16 warps: 4 per TMEM lane quarter
constexpr int kRowLd = 144;            // bytes between 4-row core matrices of transposed operands
constexpr int kTGroup = 32 * kRowLd;   // bytes per 8-feature group of a transposed operand
constexpr int kMaxNL = 32;             // widest last layer (logits + value) handled by the head
constexpr long long kWaitCycles = 2000000000LL;  // bound on any MMA wait (about 1 s)

struct Plan {
  int L;
  int K[SIMX_MAX_LAYERS], N[SIMX_MAX_LAYERS];
  int C[SIMX_MAX_LAYERS];    // forward operand width: K + 1 (ones column) rounded up to 8
  int Np[SIMX_MAX_LAYERS];   // forward MMA N: outputs rounded up to 16
  int Kp[SIMX_MAX_LAYERS];   // inputs rounded up to 16 (dW and dH MMA N)
  int Gw[SIMX_MAX_LAYERS];   // row-major G_l width: outputs rounded up to 8 (dH MMA K)
  // shared memory byte offsets
  int o_dat, o_hr, o_ones, o_ht[SIMX_MAX_LAYERS], o_wa[SIMX_MAX_LAYERS], o_wt[SIMX_MAX_LAYERS];
  int o_wl0;                 // low TF32 part of the first layer's [W_0, b_0]
  int o_misc, smem;
  // tensor memory columns
  int t_work, t_dw[SIMX_MAX_LAYERS], t_db[SIMX_MAX_LAYERS], tcols;
  int poff[SIMX_MAX_LAYERS], n_params;
  bool ok;
};

struct Args {
  LossArgs a;
  Plan p;
  float* part;     // [gridDim.x][n_params]
  double* spart;   // [gridDim.x][4]
  int64_t ntiles;
};

__device__ __forceinline__ uint32_t su32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

// TF32 value of x, rounded to nearest (ties away), as the fp32 bit pattern the MMA reads.
__device__ __forceinline__ float to_tf32(float x) {
  uint32_t u;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(u) : "f"(x));
  return __uint_as_float(u);
}

// Shared-memory matrix descriptor, no swizzle: start, leading (K-direction) and stride
// (M/N-direction) byte offsets between core matrices; bits 46-48 hold the fixed 0b001.
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
         ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | ((uint64_t)1 << 46);
}

// Instruction descriptor for kind::tf32, FP32 accumulator, both operands K-major.
__device__ __forceinline__ uint32_t idesc(int M, int N) {
  return (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void mma(uint32_t d, uint64_t ad, uint64_t bd, uint32_t id, uint32_t acc) {
  asm volatile(
      "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n}" ::"r"(d),
      "l"(ad), "l"(bd), "r"(id), "r"(acc)
      : "memory");
}

__device__ __forceinline__ void commit(uint64_t* mbar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   su32(mbar))
               : "memory");
}

// Waits for the phase of the MMA barrier, at most kWaitCycles; false on timeout.
__device__ __forceinline__ bool wait_phase(uint64_t* mbar, uint32_t phase) {
  const long long t0 = clock64();
  for (;;) {
    uint32_t done;
    asm volatile(
        "{\n.reg .pred p;\nmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        "selp.u32 %0, 1, 0, p;\n}"
        : "=r"(done)
        : "r"(su32(mbar)), "r"(phase)
        : "memory");
    if (done) return true;
    if (clock64() - t0 > kWaitCycles) return false;
  }
}

__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// Four consecutive accumulator columns of this thread's TMEM lane.
__device__ __forceinline__ float4 tm_ld4(uint32_t taddr) {
  uint32_t a, b, c, d;
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0, %1, %2, %3}, [%4];"
               : "=r"(a), "=r"(b), "=r"(c), "=r"(d)
               : "r"(taddr)
               : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
  return make_float4(__uint_as_float(a), __uint_as_float(b), __uint_as_float(c), __uint_as_float(d));
}

// tanh(x) = 1 - 2 / (e^{2x} + 1) with the hardware exponential and reciprocal: absolute
// error near 1e-7 (far below the TF32 rounding that follows), exactly +-1 once e^{2x}
// overflows or underflows.
__device__ __forceinline__ float tanh_fast(float x) {
  return 1.0f - __fdividef(2.0f, __expf(2.0f * x) + 1.0f);
}

// Issue a 4-column load without waiting; tm_wait() then completes every load issued,
// and reg_fence() keeps the compiler from using the registers before that point.
__device__ __forceinline__ void tm_ld4_nw(uint32_t taddr, uint32_t (&u)[4]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0, %1, %2, %3}, [%4];"
               : "=r"(u[0]), "=r"(u[1]), "=r"(u[2]), "=r"(u[3])
               : "r"(taddr)
               : "memory");
}
__device__ __forceinline__ void tm_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void reg_fence(uint32_t (&u)[4]) {
  asm volatile("" : "+r"(u[0]), "+r"(u[1]), "+r"(u[2]), "+r"(u[3]));
}

// Byte offset of element (r, c) in a row-major operand of width W (core matrices of
// 8 rows x 4 columns, row-group major).
__device__ __forceinline__ uint32_t rm_off(int r, int c, int W) {
  return (uint32_t)(((r >> 3) * (W >> 2) + (c >> 2)) * 128 + (r & 7) * 16 + (c & 3) * 4);
}
// Byte offset of element (feature f, row r) in a transposed (row-contiguous) operand.
__device__ __forceinline__ uint32_t tr_off(int f, int r) {
  return (uint32_t)((f >> 3) * kTGroup + (r >> 2) * kRowLd + (f & 7) * 16 + (r & 3) * 4);
}

__device__ __forceinline__ void put4(unsigned char* base, uint32_t off, float4 v) {
  *reinterpret_cast<float4*>(base + off) = v;
}
__device__ __forceinline__ void put1(unsigned char* base, uint32_t off, float v) {
  *reinterpret_cast<float*>(base + off) = v;
}
__device__ __forceinline__ float get1(const unsigned char* base, uint32_t off) {
  return *reinterpret_cast<const float*>(base + off);
}

__global__ void __launch_bounds__(kThreads, 1) k_loss_tc(const __grid_constant__ Args A) {
  extern __shared__ __align__(1024) unsigned char sm[];
  const LossArgs& a = A.a;
  const Plan& P = A.p;
  const int L = P.L;
  uint64_t* mbar = reinterpret_cast<uint64_t*>(sm + P.o_misc);
  uint32_t* tbase = reinterpret_cast<uint32_t*>(sm + P.o_misc + 8);
  int* abort_flag = reinterpret_cast<int*>(sm + P.o_misc + 12);
  __shared__ double sh_st[4][kR];

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int quarter = warp & 3;        // TMEM lane quarter = rows 32 quarter .. + 31
  const int cq = warp >> 2;            // column share: blocks of 4 columns cb with cb % 4 == cq
  const int r = 32 * quarter + lane;   // this thread's tile row (= TMEM lane)

  // constant operands: weights with the bias column, transposed weights, the ones block,
  // zero padding of the transposed activations (none of it changes between tiles)
  for (int l = 0; l < L; ++l) {
    const int K = P.K[l], N = P.N[l], C = P.C[l], Np = P.Np[l];
    const float* W = a.W[l];
    const float* b = a.b[l];
    for (int i = tid; i < Np * C; i += kThreads) {
      const int j = i / C, c = i % C;
      float v = 0.0f;
      if (j < N) v = c < K ? W[(size_t)j * K + c] : (c == K ? b[j] : 0.0f);
      const float hi = to_tf32(v);
      put1(sm + P.o_wa[l], rm_off(j, c, C), hi);
      if (l == 0) put1(sm + P.o_wl0, rm_off(j, c, C), to_tf32(v - hi));
    }
    if (l > 0) {
      const int Kp = P.Kp[l], Gw = P.Gw[l];
      for (int i = tid; i < Kp * Gw; i += kThreads) {
        const int k = i / Gw, j = i % Gw;
        const float v = (k < K && j < N) ? W[(size_t)j * K + k] : 0.0f;
        put1(sm + P.o_wt[l], rm_off(k, j, Gw), to_tf32(v));
      }
    }
    for (int i = tid; i < (P.Kp[l] - K) * kR; i += kThreads)
      put1(sm + P.o_ht[l], tr_off(K + i / kR, i % kR), 0.0f);
  }
  for (int i = tid; i < 16 * kR; i += kThreads) put1(sm + P.o_ones, tr_off(i / kR, i % kR), 1.0f);
  if (tid == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(su32(mbar)) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    *abort_flag = 0;
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tbase)),
                 "r"(P.tcols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  fence_async_smem();
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *tbase;
  const uint32_t tlane = tmem + ((uint32_t)(32 * quarter) << 16);  // this warp's lane quarter

  double st_pg = 0.0, st_v = 0.0, st_h = 0.0, st_cf = 0.0;
  const int D = P.K[0];
  const int NA = a.n_actions;
  const float inv_n = 1.0f / (float)a.n;
  uint32_t phase = 0;
  bool first = true;
  unsigned char* hr = sm + P.o_hr;
  unsigned char* dat = sm + P.o_dat;
  // db_l of output tid, summed over the CTA's tiles (threads below each layer's width)
  float dbacc[SIMX_MAX_LAYERS];
#pragma unroll
  for (int l = 0; l < SIMX_MAX_LAYERS; ++l) dbacc[l] = 0.0f;

  // One synchronisation point between a stage's shared-memory / TMEM producers and the
  // MMAs that read them; returns false when any thread saw an MMA wait time out.
  auto stage_sync = [&]() -> bool {
    fence_async_smem();
    fence_before();
    __syncthreads();
    fence_after();
    return *abort_flag == 0;
  };
  auto wait_mma = [&]() {
    if (!wait_phase(mbar, phase)) atomicOr(abort_flag, 1);
    phase ^= 1u;
    fence_after();
  };

  // Per-row inputs of the next tile are loaded into registers while the current tile
  // is computed: observation blocks cb = cq, cq + 4 (the plan keeps C_0 <= 32), and for
  // the head thread (cq == 0) the action, advantage, old log-probability and target.
  float px[8];
  int pact = 0;
  float padv = 0.0f, plpo = 0.0f, pret = 0.0f;
  bool plive = false;
  auto prefetch = [&](int64_t tile) {
    const int64_t rr = tile * kR + r;
    plive = tile < A.ntiles && rr < a.n;
    int64_t row = 0;
    if (plive) row = a.idx ? a.idx[rr] : rr;
    const int64_t t = row / a.E, e = row % a.E;
    const float* src = a.obs + t * D * a.E + e;
#pragma unroll
    for (int j = 0; j < 2; ++j)
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int f = 4 * (cq + 4 * j) + i;
        px[4 * j + i] = (plive && f < D) ? src[(int64_t)f * a.E] : 0.0f;
      }
    if (cq == 0 && plive) {
      pact = a.action[row];
      padv = a.adv[row];
      plpo = a.algo == SIMX_ALGO_PPO ? a.logp_old[row] : 0.0f;
      pret = a.has_value ? a.ret[row] : 0.0f;
    }
  };
  prefetch(blockIdx.x);
  for (int64_t tile = blockIdx.x; tile < A.ntiles; tile += gridDim.x) {
    const bool live = plive;
    const int ac_row = pact;
    const float adv_row = padv, lpo_row = plpo, ret_row = pret;
    // X (rows past n are zero; their loss gradient is zero) with the ones column
    {
      const int C = P.C[0];
      unsigned char* hr_lo = hr + kR * C * 4;  // x_lo follows x_hi in the row-major buffer
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int cb = cq + 4 * j;
        if (cb < C / 4) {
          float hi[4], lo[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int f = 4 * cb + i;
            const float x = f < D ? px[4 * j + i] : (f == D ? 1.0f : 0.0f);
            hi[i] = to_tf32(x);
            lo[i] = to_tf32(x - hi[i]);
            if (f < D) put1(sm + P.o_ht[0], tr_off(f, r), hi[i]);
          }
          put4(hr, rm_off(r, 4 * cb, C), make_float4(hi[0], hi[1], hi[2], hi[3]));
          put4(hr_lo, rm_off(r, 4 * cb, C), make_float4(lo[0], lo[1], lo[2], lo[3]));
        }
      }
    }
    prefetch(tile + gridDim.x);
    if (!stage_sync()) break;
    // forward
    for (int l = 0; l < L; ++l) {
      const int C = P.C[l], Np = P.Np[l], N = P.N[l];
      if (tid == kThreads - 32) {
        // descriptors advance by 256 bytes (16 in the address field) per K step of 8
        const uint32_t id = idesc(kR, Np);
        const uint32_t sbo = (C / 4) * 128;
        uint64_t xh = sdesc(su32(hr), 128, sbo), wh = sdesc(su32(sm + P.o_wa[l]), 128, sbo);
        uint64_t wl = sdesc(su32(sm + P.o_wl0), 128, sbo), xl = sdesc(su32(hr) + kR * C * 4, 128, sbo);
        const uint32_t d = tmem + P.t_work;
        for (int ks = 0; ks < C / 8; ++ks) {
          mma(d, xh, wh, id, ks > 0);
          if (l == 0) {  // split TF32: + x_hi w_lo + x_lo w_hi
            mma(d, xh, wl, id, 1u);
            mma(d, xl, wh, id, 1u);
          }
          xh += 16;
          wh += 16;
          wl += 16;
          xl += 16;
        }
        commit(mbar);
      }
      wait_mma();
      if (l + 1 < L) {
        // H_{l+1} = tanh(Z_l): row-major with its ones column, and transposed; the
        // thread's column blocks cb = cq + 4 j are loaded four at a time, one wait each
        const int Cn = P.C[l + 1];
        for (int j0 = 0; cq + 4 * j0 < Cn / 4; j0 += 4) {
          uint32_t u[4][4];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int cb = cq + 4 * (j0 + j);
            if (cb < Cn / 4 && 4 * cb < N) tm_ld4_nw(tlane + P.t_work + 4 * cb, u[j]);
            else u[j][0] = u[j][1] = u[j][2] = u[j][3] = 0u;
          }
          tm_wait();
#pragma unroll
          for (int j = 0; j < 4; ++j) reg_fence(u[j]);
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int cb = cq + 4 * (j0 + j);
            if (cb >= Cn / 4) break;
            float v[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const int f = 4 * cb + i;
              if (f < N) {
                const float h = tanh_fast(__uint_as_float(u[j][i]));
                put1(sm + P.o_ht[l + 1], tr_off(f, r), h);  // FP32 (the MMA reads its TF32 part)
                v[i] = to_tf32(h);
              } else {
                v[i] = f == N ? 1.0f : 0.0f;
              }
            }
            put4(hr, rm_off(r, 4 * cb, Cn), make_float4(v[0], v[1], v[2], v[3]));
          }
        }
      } else if (cq == 0) {
        // loss head for row r: G_L = dL/dZ (logits, then the value row)
        float z[kMaxNL];
        {
          uint32_t u[kMaxNL / 4][4];
#pragma unroll
          for (int cb = 0; cb < kMaxNL / 4; ++cb) {
            if (4 * cb < N) tm_ld4_nw(tlane + P.t_work + 4 * cb, u[cb]);
            else u[cb][0] = u[cb][1] = u[cb][2] = u[cb][3] = 0u;
          }
          tm_wait();
#pragma unroll
          for (int cb = 0; cb < kMaxNL / 4; ++cb) {
            reg_fence(u[cb]);
#pragma unroll
            for (int i = 0; i < 4; ++i) z[4 * cb + i] = __uint_as_float(u[cb][i]);
          }
        }
        float g[kMaxNL];
#pragma unroll
        for (int i = 0; i < kMaxNL; ++i) g[i] = 0.0f;
        if (live) {
          const int ac = ac_row;
          const float ad = adv_row;
          float m = -__uint_as_float(0x7F800000u);
#pragma unroll
          for (int i = 0; i < kMaxNL; ++i)
            if (i < NA) m = fmaxf(m, z[i]);
          float S = 0.0f;
#pragma unroll
          for (int i = 0; i < kMaxNL; ++i)
            if (i < NA) {
              g[i] = __expf(z[i] - m);
              S += g[i];
            }
          const float lse = m + __logf(S);
          const float invS = __fdividef(1.0f, S);
          float H = 0.0f, lpa = 0.0f;
#pragma unroll
          for (int i = 0; i < kMaxNL; ++i)
            if (i < NA) {
              const float lp = z[i] - lse;
              H -= g[i] * invS * lp;
              if (i == ac) lpa = lp;
            }
          float coef, pg;
          if (a.algo == SIMX_ALGO_REINFORCE) {
            coef = ad;
            pg = -ad * lpa;
          } else {
            const float rho = __expf(lpa - lpo_row);
            const float s1 = rho * ad;
            const float s2 = fminf(fmaxf(rho, 1.0f - a.clip_eps), 1.0f + a.clip_eps) * ad;
            pg = -fminf(s1, s2);
            coef = (s1 <= s2 ? ad : 0.0f) * rho;
            st_cf += fabsf(rho - 1.0f) > a.clip_eps ? 1.0 : 0.0;
          }
#pragma unroll
          for (int i = 0; i < kMaxNL; ++i)
            if (i < NA) {
              const float lp = z[i] - lse;
              const float p = g[i] * invS;
              const float onehot = (i == ac) ? 1.0f : 0.0f;
              g[i] = (-coef * (onehot - p) + a.c_entropy * p * (lp + H)) * inv_n;
            }
          if (a.has_value) {
            float zv = 0.0f;
#pragma unroll
            for (int i = 0; i < kMaxNL; ++i)
              if (i == NA) zv = z[i];
            const float dv = zv - ret_row;
            st_v += (double)dv * (double)dv;
#pragma unroll
            for (int i = 0; i < kMaxNL; ++i)
              if (i == NA) g[i] = 2.0f * a.c_value * dv * inv_n;
          }
          st_pg += pg;
          st_h += H;
        }
        const int Gw = P.Gw[l];
#pragma unroll
        for (int cb = 0; cb < kMaxNL / 4; ++cb) {
          if (4 * cb < Gw) {
            float4 v = make_float4(to_tf32(g[4 * cb]), to_tf32(g[4 * cb + 1]), to_tf32(g[4 * cb + 2]),
                                   to_tf32(g[4 * cb + 3]));
            put4(hr, rm_off(r, 4 * cb, Gw), v);
#pragma unroll
            for (int i = 0; i < 4; ++i)
              if (4 * cb + i < N) put1(dat, tr_off(4 * cb + i, r), (&v.x)[i]);
          }
        }
      }
      if (!stage_sync()) break;
    }
    if (*abort_flag) break;
    // backward
    for (int l = L - 1; l >= 0; --l) {
      const int K = P.K[l], Gw = P.Gw[l], Kp = P.Kp[l];
      if (tid == kThreads - 32) {
        // transposed operands advance 2 x 144 bytes (18 in the address field) per K step
        const uint32_t acc0 = first ? 0u : 1u;
        const uint32_t idw = idesc(kR, Kp);
        uint64_t ad = sdesc(su32(dat), kRowLd, kTGroup);
        uint64_t hd = sdesc(su32(sm + P.o_ht[l]), kRowLd, kTGroup);
        const uint32_t dw = tmem + P.t_dw[l];
        for (int ks = 0; ks < kR / 8; ++ks) {
          const uint32_t acc = ks > 0 ? 1u : acc0;
          mma(dw, ad, hd, idw, acc);
          ad += (2 * kRowLd) >> 4;
          hd += (2 * kRowLd) >> 4;
        }
        if (l > 0) {
          const uint32_t idh = idesc(kR, Kp);
          uint64_t gd = sdesc(su32(hr), 128, (Gw / 4) * 128);
          uint64_t wd = sdesc(su32(sm + P.o_wt[l]), 128, (Gw / 4) * 128);
          for (int ks = 0; ks < Gw / 8; ++ks) {
            mma(tmem + P.t_work, gd, wd, idh, ks > 0);
            gd += 16;
            wd += 16;
          }
        }
        commit(mbar);
      }
      if (tid < P.N[l]) {
        // db_l of output tid over the tile's rows, from the transposed G_l the weight
        // products read (the same TF32 values), rows in order
        const unsigned char* col = dat + (tid >> 3) * kTGroup + (tid & 7) * 16;
        float sacc = 0.0f;
#pragma unroll 4
        for (int q = 0; q < kR / 4; ++q) {
          const float4 v = *reinterpret_cast<const float4*>(col + q * kRowLd);
          sacc = __fadd_rn(__fadd_rn(__fadd_rn(__fadd_rn(sacc, v.x), v.y), v.z), v.w);
        }
        dbacc[l] = __fadd_rn(dbacc[l], sacc);
      }
      wait_mma();
      if (l > 0) {
        // G_{l-1} = dH_l * (1 - H_l^2), row-major (width Gw_{l-1}) and transposed
        const int Gn = P.Gw[l - 1];
        (void)Kp;
        for (int j0 = 0; cq + 4 * j0 < Gn / 4; j0 += 4) {
          uint32_t u[4][4];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int cb = cq + 4 * (j0 + j);
            if (cb < Gn / 4 && 4 * cb < K) tm_ld4_nw(tlane + P.t_work + 4 * cb, u[j]);
            else u[j][0] = u[j][1] = u[j][2] = u[j][3] = 0u;
          }
          tm_wait();
#pragma unroll
          for (int j = 0; j < 4; ++j) reg_fence(u[j]);
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int cb = cq + 4 * (j0 + j);
            if (cb >= Gn / 4) break;
            float v[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const int f = 4 * cb + i;
              if (f < K) {
                const float h = get1(sm + P.o_ht[l], tr_off(f, r));
                v[i] = to_tf32(__uint_as_float(u[j][i]) * (1.0f - h * h));
                put1(dat, tr_off(f, r), v[i]);
              } else {
                v[i] = 0.0f;
              }
            }
            put4(hr, rm_off(r, 4 * cb, Gn), make_float4(v[0], v[1], v[2], v[3]));
          }
        }
      }
      if (!stage_sync()) break;
    }
    if (*abort_flag) break;
    first = false;
  }

  // read out dW_l (lane j = output, column k = input) and db_l (every column holds the sum)
  float* out = A.part + (size_t)blockIdx.x * P.n_params;
  const bool ok = *abort_flag == 0;
  if (ok && !first) {
    for (int l = 0; l < L; ++l) {
      const int K = P.K[l], N = P.N[l];
      float* gW = out + P.poff[l];
      for (int cb = cq; cb < P.Kp[l] / 4; cb += 4) {
        const float4 v = tm_ld4(tlane + P.t_dw[l] + 4 * cb);
        if (r < N) {
#pragma unroll
          for (int i = 0; i < 4; ++i)
            if (4 * cb + i < K) gW[(size_t)r * K + 4 * cb + i] = (&v.x)[i];
        }
      }
      if (tid < N) gW[(size_t)N * K + tid] = dbacc[l];
    }
  } else {
    for (int i = tid; i < P.n_params; i += kThreads) out[i] = 0.0f;
  }
  // fp64 statistics of the rows this CTA owned (the cq == 0 thread of each row)
  if (cq == 0) {
    sh_st[0][r] = st_pg;
    sh_st[1][r] = st_v;
    sh_st[2][r] = st_h;
    sh_st[3][r] = st_cf;
  }
  fence_before();
  __syncthreads();
  if (tid < 4) {
    double sum = 0.0;
    for (int i = 0; i < kR; ++i) sum += sh_st[tid][i];
    A.spart[(size_t)blockIdx.x * 4 + tid] = ok ? sum : __longlong_as_double(0x7FF8000000000000LL);
  }
  if (warp == 0) {
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(P.tcols)
                 : "memory");
  }
}

int r8(int x) { return (x + 7) / 8 * 8; }
int r16(int x) { return (x + 15) / 16 * 16; }

Plan plan(const LossArgs& a) {
  Plan p{};
  p.ok = false;
  const int L = a.n_layers;
  if (L < 1 || L > SIMX_MAX_LAYERS) return p;
  for (int l = 0; l + 1 < L; ++l)
    if (a.act[l] != 0) return p;  // the hidden layers' epilogues here are tanh only
  p.L = L;
  int P = 0, hr_w = 0, maxN = 0;
  for (int l = 0; l < L; ++l) {
    const int K = a.dims[l], N = a.dims[l + 1];
    p.K[l] = K;
    p.N[l] = N;
    p.C[l] = r8(K + 1);
    p.Np[l] = r16(N);
    p.Kp[l] = r16(K);
    p.Gw[l] = r8(N);
    p.poff[l] = P;
    P += N * K + N;
    if (N > 128 || p.Np[l] > 256 || p.Kp[l] > 256) return p;  // dW rows are MMA M = 128
    hr_w = hr_w > (l == 0 ? 2 * p.C[l] : p.C[l]) ? hr_w : (l == 0 ? 2 * p.C[l] : p.C[l]);
    hr_w = hr_w > p.Gw[l] ? hr_w : p.Gw[l];
    maxN = maxN > N ? maxN : N;
  }
  if (a.dims[L] > kMaxNL || p.C[0] > 32) return p;  // head registers; prefetch of 2 blocks
  p.n_params = P;
  // shared memory: the transposed G block first, because its M = 128 reads run past its
  // own rows into the following buffers (those result rows are never read)
  int off = 0;
  p.o_dat = off;
  off += (r8(maxN) / 8) * kTGroup;
  p.o_hr = off;
  off += kR * hr_w * 4;
  p.o_ones = off;
  off += 2 * kTGroup;
  for (int l = 0; l < L; ++l) {
    p.o_ht[l] = off;
    off += (p.Kp[l] / 8) * kTGroup;
  }
  p.o_wl0 = off;
  off += p.Np[0] * p.C[0] * 4;
  for (int l = 0; l < L; ++l) {
    p.o_wa[l] = off;
    off += p.Np[l] * p.C[l] * 4;
    p.o_wt[l] = off;
    if (l > 0) off += p.Kp[l] * p.Gw[l] * 4;
  }
  p.o_misc = off;
  off += 16;
  p.smem = off;
  if (p.o_dat + 16 * kTGroup > p.smem) return p;  // the M = 128 read of G^T must stay inside
  if (p.smem + 4 * kR * 8 > 227 * 1024) return p;  // + static statistics buffer
  // tensor memory: the working accumulator, then every layer's dW and db
  int cols = 0;
  for (int l = 0; l < L; ++l) {
    cols = cols > p.Np[l] ? cols : p.Np[l];
    cols = cols > p.Kp[l] ? cols : p.Kp[l];
  }
  p.t_work = 0;
  for (int l = 0; l < L; ++l) {
    p.t_dw[l] = cols;
    cols += p.Kp[l];
    p.t_db[l] = cols;
    cols += 16;
  }
  int tc = 32;
  while (tc < cols) tc *= 2;
  if (tc > 512) return p;
  p.tcols = tc;
  p.ok = true;
  return p;
}

struct Ws {
  size_t part, spart, total;
  int grid;
};

Ws ws_layout(const LossArgs& a, const Plan& p) {
  Ws w{};
  const int64_t ntiles = (a.n + kR - 1) / kR;
  const int64_t sms = sm_count();
  w.grid = (int)(ntiles < sms ? ntiles : sms);
  if (w.grid < 1) w.grid = 1;
  w.part = 0;
  w.spart = ((size_t)w.grid * p.n_params * sizeof(float) + 255) & ~(size_t)255;
  w.total = w.spart + (size_t)w.grid * 4 * sizeof(double);
  return w;
}

}  // namespace tcl

bool loss_tc_fits(const LossArgs& a) { return tcl::plan(a).ok; }

size_t loss_tc_workspace(const LossArgs& a) {
  const tcl::Plan p = tcl::plan(a);
  return p.ok ? tcl::ws_layout(a, p).total : 0;
}

cudaError_t launch_loss_tc(const LossArgs& a, void* ws, size_t ws_bytes, cudaStream_t s) {
  const tcl::Plan p = tcl::plan(a);
  if (!p.ok) return cudaErrorInvalidValue;
  const tcl::Ws w = tcl::ws_layout(a, p);
  if (ws_bytes < w.total) return cudaErrorInvalidValue;
  char* base = static_cast<char*>(ws);
  tcl::Args A{};
  A.a = a;
  A.p = p;
  A.part = reinterpret_cast<float*>(base + w.part);
  A.spart = reinterpret_cast<double*>(base + w.spart);
  A.ntiles = (a.n + tcl::kR - 1) / tcl::kR;
  cudaFuncSetAttribute(tcl::k_loss_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, p.smem);
  tcl::k_loss_tc<<<w.grid, tcl::kThreads, p.smem, s>>>(A);
  launch_loss_reduce(A.part, w.grid, p.n_params, A.spart, a, s);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace simx
