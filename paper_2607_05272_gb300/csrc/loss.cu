// loss.cu — REINFORCE / PPO loss and its gradient with respect to every policy
// parameter over a minibatch of rollout rows (Sec. 4.3).
//
// Pipeline (fp32, deterministic for a given launch configuration):
//   1. gather the minibatch observations X [n][D] from the [T][D][E] buffer;
//   2. forward GEMMs H_l = act_l(H_{l-1} W_l^T + b_l), keeping every activation;
//   3. loss head per row: log-softmax, rho, clipped surrogate, entropy, value
//      residual -> dL/dZ of the last layer and per-block fp64 statistics;
//   4. backward per layer: dW_l = dZ_l^T H_{l-1} (split over rows, partial tiles
//      summed in split order), db_l = column sums of dZ_l, and
//      dZ_{l-1} = (dZ_l W_l) * (1 - H_{l-1}^2), written in place over H_{l-1}.
// The GEMMs use one tiled SIMT kernel (64 x 64 tiles, 4 x 4 per thread) whose
// operands are addressed through strides, so transposes cost nothing.
#include <cstdint>

#include "devmath.cuh"
#include "kernels.h"

namespace simx {

constexpr int kBM = 64, kBN = 64, kBK = 16, kGemmThreads = 256;
// EPI_BIAS_ACT: + bias, then the activation `act` (0 tanh, 1 identity, 2 GELU, which also
// writes its derivative to D); EPI_DACT: times the derivative of `act` (1 - H^2 for tanh,
// D for GELU, 1 for identity).
enum Epi : int { EPI_NONE = 0, EPI_BIAS = 1, EPI_BIAS_ACT = 2, EPI_DACT = 3 };

struct Gemm {
  const float* A;  // A(i, k) = A[i * sai + k * sak]
  int64_t sai, sak;
  const float* B;  // B(k, j) = B[k * sbk + j * sbj]
  int64_t sbk, sbj;
  float* C;        // C(i, j) = C[i * ldc + j] (+ split * split_stride)
  int64_t ldc;
  int64_t M, N, K;
  int64_t k_per_split;
  int64_t split_stride;
  const float* bias;  // [N]
  const float* H;     // EPI_DACT, tanh: multiply by (1 - H(i, j)^2), H(i, j) = H[i * ldc + j]
  float* D;           // GELU derivative, D(i, j) = D[i * ldc + j]: written by EPI_BIAS_ACT, read by EPI_DACT
  int epi;
  int act;
  int mode_a, mode_b;  // operand load modes (load_tile), set by gemm()
};

// One operand's 64 x 16 tile X(r, k) = X[r * sr + k * sk], r in [r0, r0 + 64) (rows of
// A or columns of B), k in [k0, k0 + 16), four values per thread.  mode 1: 16-byte loads
// along k (sk == 1, sr % 4 == 0, 16-byte base, k0 % 4 == 0); mode 2: 16-byte loads along
// r (sr == 1, sk % 4 == 0, 16-byte base); they serve full tiles, element loads with
// bounds serve the rest and modes 0 and 3 (consecutive threads walking r, or k when the
// operand is contiguous along k).  v[c] goes to shared (kk[c], rr[c]).
struct TileLoad {
  float v[4];
  int kk[4], rr[4];
};

__device__ __forceinline__ void load_tile(const float* __restrict__ X, int64_t sr, int64_t sk,
                                          int mode, int64_t r0, int64_t rlim, int64_t k0,
                                          int64_t ke, TileLoad& t) {
  const int tid = threadIdx.x;
  const bool full = r0 + kBM <= rlim && k0 + kBK <= ke;
  if (full && mode == 1) {
    const int r = tid / 4, kq = tid % 4;
    const float4 q = *reinterpret_cast<const float4*>(X + (r0 + r) * sr + k0 + 4 * kq);
    t.v[0] = q.x, t.v[1] = q.y, t.v[2] = q.z, t.v[3] = q.w;
#pragma unroll
    for (int c = 0; c < 4; ++c) t.kk[c] = 4 * kq + c, t.rr[c] = r;
  } else if (full && mode == 2) {
    const int k = tid / 16, rq = tid % 16;
    const float4 q = *reinterpret_cast<const float4*>(X + r0 + 4 * rq + (k0 + k) * sk);
    t.v[0] = q.x, t.v[1] = q.y, t.v[2] = q.z, t.v[3] = q.w;
#pragma unroll
    for (int c = 0; c < 4; ++c) t.kk[c] = k, t.rr[c] = 4 * rq + c;
  } else {
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int e = tid + kGemmThreads * c;
      int k, r;
      if (mode == 1 || mode == 3) {  // consecutive threads walk k
        k = e % kBK;
        r = e / kBK;
      } else {
        r = e % kBM;
        k = e / kBM;
      }
      const int64_t rg = r0 + r, kg = k0 + k;
      t.v[c] = (rg < rlim && kg < ke) ? X[rg * sr + kg * sk] : 0.0f;
      t.kk[c] = k;
      t.rr[c] = r;
    }
  }
}

// C(i, j) = sum over k in [kb, ke) of A(i, k) B(k, j), k in increasing order (one fma
// chain per output), then the epilogue.  64 x 64 output tile per block, each thread a
// contiguous 4 x 4 block read from shared memory as 16-byte rows; the next k tile is
// loaded into registers while the current one is multiplied (two shared buffers, one
// barrier per tile).
__global__ void __launch_bounds__(kGemmThreads) k_gemm(const __grid_constant__ Gemm g) {
  constexpr int kLd = kBM + 4;
  __shared__ __align__(16) float As[2][kBK][kLd];
  __shared__ __align__(16) float Bs[2][kBK][kLd];
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int64_t i0 = (int64_t)blockIdx.y * kBM, j0 = (int64_t)blockIdx.x * kBN;
  const int64_t kb = (int64_t)blockIdx.z * g.k_per_split;
  const int64_t ke = kb + g.k_per_split < g.K ? kb + g.k_per_split : g.K;
  float acc[4][4];
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int b = 0; b < 4; ++b) acc[a][b] = 0.0f;
  TileLoad ta, tb;
  int cur = 0;
  if (kb < ke) {
    load_tile(g.A, g.sai, g.sak, g.mode_a, i0, g.M, kb, ke, ta);
    load_tile(g.B, g.sbj, g.sbk, g.mode_b, j0, g.N, kb, ke, tb);
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      As[0][ta.kk[c]][ta.rr[c]] = ta.v[c];
      Bs[0][tb.kk[c]][tb.rr[c]] = tb.v[c];
    }
  }
  __syncthreads();
  for (int64_t k0 = kb; k0 < ke; k0 += kBK) {
    const bool more = k0 + kBK < ke;
    if (more) {
      load_tile(g.A, g.sai, g.sak, g.mode_a, i0, g.M, k0 + kBK, ke, ta);
      load_tile(g.B, g.sbj, g.sbk, g.mode_b, j0, g.N, k0 + kBK, ke, tb);
    }
#pragma unroll
    for (int kk = 0; kk < kBK; ++kk) {
      const float4 av = *reinterpret_cast<const float4*>(&As[cur][kk][4 * ty]);
      const float4 bv = *reinterpret_cast<const float4*>(&Bs[cur][kk][4 * tx]);
      const float a4[4] = {av.x, av.y, av.z, av.w}, b4[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
      for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) acc[a][b] = __fmaf_rn(a4[a], b4[b], acc[a][b]);
    }
    if (more) {
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        As[cur ^ 1][ta.kk[c]][ta.rr[c]] = ta.v[c];
        Bs[cur ^ 1][tb.kk[c]][tb.rr[c]] = tb.v[c];
      }
    }
    __syncthreads();
    cur ^= 1;
  }
  float* C = g.C + (int64_t)blockIdx.z * g.split_stride;
#pragma unroll
  for (int a = 0; a < 4; ++a) {
    const int64_t i = i0 + 4 * ty + a;
    if (i >= g.M) continue;
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      const int64_t j = j0 + 4 * tx + b;
      if (j >= g.N) continue;
      float v = acc[a][b];
      if (g.epi == EPI_BIAS || g.epi == EPI_BIAS_ACT) v = __fadd_rn(v, g.bias[j]);
      if (g.epi == EPI_BIAS_ACT) {
        if (g.act == 0) v = det_tanh(v);
        else if (g.act == 2) det_gelu_grad(v, v, g.D[i * g.ldc + j]);
      }
      if (g.epi == EPI_DACT) {
        if (g.act == 0) {
          const float h = g.H[i * g.ldc + j];
          v = v * (1.0f - h * h);
        } else if (g.act == 2) {
          v = v * g.D[i * g.ldc + j];
        }
      }
      C[i * g.ldc + j] = v;
    }
  }
}

// Load mode of an operand X(r, k) = X[r * sr + k * sk] for load_tile: 16-byte loads need
// a 16-byte base, the other stride a multiple of 4, and (along k) tiles starting on a
// multiple of 4, which k_per_split % 16 == 0 (or a single split from k = 0) provides.
static int load_mode(const float* X, int64_t sr, int64_t sk, int64_t k_per_split, int splits) {
  const bool aligned = (reinterpret_cast<uintptr_t>(X) & 15) == 0;
  const bool k_ok = splits == 1 || k_per_split % 16 == 0;
  if (aligned && sk == 1 && sr % 4 == 0 && k_ok) return 1;
  if (aligned && sr == 1 && sk % 4 == 0) return 2;
  return sk == 1 ? 3 : 0;  // element loads, walking the contiguous direction
}

static cudaError_t gemm(const Gemm& g0, int splits, cudaStream_t s) {
  Gemm g = g0;
  g.mode_a = load_mode(g.A, g.sai, g.sak, g.k_per_split, splits);
  g.mode_b = load_mode(g.B, g.sbj, g.sbk, g.k_per_split, splits);
  const dim3 grid((unsigned)((g.N + kBN - 1) / kBN), (unsigned)((g.M + kBM - 1) / kBM), (unsigned)splits);
  k_gemm<<<grid, kGemmThreads, 0, s>>>(g);
  count_launches(1);
  return cudaGetLastError();
}

// X[r][d] = obs[t][d][e] with (t, e) = (row / E, row % E), row = idx[r] (or r).
__global__ void k_gather(const float* __restrict__ obs, const int64_t* __restrict__ idx, int64_t n,
                         int D, int64_t E, float* __restrict__ X) {
  const int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (q >= n * D) return;
  const int64_t r = q / D;
  const int d = (int)(q % D);
  const int64_t row = idx ? idx[r] : r;
  const int64_t t = row / E, e = row % E;
  X[q] = obs[(t * D + d) * E + e];
}

// Loss head: Z [n][Nl] (A logits + value) -> dZ in place; per-block fp64 partial
// sums of {policy term, squared value error, entropy, clipped} into part[block][4].
constexpr int kHeadThreads = 128;
__global__ void __launch_bounds__(kHeadThreads)
k_loss_head(float* __restrict__ Z, int64_t n, int Nl, int A, int has_value,
            const uint8_t* __restrict__ action, const float* __restrict__ logp_old,
            const float* __restrict__ adv, const float* __restrict__ ret,
            const int64_t* __restrict__ idx, int algo, float eps, float cv, float ce,
            double* __restrict__ part) {
  __shared__ double sh[4][kHeadThreads];
  const int64_t r = (int64_t)blockIdx.x * kHeadThreads + threadIdx.x;
  double pgv = 0.0, vv = 0.0, hv = 0.0, cf = 0.0;
  if (r < n) {
    float* z = Z + r * Nl;
    const int64_t row = idx ? idx[r] : r;
    const int a = action[row];
    const float ad = adv[row];
    float m = z[0];
    for (int i = 1; i < A; ++i) m = fmaxf(m, z[i]);
    float S = 0.0f;
    for (int i = 0; i < A; ++i) S += det_exp(z[i] - m);
    const float lse = m + det_log(S);
    float H = 0.0f;
    for (int i = 0; i < A; ++i) {
      const float lp = z[i] - lse;
      H -= det_exp(lp) * lp;
    }
    const float lpa = z[a] - lse;
    float coef, pg;
    if (algo == SIMX_ALGO_REINFORCE) {
      coef = ad;
      pg = -ad * lpa;
    } else {
      const float rho = det_exp(lpa - logp_old[row]);
      const float s1 = rho * ad;
      const float s2 = fminf(fmaxf(rho, 1.0f - eps), 1.0f + eps) * ad;
      pg = -fminf(s1, s2);
      coef = (s1 <= s2 ? ad : 0.0f) * rho;
      cf = fabsf(rho - 1.0f) > eps ? 1.0 : 0.0;
    }
    const float inv_n = 1.0f / (float)n;
    for (int i = 0; i < A; ++i) {
      const float lp = z[i] - lse;
      const float p = det_exp(lp);
      const float onehot = (i == a) ? 1.0f : 0.0f;
      z[i] = (-coef * (onehot - p) + ce * p * (lp + H)) * inv_n;
    }
    if (has_value) {
      const float dv = z[A] - ret[row];
      vv = (double)dv * (double)dv;
      z[A] = 2.0f * cv * dv * inv_n;
    }
    pgv = pg;
    hv = H;
  }
  sh[0][threadIdx.x] = pgv;
  sh[1][threadIdx.x] = vv;
  sh[2][threadIdx.x] = hv;
  sh[3][threadIdx.x] = cf;
  __syncthreads();
  for (int d = kHeadThreads / 2; d > 0; d >>= 1) {
    if ((int)threadIdx.x < d)
      for (int q = 0; q < 4; ++q) sh[q][threadIdx.x] += sh[q][threadIdx.x + d];
    __syncthreads();
  }
  if (threadIdx.x < 4) part[(int64_t)blockIdx.x * 4 + threadIdx.x] = sh[threadIdx.x][0];
}

__global__ void k_loss_stats(const double* __restrict__ part, int nblocks, int64_t n, int has_value,
                             float cv, float ce, float* __restrict__ stats) {
  __shared__ double sh[4][256];
  double a[4] = {0, 0, 0, 0};
  for (int b = threadIdx.x; b < nblocks; b += 256)
    for (int q = 0; q < 4; ++q) a[q] += part[(int64_t)b * 4 + q];
  for (int q = 0; q < 4; ++q) sh[q][threadIdx.x] = a[q];
  __syncthreads();
  for (int d = 128; d > 0; d >>= 1) {
    if ((int)threadIdx.x < d)
      for (int q = 0; q < 4; ++q) sh[q][threadIdx.x] += sh[q][threadIdx.x + d];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const double pg = sh[0][0] / (double)n, v = sh[1][0] / (double)n, H = sh[2][0] / (double)n;
    const double L = pg + (has_value ? (double)cv * v : 0.0) - (double)ce * H;
    stats[0] = (float)L;
    stats[1] = (float)pg;
    stats[2] = (float)v;
    stats[3] = (float)H;
    stats[4] = (float)(sh[3][0] / (double)n);
  }
}

// grad_W[j] = sum over splits of part[split][j] (in split order); db = column sums.
__global__ void k_reduce_splits(const float* __restrict__ part, int splits, int64_t len,
                                float* __restrict__ out) {
  const int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= len) return;
  float acc = 0.0f;
  for (int s = 0; s < splits; ++s) acc += part[(int64_t)s * len + j];
  out[j] = acc;
}

// db[j] = sum_r dZ[r][j], rows split into chunks, partial sums to part[chunk][N].
__global__ void k_colsum(const float* __restrict__ dZ, int64_t n, int N, int64_t rows_per,
                         float* __restrict__ part) {
  const int j = threadIdx.x;
  if (j >= N) return;
  const int64_t r0 = (int64_t)blockIdx.x * rows_per;
  const int64_t r1 = r0 + rows_per < n ? r0 + rows_per : n;
  float acc = 0.0f;
  for (int64_t r = r0; r < r1; ++r) acc += dZ[r * N + j];
  part[(int64_t)blockIdx.x * N + j] = acc;
}

struct WsLayout {
  size_t X, H[SIMX_MAX_LAYERS], Dg[SIMX_MAX_LAYERS], Z, part, statp, total;
  int splits[SIMX_MAX_LAYERS], head_blocks;
};

// Row splits of layer l's dW product (output N x K tiles of 64 x 64, reduction over the
// n rows): one per 2048 rows, and at least enough that the product launches two blocks
// per SM, without going below 64 rows per split or above 512 splits.  A fixed function
// of the sizes, so the summation order is the same on every run.
static int dw_splits(int64_t n, int N, int K) {
  const int64_t tiles = (int64_t)((N + kBM - 1) / kBM) * ((K + kBN - 1) / kBN);
  int64_t s = (n + 2047) / 2048;
  const int64_t fill = (2 * (int64_t)sm_count() + tiles - 1) / tiles;
  if (s < fill) s = fill;
  const int64_t most = (n + 63) / 64;
  if (s > most) s = most;
  if (s > 512) s = 512;
  if (s < 1) s = 1;
  return (int)s;
}

static WsLayout layout(const LossArgs& a) {
  WsLayout w{};
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += (bytes + 255) & ~(size_t)255;
    return o;
  };
  const int64_t n = a.n;
  w.X = take((size_t)n * a.dims[0] * sizeof(float));
  for (int l = 1; l < a.n_layers; ++l) w.H[l] = take((size_t)n * a.dims[l] * sizeof(float));
  for (int l = 1; l < a.n_layers; ++l)  // GELU derivative of layer l's input
    w.Dg[l] = a.act[l - 1] == 2 ? take((size_t)n * a.dims[l] * sizeof(float)) : 0;
  w.Z = take((size_t)n * a.dims[a.n_layers] * sizeof(float));
  size_t maxw = 0;  // the largest split-partial buffer: splits x N x K floats
  for (int l = 0; l < a.n_layers; ++l) {
    w.splits[l] = dw_splits(n, a.dims[l + 1], a.dims[l]);
    const size_t sz = (size_t)w.splits[l] * a.dims[l + 1] * a.dims[l];
    if (sz > maxw) maxw = sz;
  }
  w.part = take(maxw * sizeof(float));
  w.head_blocks = (int)((n + kHeadThreads - 1) / kHeadThreads);
  w.statp = take((size_t)w.head_blocks * 4 * sizeof(double));
  w.total = off;
  return w;
}

// Large enough for every path, so that the size does not depend on the precision.
size_t loss_workspace_bytes(const LossArgs& a) {
  const size_t f = loss_fused_fits(a) ? loss_fused_workspace(a) : layout(a).total;
  const bool tc = loss_tc_fits(a);
  const size_t t = tc ? loss_tc_workspace(a) : loss_wide_workspace(a);
  return f > t ? f : t;
}

// Grid policies take the fused FP32 kernel (their forward's rounding and straight-through
// gradient live there).  TF32 requests whose policy fits the one-SM tensor-core kernel take
// it (loss_tc.cu), and
// wider tanh policies (layers up to 256) the streamed tensor-core kernels (loss_wide.cu);
// otherwise policies whose parameters and per-tile activations fit in shared memory take
// the fused FP32 one-kernel path (loss_fused.cu), and wider ones the GEMM pipeline below.
cudaError_t launch_loss_grad(const LossArgs& a, void* ws, size_t ws_bytes, cudaStream_t s) {
  if (a.grid)   // grid policies: the fused FP32 kernel, whatever the precision asked for
    return loss_fused_fits(a) ? launch_loss_fused(a, ws, ws_bytes, s) : cudaErrorInvalidValue;
  if (a.precision == SIMX_PREC_TF32 && loss_tc_fits(a)) return launch_loss_tc(a, ws, ws_bytes, s);
  if (a.precision == SIMX_PREC_TF32 && loss_wide_fits(a)) return launch_loss_wide(a, ws, ws_bytes, s);
  if (loss_fused_fits(a)) return launch_loss_fused(a, ws, ws_bytes, s);
  const WsLayout w = layout(a);
  if (ws_bytes < w.total) return cudaErrorInvalidValue;
  char* base = static_cast<char*>(ws);
  const int64_t n = a.n;
  const int L = a.n_layers;
  float* X = reinterpret_cast<float*>(base + w.X);
  float* Hs[SIMX_MAX_LAYERS + 1];
  Hs[0] = X;
  float* Dg[SIMX_MAX_LAYERS + 1] = {};
  for (int l = 1; l < L; ++l) {
    Hs[l] = reinterpret_cast<float*>(base + w.H[l]);
    if (a.act[l - 1] == 2) Dg[l] = reinterpret_cast<float*>(base + w.Dg[l]);
  }
  float* Z = reinterpret_cast<float*>(base + w.Z);
  float* part = reinterpret_cast<float*>(base + w.part);
  double* statp = reinterpret_cast<double*>(base + w.statp);
  const int D = a.dims[0];
  {
    const int64_t tot = n * D;
    k_gather<<<(unsigned)((tot + 255) / 256), 256, 0, s>>>(a.obs, a.idx, n, D, a.E, X);
    count_launches(1);
  }
  // forward
  for (int l = 0; l < L; ++l) {
    const int K = a.dims[l], N = a.dims[l + 1];
    Gemm g{};
    g.A = Hs[l];
    g.sai = K;
    g.sak = 1;
    g.B = a.W[l];  // B(k, j) = W[j][k]
    g.sbk = 1;
    g.sbj = K;
    g.C = (l + 1 < L) ? Hs[l + 1] : Z;
    g.ldc = N;
    g.M = n;
    g.N = N;
    g.K = K;
    g.k_per_split = K;
    g.split_stride = 0;
    g.bias = a.b[l];
    g.epi = (l + 1 < L) ? EPI_BIAS_ACT : EPI_BIAS;
    g.act = a.act[l];
    g.D = (l + 1 < L) ? Dg[l + 1] : nullptr;
    cudaError_t e = gemm(g, 1, s);
    if (e != cudaSuccess) return e;
  }
  const int NL = a.dims[L];
  k_loss_head<<<w.head_blocks, kHeadThreads, 0, s>>>(Z, n, NL, a.n_actions, a.has_value, a.action,
                                                     a.logp_old, a.adv, a.ret, a.idx, a.algo,
                                                     a.clip_eps, a.c_value, a.c_entropy, statp);
  k_loss_stats<<<1, 256, 0, s>>>(statp, w.head_blocks, n, a.has_value, a.c_value, a.c_entropy, a.stats);
  count_launches(2);
  // backward
  size_t goff[SIMX_MAX_LAYERS];
  {
    size_t o = 0;
    for (int l = 0; l < L; ++l) {
      goff[l] = o;
      o += (size_t)a.dims[l + 1] * a.dims[l] + a.dims[l + 1];
    }
  }
  const float* dZ = Z;
  for (int l = L - 1; l >= 0; --l) {
    const int K = a.dims[l], N = a.dims[l + 1];
    const int splits = w.splits[l];
    const int64_t kps = (n + splits - 1) / splits;
    // dW = dZ^T H_in : M = N, N = K, reduction over rows
    Gemm g{};
    g.A = dZ;  // A(i, k) = dZ[k][i]
    g.sai = 1;
    g.sak = N;
    g.B = Hs[l];  // B(k, j) = H[k][j]
    g.sbk = K;
    g.sbj = 1;
    g.C = part;
    g.ldc = K;
    g.M = N;
    g.N = K;
    g.K = n;
    g.k_per_split = kps;
    g.split_stride = (int64_t)N * K;
    g.epi = EPI_NONE;
    cudaError_t e = gemm(g, splits, s);
    if (e != cudaSuccess) return e;
    float* gW = a.grad + goff[l];
    float* gb = gW + (size_t)N * K;
    k_reduce_splits<<<(unsigned)(((int64_t)N * K + 255) / 256), 256, 0, s>>>(part, splits, (int64_t)N * K, gW);
    // db: column sums with the same row splits
    float* bpart = part;  // the dW partials are consumed by the reduce above
    k_colsum<<<splits, ((N + 31) / 32) * 32, 0, s>>>(dZ, n, N, kps, bpart);
    k_reduce_splits<<<(unsigned)((N + 255) / 256), 256, 0, s>>>(bpart, splits, N, gb);
    count_launches(3);
    if (l > 0) {
      // dZ of layer l-1 = (dZ W) * act'(Z_{l-1}) (1 - H^2 for tanh, H = Hs[l]), in place
      Gemm d{};
      d.A = dZ;  // A(i, k) = dZ[i][k], k over N
      d.sai = N;
      d.sak = 1;
      d.B = a.W[l];  // B(k, j) = W[k][j]
      d.sbk = K;
      d.sbj = 1;
      d.C = Hs[l];
      d.ldc = K;
      d.M = n;
      d.N = K;
      d.K = N;
      d.k_per_split = N;
      d.split_stride = 0;
      d.H = Hs[l];
      d.D = Dg[l];
      d.act = a.act[l - 1];
      d.epi = EPI_DACT;
      e = gemm(d, 1, s);
      if (e != cudaSuccess) return e;
      dZ = Hs[l];
    }
  }
  return cudaGetLastError();
}

}  // namespace simx
