// loss_wide.cu — REINFORCE / PPO loss gradient (Sec. 4.3) on the tensor cores for tanh
// policies whose layers are up to 256 wide (c3 / c5: 13-128-128-17, c4: 28-256-256-49),
// too wide for loss_tc.cu's kernel, which holds every operand of a policy in one SM.
//
// Notation: L layers, H_0 = X (the minibatch's observations), Z_l = H_l W_l^T + b_l,
// H_{l+1} = tanh(Z_l); G_l = dL/dZ_l.  Backward: dH_l = G_l W_l and
// G_{l-1} = dH_l * (1 - H_l^2); dW_l = G_l^T H_l, db_l = sum over rows of G_l.
// Every matrix product is a chain of tcgen05.mma kind::tf32 (TF32 inputs, FP32
// accumulation in tensor memory) with M = 128.  Three kernels per call:
//
//   k_lw_prep  the policy's weights as MMA operand images in global memory: W_l (the
//              forward B operand) and W_l^T (the backward one) cut into chunks of 32 K
//              values, each chunk laid out exactly as the shared-memory operand so that
//              one bulk copy moves it; TF32 rounded.  The first layer's image is
//              [W_hi | W_lo | W_hi], the split-TF32 product x_hi w_hi + x_hi w_lo +
//              x_lo w_hi as one GEMM against [x_hi | x_hi | x_lo] (raw observations reach
//              magnitudes in the hundreds; one TF32 pass there moves saturated tanh units'
//              derivatives by percents).
//   k_lw_rows  a cluster of two CTAs per 128-row tile: the whole forward pass, the loss
//              head and the backward pass down to G_0 for its rows.  The A operand (the
//              tile's activations, or G) stays resident in both CTAs' shared memory; each
//              CTA computes half of the outputs of every product but the last layer's
//              (its half of the rows of each weight chunk, which stream through a ring of
//              shared-memory stages by bulk copies, the MMAs of chunk c queued before the
//              stage of chunk c - 1 is refilled) and writes its half of the next operand
//              into both A buffers (distributed shared memory, a cluster barrier on each
//              side); the loss head is split by rows.  H_l and G_l go to global memory as
//              feature-major images (the layout of the weight-gradient products).
//   k_lw_dw    [dW_l | db_l] = G_l^T [H_l | 1] with K = the rows, split over CTAs by
//              (layer, block of 128 outputs, row range); each CTA writes its slice of
//              one full-length partial gradient per row range, which the block reduction
//              shared with the other loss paths sums in range order (deterministic).
//
// Elementwise work between the products (bias, tanh, the loss head, 1 - h^2) is done
// in FP32 by threads reading the accumulators with tcgen05.ld: thread = TMEM lane =
// tile row, the two warps of a lane quarter splitting the columns.  Accuracy is that of
// TF32 inputs (about 1e-3 relative per product), held to 1e-2 by the tests; the FP32 SIMT
// kernels are the exact alternative.
#include <cstdint>

#include "kernels.h"
#include "tc_common.cuh"

namespace simx {
namespace lw {

using namespace tcx;

constexpr int kR = 128;            // rows per tile (MMA M)
constexpr int kThreads = 512;      // k_lw_rows: 16 warps, 4 per TMEM lane quarter
constexpr int kDwThreads = 256;    // k_lw_dw: 8 warps, 2 per lane quarter
constexpr int kKC = 32;            // K values per streamed chunk
constexpr int kMaxStages = 6;
constexpr long long kWaitCycles = 2000000000LL;  // bound on any wait (about 1 s)

int r16(int x) { return (x + 15) / 16 * 16; }
int r32(int x) { return (x + 31) / 32 * 32; }

struct Plan {
  bool ok;
  int L, n_params;
  int K[SIMX_MAX_LAYERS], N[SIMX_MAX_LAYERS];
  int Ka[SIMX_MAX_LAYERS];   // forward A width (GEMM K): 3 r32(K_0) for layer 0, r32(K_l) after
  int Nf[SIMX_MAX_LAYERS];   // forward outputs: r32(N_l) split in two halves, r16 for the last layer
  int Gk[SIMX_MAX_LAYERS];   // backward A width (GEMM K of dH_l = G_l W_l): r32(N_l)
  int Kb[SIMX_MAX_LAYERS];   // backward products' outputs: r32(K_l), in two halves of hK
  int hN[SIMX_MAX_LAYERS];   // forward MMA N of one CTA: Nf / 2 (split) or Nf (last layer)
  int hK[SIMX_MAX_LAYERS];   // backward MMA N of one CTA: Kb / 2
  int Fh[SIMX_MAX_LAYERS];   // features of the H_l image: r16(K_l)
  int Fg[SIMX_MAX_LAYERS];   // features of the G_l image: r16(N_l)
  int poff[SIMX_MAX_LAYERS];
  // k_lw_rows
  int a_bytes, stage_bytes, nstages, smem, tcols;
  int hs_off;                // the loss head's scratch inside the A buffer (3 KB)
  int b_off[SIMX_MAX_LAYERS];  // the biases, copied to shared memory after the misc area
  int b_total;
  // k_lw_dw
  int mt0[SIMX_MAX_LAYERS];  // first work item of layer l (blocks of 128 outputs)
  int mt_total, S, dw_stage_bytes, dw_nstages, dw_smem, dw_tcols;
  int64_t n_pad, ntiles, nchunks;
  // workspace byte offsets
  size_t wf[SIMX_MAX_LAYERS], wb[SIMX_MAX_LAYERS], img_h[SIMX_MAX_LAYERS], img_g[SIMX_MAX_LAYERS];
  size_t part, spart, total;
  int64_t wf_elems[SIMX_MAX_LAYERS], wb_elems[SIMX_MAX_LAYERS];
};

struct Args {
  LossArgs a;
  Plan p;
  unsigned char* ws;
};

// Byte offset of feature f inside a 32-row block of a feature-major image: blocks of 32
// rows, in each block the feature groups of 8 one after another, each group the K-major
// operand of 8 features x 32 rows (8 core matrices of 4 rows, 128 bytes apart); so
// (feature f, row r) is at block (r / 32) + img_col(f) + ((r % 32) / 4) * 128 + (r % 4) * 4.
__device__ __forceinline__ uint32_t img_col(int f) { return (uint32_t)((f >> 3) * 1024 + (f & 7) * 16); }

// 4 x 4 transposes inside each group of 4 lanes: afterwards lane 4m + j holds, at
// v[4a + i], what lane 4m + i held at v[4a + j] (applied twice it is the identity).
__device__ __forceinline__ void quad_transpose(float (&v)[16], int j) {
#pragma unroll
  for (int a = 0; a < 4; ++a) {
#pragma unroll
    for (int b = 0; b < 2; ++b) {
      const float send = (j & 2) ? v[4 * a + b] : v[4 * a + b + 2];
      const float recv = __shfl_xor_sync(0xFFFFFFFFu, send, 2);
      if (j & 2) v[4 * a + b] = recv;
      else v[4 * a + b + 2] = recv;
    }
#pragma unroll
    for (int b = 0; b < 4; b += 2) {
      const float send = (j & 1) ? v[4 * a + b] : v[4 * a + b + 1];
      const float recv = __shfl_xor_sync(0xFFFFFFFFu, send, 1);
      if (j & 1) v[4 * a + b] = recv;
      else v[4 * a + b + 1] = recv;
    }
  }
}

// The 32-row block of an image of F features that holds this warp's rows.
__device__ __forceinline__ size_t img_blk(int64_t grow, int F) {
  return (size_t)((grow >> 5) * (F >> 3)) * 1024;
}

// This warp's 32 rows x features c0 .. c0 + 15 (v: the lane's row) into an image block:
// after the transpose each lane stores whole 16-byte segments (one feature, 4 rows), so
// the warp writes contiguous runs.  v is transposed in place.
__device__ __forceinline__ void img_store16(unsigned char* blk, int c0, float (&v)[16], int lane) {
  quad_transpose(v, lane & 3);
  const int m = lane >> 2, j = lane & 3;
#pragma unroll
  for (int a = 0; a < 4; ++a)
    *reinterpret_cast<float4*>(blk + img_col(c0 + 4 * a + j) + m * 128) =
        make_float4(v[4 * a], v[4 * a + 1], v[4 * a + 2], v[4 * a + 3]);
}

// The inverse: features c0 .. c0 + 15 of the lane's row from an image block.
__device__ __forceinline__ void img_load16(const unsigned char* blk, int c0, float (&v)[16], int lane) {
  const int m = lane >> 2, j = lane & 3;
#pragma unroll
  for (int a = 0; a < 4; ++a) {
    const float4 t = *reinterpret_cast<const float4*>(blk + img_col(c0 + 4 * a + j) + m * 128);
    v[4 * a] = t.x;
    v[4 * a + 1] = t.y;
    v[4 * a + 2] = t.z;
    v[4 * a + 3] = t.w;
  }
  quad_transpose(v, j);
}

// Byte offset of (row j, value kk) inside one 32-value chunk of a weight image.
__device__ __forceinline__ uint32_t chunk_off(int j, int kk) {
  return (uint32_t)((j >> 3) * 1024 + (kk >> 2) * 128 + (j & 7) * 16 + (kk & 3) * 4);
}

// ---------------------------------------------------------------------------------
// k_lw_prep: the weight operand images of every layer (TF32 rounded, zero padded).
// ---------------------------------------------------------------------------------
__global__ void k_lw_prep(const __grid_constant__ Args A) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const LossArgs& a = A.a;
  const Plan& P = A.p;
  int64_t total = 0;
  for (int l = 0; l < P.L; ++l) total += P.wf_elems[l] + P.wb_elems[l];
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x) {
    int64_t q = i;
    int l = 0;
    bool fwd = true;
    for (; l < P.L; ++l) {
      if (q < P.wf_elems[l]) { fwd = true; break; }
      q -= P.wf_elems[l];
      if (q < P.wb_elems[l]) { fwd = false; break; }
      q -= P.wb_elems[l];
    }
    const int K = P.K[l], N = P.N[l];
    const float* W = a.W[l];
    if (fwd) {
      // chunk c of Nf rows x 32 values; element (row j = output, kk)
      const int Nf = P.Nf[l];
      const int c = (int)(q / (Nf * kKC)), rem = (int)(q % (Nf * kKC));
      const int j = rem / kKC, kk = rem % kKC;
      float v;
      if (l == 0) {
        const int per = P.Ka[0] / 3 / kKC;  // chunks of one copy of K_0
        const int part = c / per, k = kKC * (c % per) + kk;
        const float w = (j < N && k < K) ? W[(size_t)j * K + k] : 0.0f;
        const float hi = to_tf32(w);
        v = part == 1 ? to_tf32(w - hi) : hi;
      } else {
        const int k = kKC * c + kk;
        v = (j < N && k < K) ? to_tf32(W[(size_t)j * K + k]) : 0.0f;
      }
      float* dst = reinterpret_cast<float*>(A.ws + P.wf[l] + (size_t)c * Nf * kKC * 4 + chunk_off(j, kk));
      *dst = v;
    } else {
      // chunk c of Kb rows (input units k) x 32 values (outputs j = 32 c + jj)
      const int Kb = P.Kb[l];
      const int c = (int)(q / (Kb * kKC)), rem = (int)(q % (Kb * kKC));
      const int k = rem / kKC, jj = rem % kKC;
      const int j = kKC * c + jj;
      const float v = (k < K && j < N) ? to_tf32(W[(size_t)j * K + k]) : 0.0f;
      float* dst = reinterpret_cast<float*>(A.ws + P.wb[l] + (size_t)c * Kb * kKC * 4 + chunk_off(k, jj));
      *dst = v;
    }
  }
}

// ---------------------------------------------------------------------------------
// k_lw_rows: forward, loss head and backward of one 128-row tile.
// ---------------------------------------------------------------------------------
__device__ __forceinline__ float tanh_fast(float x) {
  return 1.0f - __fdividef(2.0f, __expf(2.0f * x) + 1.0f);
}

struct Smem {
  unsigned char* abuf;     // the resident A operand (activations or G of the tile)
  unsigned char* stages;   // ring of weight chunks
  uint64_t* full;          // [kMaxStages] chunk landed (bulk copy transactions)
  uint64_t* mmab;          // [kMaxStages] MMAs reading the stage completed
  uint64_t* drain;         // every MMA of the CTA completed (end of kernel)
  uint64_t* accb;          // the accumulator of the current GEMM is complete
  uint32_t* tbase;         // tensor memory base address
  int* abort_flag;         // a wait timed out: stop issuing work
  double* dstat;           // [4 warps][4] statistics
};

__device__ __forceinline__ Smem carve(unsigned char* sm, const Plan& P, int stage_bytes, int nstages,
                                      int a_bytes) {
  Smem s;
  s.abuf = sm;
  s.stages = sm + a_bytes;
  unsigned char* m = sm + a_bytes + (size_t)nstages * stage_bytes;
  s.full = reinterpret_cast<uint64_t*>(m);
  s.mmab = s.full + kMaxStages;
  s.drain = s.mmab + kMaxStages;
  s.accb = s.drain + 1;
  s.tbase = reinterpret_cast<uint32_t*>(s.accb + 1);
  s.abort_flag = reinterpret_cast<int*>(s.tbase + 1);
  s.dstat = reinterpret_cast<double*>(m + 128);
  (void)P;
  return s;
}

// The weight chunks of k_lw_rows in the order its GEMMs consume them (forward layers
// 0 .. L-1, then the backward products of layers L-1 .. 1): GEMM g takes the global
// chunks k0[g] .. k0[g + 1] - 1; chunk k goes through stage k % S.
struct Sched {
  int ng, total;
  int k0[2 * SIMX_MAX_LAYERS];
  const unsigned char* src[2 * SIMX_MAX_LAYERS];
  uint32_t bytes[2 * SIMX_MAX_LAYERS];    // copied per chunk (this CTA's half of the rows)
  uint32_t stride[2 * SIMX_MAX_LAYERS];   // between the chunks of the image
};

// rank: this CTA's half of the split products (its output rows of each weight chunk).
__device__ Sched make_sched(const Plan& P, unsigned char* ws, int rank) {
  Sched q;
  q.ng = 2 * P.L - 1;
  int k = 0;
  for (int g = 0; g < q.ng; ++g) {
    q.k0[g] = k;
    if (g < P.L) {
      q.stride[g] = (uint32_t)P.Nf[g] * kKC * 4u;
      q.bytes[g] = (uint32_t)P.hN[g] * kKC * 4u;
      q.src[g] = ws + P.wf[g] + (P.hN[g] < P.Nf[g] ? (size_t)rank * q.bytes[g] : 0);
      k += P.Ka[g] / kKC;
    } else {
      const int l = 2 * P.L - 1 - g;
      q.stride[g] = (uint32_t)P.Kb[l] * kKC * 4u;
      q.bytes[g] = (uint32_t)P.hK[l] * kKC * 4u;
      q.src[g] = ws + P.wb[l] + (size_t)rank * q.bytes[g];
      k += P.Gk[l] / kKC;
    }
  }
  q.k0[q.ng] = k;
  q.total = k;
  return q;
}

// Thread 0: the bulk copy of global chunk k into its stage, once the MMAs that read the
// stage's previous chunk have completed (each stage barrier is waited on only after the
// use before it completed, so a parity names one phase).
__device__ bool load_chunk(const Smem& s, const Sched& q, int S, int stage_bytes, int k) {
  const int st = k % S;
  if (k >= S && !mbar_wait(&s.mmab[st], (uint32_t)(((k - S) / S) & 1), kWaitCycles)) return false;
  int g = 0;
  while (q.k0[g + 1] <= k) ++g;
  const uint32_t b = q.bytes[g];
  mbar_arrive_expect_tx(&s.full[st], b);
  bulk_g2s(s.stages + (size_t)st * stage_bytes, q.src[g] + (size_t)(k - q.k0[g]) * q.stride[g], b,
           &s.full[st]);
  return true;
}

// GEMM g  D = A B^T: A resident at a_addr (row-group stride a_sbo), the B chunks through
// the stage ring, by two threads that never wait for each other's instructions: the MMA
// thread (warp 1) waits for each chunk to land and queues its MMAs, the load thread
// (warp 0, which issued the first chunks before the tile's gather) refills each stage
// once the MMAs that read it completed, up to chunk k0[g + 1] + S - 1: on into the next
// GEMM's chunks, which arrive while the other threads work on this GEMM's result.  The
// accumulator's completion is announced on accb (one phase per GEMM), which every thread
// waits on.  A wait that times out sets the abort flag and returns (accb is then never
// committed and the other threads' waits time out too).
__device__ void gemm_mma(const Smem& s, const Sched& q, int S, int stage_bytes, int g,
                         uint32_t a_addr, uint32_t a_sbo, int Nmma, uint32_t dtm) {
  const uint32_t id = idesc_tf32(kR, Nmma);
  for (int k = q.k0[g]; k < q.k0[g + 1]; ++k) {
    const int st = k % S, c = k - q.k0[g];
    if (!mbar_wait(&s.full[st], (uint32_t)((k / S) & 1), kWaitCycles)) {
      *s.abort_flag = 1;
      return;
    }
    fence_after();
    const uint32_t bs = su32(s.stages + (size_t)st * stage_bytes);
#pragma unroll
    for (int ks = 0; ks < kKC / 8; ++ks)
      mma_tf32(dtm, sdesc(a_addr + (uint32_t)c * 1024u + (uint32_t)ks * 256u, 128, a_sbo),
               sdesc(bs + (uint32_t)ks * 256u, 128, 1024), id, (c | ks) ? 1u : 0u);
    commit(&s.mmab[st]);
  }
  commit(s.accb);
}

__device__ void gemm_load(const Smem& s, const Sched& q, int S, int stage_bytes, int g, int& issued) {
  const int end = q.k0[g + 1] + S - 1;
  const int upto = end < q.total ? end : q.total;
  while (issued < upto) {
    if (!load_chunk(s, q, S, stage_bytes, issued)) {
      *s.abort_flag = 1;
      return;
    }
    ++issued;
  }
}

// The end of a kernel, so that nothing is in flight when the CTA's shared and tensor
// memory are released: the load thread waits (bounded) for its last S loads to land (all
// of them were consumed unless a wait timed out), the MMA thread for every MMA it issued.
__device__ void drain_loads(const Smem& s, int S, int issued) {
  for (int k = issued > S ? issued - S : 0; k < issued; ++k)
    mbar_wait(&s.full[k % S], (uint32_t)((k / S) & 1), kWaitCycles);
}
__device__ void drain_mma(const Smem& s) {
  commit(s.drain);
  mbar_wait(s.drain, 0u, kWaitCycles);
}


// The two CTAs of a cluster share one 128-row tile: each computes half of the outputs of
// every split product (rank r: rows r * half .. of each weight chunk), and writes its half
// of the next operand into both CTAs' A buffers (distributed shared memory); the loss head
// is split by rows instead (the last layer runs whole in both CTAs).
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t peer_addr(uint32_t saddr, uint32_t rank) {
  uint32_t d;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(d) : "r"(saddr), "r"(rank));
  return d;
}
__device__ __forceinline__ void st_peer4(uint32_t addr, float4 v) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(v.x), "f"(v.y),
               "f"(v.z), "f"(v.w)
               : "memory");
}
// Every thread of both CTAs: their shared-memory writes (local and remote) made visible,
// the tensor cores included, before either goes on.
__device__ __forceinline__ void cluster_sync() {
  asm volatile("fence.proxy.async.shared::cluster;" ::: "memory");
  fence_before();
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
  fence_after();
}

__global__ void __launch_bounds__(kThreads, 1) k_lw_rows(const __grid_constant__ Args A) {
  extern __shared__ __align__(1024) unsigned char sm[];
  const LossArgs& a = A.a;
  const Plan& P = A.p;
  const int L = P.L, S = P.nstages;
  const Smem s = carve(sm, P, P.stage_bytes, S, P.a_bytes);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int quarter = warp & 3, cq = warp >> 2;   // lane quarter; column share 0..3
  const int r = 32 * quarter + lane;
  const int rank = (int)cluster_rank();
  const int64_t tile = blockIdx.x >> 1;
  const int64_t grow = tile * kR + r;   // row of the padded minibatch
  const bool live = grow < a.n;

  // The kernel is launched while k_lw_prep still runs (programmatic dependent launch):
  // everything up to the first read of the weight images (barriers, tensor memory, biases,
  // the observation gather) overlaps it; griddepcontrol.wait then waits for its images.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  // thread 0 (the load thread): barriers, then the first weight chunks on their way
  // before anything else; thread 32 (the MMA thread) the same chunk schedule
  Sched sch;
  int issued = 0;
  if (tid == 32) sch = make_sched(P, A.ws, rank);
  if (tid == 0) {
    for (int i = 0; i < kMaxStages; ++i) {
      mbar_init(&s.full[i], 1);
      mbar_init(&s.mmab[i], 1);
    }
    mbar_init(s.drain, 1);
    mbar_init(s.accb, 1);
    mbar_fence_init();
    *s.abort_flag = 0;
    asm volatile("griddepcontrol.wait;" ::: "memory");
    sch = make_sched(P, A.ws, rank);
    const int upto = S - 1 < sch.total ? S - 1 : sch.total;
    for (; issued < upto; ++issued) load_chunk(s, sch, S, P.stage_bytes, issued);
  }
  if (warp == 0) tm_alloc(s.tbase, (uint32_t)P.tcols);
  // every layer's bias into shared memory (zero past each layer's outputs)
  float* sbias = reinterpret_cast<float*>(sm + P.a_bytes + (size_t)S * P.stage_bytes + 256);
  for (int l = 0; l < L; ++l)
    for (int i = tid; i < (P.N[l] + 15) / 16 * 16; i += kThreads)
      sbias[P.b_off[l] + i] = i < P.N[l] ? __ldg(a.b[l] + i) : 0.0f;

  // the tile's observations (both CTAs, every row): x_hi, x_hi, x_lo side by side in the A
  // buffer (split TF32); rank 0 writes the FP32 values to the H_0 image
  int64_t row = 0;
  if (live) row = a.idx ? __ldg(a.idx + grow) : grow;
  const int64_t t = row / a.E, e = row % a.E;
  const int D = P.K[0];
  {
    const int Kc = P.Ka[0] / 3, W0 = P.Ka[0], F0 = P.Fh[0];
    unsigned char* img = A.ws + P.img_h[0] + img_blk(grow, F0);
    // 16 features per pass: every gather load issued before any store
    for (int c0 = 16 * cq; c0 < Kc; c0 += 64) {
      float x[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const int f = c0 + i;
        x[i] = (live && f < D) ? __ldg(a.obs + (t * D + f) * a.E + e) : 0.0f;
      }
#pragma unroll
      for (int qq = 0; qq < 4; ++qq) {
        float hi[4], lo[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          hi[i] = to_tf32(x[4 * qq + i]);
          lo[i] = to_tf32(x[4 * qq + i] - hi[i]);
        }
        const int k = c0 + 4 * qq;
        const float4 h4 = make_float4(hi[0], hi[1], hi[2], hi[3]);
        *reinterpret_cast<float4*>(s.abuf + rm_off(r, k, W0)) = h4;
        *reinterpret_cast<float4*>(s.abuf + rm_off(r, Kc + k, W0)) = h4;
        *reinterpret_cast<float4*>(s.abuf + rm_off(r, 2 * Kc + k, W0)) = make_float4(lo[0], lo[1], lo[2], lo[3]);
      }
      if (rank == 0 && c0 < F0) img_store16(img, c0, x, lane);
    }
  }
  int ac = 0;
  float adv = 0.0f, lpo = 0.0f, ret = 0.0f;
  if (live) {
    ac = __ldg(a.action + row);
    adv = __ldg(a.adv + row);
    lpo = a.algo == SIMX_ALGO_PPO ? __ldg(a.logp_old + row) : 0.0f;
    ret = a.has_value ? __ldg(a.ret + row) : 0.0f;
  }
  asm volatile("griddepcontrol.wait;" ::: "memory");
  fence_async_smem();
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *s.tbase;
  const uint32_t tl = tmem + ((uint32_t)(32 * quarter) << 16);   // this warp's lane quarter
  const uint32_t abuf_addr = su32(s.abuf);
  const uint32_t peer = peer_addr(abuf_addr, (uint32_t)(rank ^ 1));   // the other CTA's A buffer
  int ngemm = 0;
  double st_pg = 0.0, st_v = 0.0, st_h = 0.0, st_cf = 0.0;
  const float inv_n = 1.0f / (float)a.n;

  // a float4 of the next operand into both CTAs' A buffers
  auto put_both = [&](uint32_t off, float4 v) {
    *reinterpret_cast<float4*>(s.abuf + off) = v;
    st_peer4(peer + off, v);
  };

  // The feature-major image rows an epilogue produces (FP32 H or G for the weight-gradient
  // kernel) wait in the second half of the tensor memory and go out while the next
  // product runs: the stores of all CTAs at once are bound by L2 bandwidth, the product
  // by the MMA issue, so overlapped they cost the longer of the two.  pend_*: the thread's
  // staged block (image, its features, first column, columns) until flushed.
  const uint32_t tstage = (uint32_t)P.tcols / 2;
  unsigned char* pend_img = nullptr;
  int pend_F = 0, pend_j0 = 0, pend_w = 0;
  auto stage_img = [&](int c0, const float (&v)[16]) { tm_st16_nw(tl + tstage + (uint32_t)c0, v); };
  auto flush = [&]() {
    if (!pend_img) return;
    for (int c0 = 16 * cq; c0 < pend_w; c0 += 64) {
      const int jg = pend_j0 + c0;
      if (jg < pend_F) {
        uint32_t u[16];
        tm_ld16_nw(tl + tstage + (uint32_t)c0, u);
        tm_wait();
        reg_fence16(u);
        float v[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(u[i]);
        img_store16(pend_img, jg, v, lane);
      }
    }
    pend_img = nullptr;
  };

  // GEMM g: threads 0 and 32 feed and issue it, every thread then waits for the
  // accumulator; then both CTAs meet, so that neither writes into the other's A buffer
  // while its products run.
  // After an abort no more work is issued, but every cluster barrier is still reached.
  auto gemm = [&](int g, int a_width, int Nmma) {
    const bool go = *s.abort_flag == 0;
    if (warp == 0) {
      if (lane == 0 && go) gemm_load(s, sch, S, P.stage_bytes, g, issued);
      __syncwarp();
    } else if (warp == 1) {
      if (lane == 0 && go)
        gemm_mma(s, sch, S, P.stage_bytes, g, abuf_addr, (uint32_t)(a_width / 4) * 128u, Nmma, tmem);
      __syncwarp();
    }
    flush();   // the previous epilogue's image rows, while the products run
    if (go && !mbar_wait_idle(s.accb, (uint32_t)(ngemm & 1), kWaitCycles)) atomicOr(s.abort_flag, 1);
    ++ngemm;
    __syncwarp();
    fence_after();
    cluster_sync();
  };

  // Columns c0 .. c0 + 15 of this thread's accumulator row (one warp-wide load; columns
  // from ncols on read as 0).  The allocation covers them: tcols is a power of two at
  // least as large as every 32-rounded width read here.
  auto ld16 = [&](int c0, int ncols, float (&z)[16]) {
    uint32_t u[16];
    tm_ld16_nw(tl + (uint32_t)c0, u);
    tm_wait();
    reg_fence16(u);
#pragma unroll
    for (int i = 0; i < 16; ++i) z[i] = c0 + i < ncols ? __uint_as_float(u[i]) : 0.0f;
  };

  // ---- forward
  for (int l = 0; l < L; ++l) {
    const int hN = P.hN[l];
    gemm(l, P.Ka[l], hN);
    const bool ok = *s.abort_flag == 0;
    const int Nl = P.N[l];
    const float* bias = sbias + P.b_off[l];
    if (l + 1 < L) {
      // H_{l+1} = tanh(Z_l + b_l) for this CTA's half of the outputs: TF32 into both A
      // buffers (width Ka[l+1] = Nf[l], zero padded), FP32 into the H_{l+1} image
      const int Wn = P.Ka[l + 1], Fn = P.Fh[l + 1], j0h = rank * hN;
      unsigned char* img = A.ws + P.img_h[l + 1] + img_blk(grow, Fn);
      uint32_t u[16];
      if (ok && 16 * cq < hN) tm_ld16_nw(tl + (uint32_t)(16 * cq), u);
      for (int c0 = 16 * cq; ok && c0 < hN; c0 += 64) {
        const int jg = j0h + c0;
        float z[16], bv[16], h[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) bv[i] = jg + i < Nl ? bias[jg + i] : 0.0f;
        tm_wait();
        reg_fence16(u);
#pragma unroll
        for (int i = 0; i < 16; ++i) z[i] = jg + i < Nl ? __uint_as_float(u[i]) : 0.0f;
        if (c0 + 64 < hN) tm_ld16_nw(tl + (uint32_t)(c0 + 64), u);
#pragma unroll
        for (int i = 0; i < 16; ++i) h[i] = jg + i < Nl ? tanh_fast(z[i] + bv[i]) : 0.0f;
#pragma unroll
        for (int qq = 0; qq < 4; ++qq)
          put_both(rm_off(r, jg + 4 * qq, Wn),
                   make_float4(to_tf32(h[4 * qq]), to_tf32(h[4 * qq + 1]), to_tf32(h[4 * qq + 2]),
                               to_tf32(h[4 * qq + 3])));
        if (jg < Fn) stage_img(c0, h);
      }
      if (ok) {
        tm_wait_st();
        pend_img = img;
        pend_F = Fn;
        pend_j0 = j0h;
        pend_w = hN;
      }
    } else {
      // loss head over the whole last layer (both CTAs hold it): rank r takes lane
      // quarters 2r and 2r + 1; the four warps of a quarter share each row, one 16-column
      // block in four each, and the row's max, sum, entropy, chosen log-probability and
      // value meet in a scratch (the A buffer past G's columns), in a fixed order
      const bool mine = ok && (quarter >> 1) == rank;
      const int NA = a.n_actions;
      const int Wg = P.Gk[l], Fg = P.Fg[l];
      float* red = reinterpret_cast<float*>(s.abuf + P.hs_off);   // [4][128]
      float* lz = red + 4 * kR;                                     // [2][128]
      float mloc = -__uint_as_float(0x7F800000u);
      for (int c0 = 16 * cq; mine && c0 < NA; c0 += 64) {
        float z[16];
        ld16(c0, Nl, z);
#pragma unroll
        for (int i = 0; i < 16; ++i)
          if (c0 + i < NA) mloc = fmaxf(mloc, z[i] + bias[c0 + i]);
      }
      red[cq * kR + r] = mloc;
      __syncthreads();
      const float m = fmaxf(fmaxf(red[r], red[kR + r]), fmaxf(red[2 * kR + r], red[3 * kR + r]));
      __syncthreads();
      float sloc = 0.0f;
      for (int c0 = 16 * cq; mine && c0 < NA; c0 += 64) {
        float z[16];
        ld16(c0, Nl, z);
#pragma unroll
        for (int i = 0; i < 16; ++i)
          if (c0 + i < NA) sloc += __expf(z[i] + bias[c0 + i] - m);
      }
      red[cq * kR + r] = sloc;
      __syncthreads();
      const float Ssum = ((red[r] + red[kR + r]) + red[2 * kR + r]) + red[3 * kR + r];
      const float lse = m + __logf(Ssum);
      __syncthreads();
      float hloc = 0.0f;
      for (int c0 = 16 * cq; mine && c0 < Nl; c0 += 64) {
        float z[16];
        ld16(c0, Nl, z);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int j = c0 + i;
          if (j < NA) {
            const float lp = z[i] + bias[j] - lse;
            hloc -= __expf(lp) * lp;
            if (j == ac) lz[r] = lp;
          } else if (j == NA && j < Nl) {
            lz[kR + r] = z[i] + bias[j];
          }
        }
      }
      red[cq * kR + r] = hloc;
      __syncthreads();
      if (mine) {
        const float Hent = ((red[r] + red[kR + r]) + red[2 * kR + r]) + red[3 * kR + r];
        const float lpa = lz[r];
        const float zv = Nl > NA ? lz[kR + r] : 0.0f;
        float coef = 0.0f, dv = 0.0f;
        if (live) {
          float pg;
          double cf = 0.0;
          if (a.algo == SIMX_ALGO_REINFORCE) {
            coef = adv;
            pg = -adv * lpa;
          } else {
            const float rho = __expf(lpa - lpo);
            const float s1 = rho * adv;
            const float s2 = fminf(fmaxf(rho, 1.0f - a.clip_eps), 1.0f + a.clip_eps) * adv;
            pg = -fminf(s1, s2);
            coef = (s1 <= s2 ? adv : 0.0f) * rho;
            cf = fabsf(rho - 1.0f) > a.clip_eps ? 1.0 : 0.0;
          }
          if (a.has_value) dv = zv - ret;
          if (cq == 0) {   // one thread per row keeps the row's statistics
            st_cf += cf;
            st_v += (double)dv * (double)dv;
            st_pg += pg;
            st_h += Hent;
          }
        }
        // G_{L-1} of this CTA's rows: TF32 into both A buffers (width Gk), FP32 into the
        // G image
        unsigned char* img = A.ws + P.img_g[l] + img_blk(grow, Fg);
        for (int c0 = 16 * cq; c0 < Wg; c0 += 64) {
          float z[16], bv[16], g[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) bv[i] = c0 + i < NA ? bias[c0 + i] : 0.0f;
          ld16(c0, Nl, z);
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const int j = c0 + i;
            float v = 0.0f;
            if (live && j < NA) {
              const float lp = z[i] + bv[i] - lse;
              const float p = __expf(lp);
              const float onehot = (j == ac) ? 1.0f : 0.0f;
              v = (-coef * (onehot - p) + a.c_entropy * p * (lp + Hent)) * inv_n;
            } else if (live && a.has_value && j == NA) {
              v = 2.0f * a.c_value * dv * inv_n;
            }
            g[i] = v;
          }
#pragma unroll
          for (int qq = 0; qq < 4; ++qq)
            put_both(rm_off(r, c0 + 4 * qq, Wg),
                     make_float4(to_tf32(g[4 * qq]), to_tf32(g[4 * qq + 1]), to_tf32(g[4 * qq + 2]),
                                 to_tf32(g[4 * qq + 3])));
          if (c0 < Fg) stage_img(c0, g);
        }
        tm_wait_st();
        pend_img = img;
        pend_F = Fg;
        pend_j0 = 0;
        pend_w = Wg;
      }
    }
    cluster_sync();
  }
  // ---- backward: dH_l = G_l W_l, G_{l-1} = dH_l (1 - H_l^2), this CTA's half of dH_l
  for (int l = L - 1; l >= 1; --l) {
    const int hK = P.hK[l];
    gemm(2 * L - 1 - l, P.Gk[l], hK);
    const bool ok = *s.abort_flag == 0;
    const int Kl = P.K[l], Fh = P.Fh[l], Fg = P.Fg[l - 1];
    const int Wg = l - 1 >= 1 ? P.Gk[l - 1] : 0;
    const int j0h = rank * hK;
    const unsigned char* himg = A.ws + P.img_h[l] + img_blk(grow, Fh);
    unsigned char* gimg = A.ws + P.img_g[l - 1] + img_blk(grow, Fg);
    uint32_t u[16];
    if (ok && 16 * cq < hK) tm_ld16_nw(tl + (uint32_t)(16 * cq), u);
    for (int c0 = 16 * cq; ok && c0 < hK; c0 += 64) {
      const int jg = j0h + c0;
      float z[16], hv[16], g[16];
      if (jg < Fh) img_load16(himg, jg, hv, lane);
      else
#pragma unroll
        for (int i = 0; i < 16; ++i) hv[i] = 0.0f;
      tm_wait();
      reg_fence16(u);
#pragma unroll
      for (int i = 0; i < 16; ++i) z[i] = jg + i < Kl ? __uint_as_float(u[i]) : 0.0f;
      if (c0 + 64 < hK) tm_ld16_nw(tl + (uint32_t)(c0 + 64), u);
#pragma unroll
      for (int i = 0; i < 16; ++i) g[i] = jg + i < Kl ? z[i] * (1.0f - hv[i] * hv[i]) : 0.0f;
      if (jg < Wg)
#pragma unroll
        for (int qq = 0; qq < 4; ++qq)
          put_both(rm_off(r, jg + 4 * qq, Wg),
                   make_float4(to_tf32(g[4 * qq]), to_tf32(g[4 * qq + 1]), to_tf32(g[4 * qq + 2]),
                               to_tf32(g[4 * qq + 3])));
      if (jg < Fg) stage_img(c0, g);
    }
    if (ok) {
      tm_wait_st();
      pend_img = gimg;
      pend_F = Fg;
      pend_j0 = j0h;
      pend_w = hK;
    }
    if (Wg) cluster_sync();   // G_0 is not an operand here: nothing went to the peer
  }
  flush();   // G_0's image rows

  // ---- end: nothing in flight, statistics of the CTA's rows, tensor memory released
  if (tid == 0) drain_loads(s, S, issued);
  if (tid == 32) drain_mma(s);
  if (cq == 0) {
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) {
      st_pg += __shfl_xor_sync(0xFFFFFFFFu, st_pg, d);
      st_v += __shfl_xor_sync(0xFFFFFFFFu, st_v, d);
      st_h += __shfl_xor_sync(0xFFFFFFFFu, st_h, d);
      st_cf += __shfl_xor_sync(0xFFFFFFFFu, st_cf, d);
    }
    if (lane == 0) {
      s.dstat[4 * warp + 0] = st_pg;
      s.dstat[4 * warp + 1] = st_v;
      s.dstat[4 * warp + 2] = st_h;
      s.dstat[4 * warp + 3] = st_cf;
    }
  }
  fence_before();
  __syncthreads();
  if (tid < 4) {
    const double v = s.dstat[tid] + s.dstat[4 + tid] + s.dstat[8 + tid] + s.dstat[12 + tid];
    double* sp = reinterpret_cast<double*>(A.ws + P.spart);
    sp[(size_t)blockIdx.x * 4 + tid] = *s.abort_flag == 0 ? v : __longlong_as_double(0x7FF8000000000000LL);
  }
  if (warp == 0) {
    fence_after();
    tm_dealloc(tmem, (uint32_t)P.tcols);
  }
}

// ---------------------------------------------------------------------------------
// k_lw_dw: [dW_l | db_l] of one block of 128 outputs of layer l over one row range.
// ---------------------------------------------------------------------------------
__global__ void __launch_bounds__(kDwThreads, 1) k_lw_dw(const __grid_constant__ Args A) {
  extern __shared__ __align__(1024) unsigned char sm[];
  const Plan& P = A.p;
  const int S = P.dw_nstages, SB = P.dw_stage_bytes;
  // the first 2 KB hold one mbarrier per stage on which the db warps release it
  const Smem s = carve(sm, P, SB, S, 2048);
  uint64_t* dbe = reinterpret_cast<uint64_t*>(sm);
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int quarter = warp & 3, cq = warp >> 2;
  const int item = blockIdx.x % P.mt_total, split = blockIdx.x / P.mt_total;
  int l = 0;
  while (l + 1 < P.L && P.mt0[l + 1] <= item) ++l;
  const int mt = item - P.mt0[l];
  const int64_t c_lo = (int64_t)split * P.nchunks / P.S, c_hi = (int64_t)(split + 1) * P.nchunks / P.S;
  const int nc = (int)(c_hi - c_lo);
  const int Fh = P.Fh[l], Fg = P.Fg[l];
  const int ng = (Fg >> 3) - 16 * mt < 16 ? (Fg >> 3) - 16 * mt : 16;   // feature groups of G
  const uint32_t aA = (uint32_t)ng * 1024u, bB = (uint32_t)Fh * 128u;

  if (tid == 0) {
    for (int i = 0; i < kMaxStages; ++i) {
      mbar_init(&s.full[i], 1);
      mbar_init(&s.mmab[i], 1);
    }
    mbar_init(s.drain, 1);
    mbar_init(s.accb, 1);
    for (int i = 0; i < kMaxStages; ++i) mbar_init(&dbe[i], kDwThreads / 32 - 4);
    mbar_fence_init();
    *s.abort_flag = 0;
  }
  if (warp == 0) tm_alloc(s.tbase, (uint32_t)P.dw_tcols);
  // launched while k_lw_rows runs: the images it writes are read only after this wait
  asm volatile("griddepcontrol.wait;" ::: "memory");
  fence_async_smem();
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *s.tbase;
  int issued = 0;

  // thread 0 streams the row chunks of G and H through the stages, each refilled once the
  // MMAs that read it completed and the db warps released it; thread 32 queues each
  // chunk's dW MMAs as it lands; warps 4 .. 7 add the chunk's G rows into db_l (one thread
  // per output, rows in order: db = G^T 1 in FP32 on the CUDA cores, beside the MMAs)
  float db = 0.0f;
  const int jl = tid - 128;   // db warps: this thread's output in the block
  if (warp == 0 && lane == 0 && nc > 0) {
    const unsigned char* gsrc = A.ws + P.img_g[l];
    const unsigned char* hsrc = A.ws + P.img_h[l];
    for (int c = 0; c < nc; ++c) {
      const int st = c % S;
      const uint32_t par = (uint32_t)(((c - S) / S) & 1);
      if (c >= S && (!mbar_wait(&s.mmab[st], par, kWaitCycles) || !mbar_wait(&dbe[st], par, kWaitCycles))) {
        *s.abort_flag = 1;
        break;
      }
      const int64_t rc = c_lo + c;
      unsigned char* dst = s.stages + (size_t)st * SB;
      mbar_arrive_expect_tx(&s.full[st], aA + bB);
      bulk_g2s(dst, gsrc + (size_t)(rc * (Fg >> 3) + 16 * mt) * 1024, aA, &s.full[st]);
      bulk_g2s(dst + 16384, hsrc + (size_t)rc * (Fh >> 3) * 1024, bB, &s.full[st]);
      issued = c + 1;
    }
  } else if (warp == 1 && lane == 0 && nc > 0) {
    const uint32_t idw = idesc_tf32(kR, Fh);
    bool fine = true;
    for (int c = 0; c < nc; ++c) {
      const int st = c % S;
      if (!mbar_wait(&s.full[st], (uint32_t)((c / S) & 1), kWaitCycles)) {
        fine = false;
        break;
      }
      fence_after();
      const uint32_t sa = su32(s.stages + (size_t)st * SB), sb = sa + 16384;
#pragma unroll
      for (int ks = 0; ks < kKC / 8; ++ks) {
        const uint64_t ad = sdesc(sa + (uint32_t)ks * 256u, 128, 1024);
        const uint32_t acc = (c | ks) ? 1u : 0u;
        mma_tf32(tmem, ad, sdesc(sb + (uint32_t)ks * 256u, 128, 1024), idw, acc);
      }
      commit(&s.mmab[st]);
    }
    if (fine) commit(s.accb);
    else *s.abort_flag = 1;
  } else if (warp >= 4 && nc > 0) {
    // output jl's 32 rows of a chunk: 8 consecutive 16-byte core-matrix rows of its group
    const uint32_t goff = (uint32_t)((jl >> 3) * 1024 + (jl & 7) * 16);
    for (int c = 0; c < nc; ++c) {
      const int st = c % S;
      if (*s.abort_flag || !mbar_wait_idle(&s.full[st], (uint32_t)((c / S) & 1), kWaitCycles)) {
        atomicOr(s.abort_flag, 1);
        break;
      }
      if (jl < ng * 8) {
        const unsigned char* g = s.stages + (size_t)st * SB + goff;
#pragma unroll
        for (int q = 0; q < kKC / 4; ++q) {
          const float4 v = *reinterpret_cast<const float4*>(g + q * 128);
          db = __fadd_rn(__fadd_rn(__fadd_rn(__fadd_rn(db, v.x), v.y), v.z), v.w);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&dbe[st]);
    }
  }
  __syncwarp();
  if (nc > 0 && !mbar_wait_idle(s.accb, 0u, kWaitCycles)) atomicOr(s.abort_flag, 1);
  fence_after();
  __syncthreads();
  const bool ok = *s.abort_flag == 0;

  // read out: lane m = output j = 128 mt + m; columns k < K_l of dW, column Fh of db.
  // dW goes through a row-major tile in the (now idle) stages, row stride = 4 words past a
  // multiple of 32 (a warp's 16-byte row writes hit every bank once per 8 rows), and then
  // to the partial gradient row by row, a warp writing 128 contiguous bytes at a time.
  const int Kl = P.K[l], Nl = P.N[l];
  const int j = 128 * mt + 32 * quarter + lane;
  float* out = reinterpret_cast<float*>(A.ws + P.part) + (size_t)split * P.n_params + P.poff[l];
  const uint32_t tl = tmem + ((uint32_t)(32 * quarter) << 16);
  const float nanv = __uint_as_float(0x7FC00000u);
  float* tile = reinterpret_cast<float*>(s.stages);
  const int ldt = (Kl + 31) / 32 * 32 + 4;
  float* trow = tile + (size_t)(32 * quarter + lane) * ldt;
  for (int c0 = 16 * cq; c0 < Fh; c0 += 32) {
    uint32_t u[4][4];
#pragma unroll
    for (int q = 0; q < 4; ++q) tm_ld4_nw(tl + (uint32_t)(c0 + 4 * q), u[q]);
    tm_wait();
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      reg_fence(u[q]);
      const int k = c0 + 4 * q;
      if (k < Kl) {
        float4 v;
        v.x = nc == 0 ? 0.0f : (ok ? __uint_as_float(u[q][0]) : nanv);
        v.y = nc == 0 ? 0.0f : (ok ? __uint_as_float(u[q][1]) : nanv);
        v.z = nc == 0 ? 0.0f : (ok ? __uint_as_float(u[q][2]) : nanv);
        v.w = nc == 0 ? 0.0f : (ok ? __uint_as_float(u[q][3]) : nanv);
        *reinterpret_cast<float4*>(trow + k) = v;
      }
    }
  }
  __syncthreads();
  {
    const int rows = Nl - 128 * mt < 128 ? Nl - 128 * mt : 128;
    float* dst = out + (size_t)(128 * mt) * Kl;
    for (int rr = warp; rr < rows; rr += kDwThreads / 32)
      for (int k = lane; k < Kl; k += 32) dst[(size_t)rr * Kl + k] = tile[(size_t)rr * ldt + k];
  }
  if (warp >= 4 && 128 * mt + jl < Nl)
    out[(size_t)Nl * Kl + 128 * mt + jl] = nc == 0 ? 0.0f : (ok ? db : nanv);
  if (tid == 0) drain_loads(s, S, issued);
  if (tid == 32) drain_mma(s);
  fence_before();
  __syncthreads();
  if (warp == 0) {
    fence_after();
    tm_dealloc(tmem, (uint32_t)P.dw_tcols);
  }
}

// ---------------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------------
size_t al256(size_t x) { return (x + 255) & ~(size_t)255; }

int pow2_cols(int need) {
  int c = 32;
  while (c < need) c *= 2;
  return c;
}

Plan plan(const LossArgs& a) {
  Plan p{};
  p.ok = false;
  const int L = a.n_layers;
  if (L < 2 || L > SIMX_MAX_LAYERS || a.n < 1) return p;
  for (int l = 0; l + 1 < L; ++l)
    if (a.act[l] != 0) return p;  // tanh hidden layers only
  p.L = L;
  int P = 0, maxA = 0, maxB = 0, maxFh = 0, tneed = 0;
  for (int l = 0; l < L; ++l) {
    const int K = a.dims[l], N = a.dims[l + 1];
    if (K < 1 || N < 1 || K > 256 || N > 256) return p;
    p.K[l] = K;
    p.N[l] = N;
    p.Ka[l] = l == 0 ? 3 * r32(K) : r32(K);
    p.Nf[l] = l + 1 < L ? r32(N) : r16(N);
    p.hN[l] = l + 1 < L ? p.Nf[l] / 2 : p.Nf[l];
    p.Gk[l] = r32(N);
    p.Kb[l] = r32(K);
    p.hK[l] = p.Kb[l] / 2;
    p.Fh[l] = r16(K);
    p.Fg[l] = r16(N);
    p.poff[l] = P;
    P += N * K + N;
    maxA = maxA > p.Ka[l] ? maxA : p.Ka[l];
    if (l >= 1) maxA = maxA > p.Gk[l] ? maxA : p.Gk[l];
    maxB = maxB > p.hN[l] ? maxB : p.hN[l];
    if (l >= 1) maxB = maxB > p.hK[l] ? maxB : p.hK[l];
    maxFh = maxFh > p.Fh[l] ? maxFh : p.Fh[l];
    tneed = tneed > p.hN[l] ? tneed : p.hN[l];
    if (l >= 1) tneed = tneed > p.hK[l] ? tneed : p.hK[l];
  }
  p.n_params = P;
  const int limit = 227 * 1024, misc = 256;
  // the head's scratch follows G_{L-1} in the A buffer: make the buffer long enough
  p.hs_off = kR * p.Gk[L - 1] * 4;
  if (maxA < p.Gk[L - 1] + 6) maxA = (p.Gk[L - 1] + 6 + 31) / 32 * 32;
  p.a_bytes = kR * maxA * 4;
  p.stage_bytes = maxB * kKC * 4;
  p.nstages = kMaxStages;
  while (p.nstages > 2 && p.a_bytes + p.nstages * p.stage_bytes + misc > limit) --p.nstages;
  // the biases of every layer follow the misc area
  p.b_total = 0;
  for (int l = 0; l < L; ++l) {
    p.b_off[l] = p.b_total;
    p.b_total += (p.N[l] + 15) / 16 * 16;
  }
  while (p.nstages > 2 && p.a_bytes + p.nstages * p.stage_bytes + misc + 4 * p.b_total > limit) --p.nstages;
  p.smem = p.a_bytes + p.nstages * p.stage_bytes + misc + 4 * p.b_total;
  if (p.smem > limit) return p;
  p.tcols = pow2_cols(2 * tneed);   // accumulators, then the staged image rows
  if (p.tcols > 512) return p;
  // weight-gradient products
  p.mt_total = 0;
  for (int l = 0; l < L; ++l) {
    p.mt0[l] = p.mt_total;
    p.mt_total += (p.N[l] + 127) / 128;
  }
  p.n_pad = (a.n + kR - 1) / kR * kR;
  p.ntiles = p.n_pad / kR;
  p.nchunks = p.n_pad / kKC;
  int64_t S = sm_count() / p.mt_total;
  if (S < 1) S = 1;
  if (S > p.nchunks) S = p.nchunks;
  p.S = (int)S;
  p.dw_stage_bytes = 16384 + maxFh * 128;
  p.dw_nstages = 3;
  p.dw_smem = 2048 + p.dw_nstages * p.dw_stage_bytes + misc;
  if (p.dw_smem > limit) return p;
  // the dW read-out tile (128 rows, row stride r32(K) + 4 floats) reuses the stages
  for (int l = 0; l < L; ++l)
    if ((size_t)128 * ((p.K[l] + 31) / 32 * 32 + 4) * 4 > (size_t)p.dw_nstages * p.dw_stage_bytes) return p;
  p.dw_tcols = pow2_cols(maxFh);
  if (p.dw_tcols > 512) return p;
  // workspace
  size_t off = 0;
  for (int l = 0; l < L; ++l) {
    p.wf_elems[l] = (int64_t)(p.Ka[l] / kKC) * p.Nf[l] * kKC;
    p.wb_elems[l] = l >= 1 ? (int64_t)(p.Gk[l] / kKC) * p.Kb[l] * kKC : 0;
    p.wf[l] = off;
    off = al256(off + (size_t)p.wf_elems[l] * 4);
    p.wb[l] = off;
    off = al256(off + (size_t)p.wb_elems[l] * 4);
  }
  for (int l = 0; l < L; ++l) {
    p.img_h[l] = off;
    off = al256(off + (size_t)p.n_pad * p.Fh[l] * 4);
    p.img_g[l] = off;
    off = al256(off + (size_t)p.n_pad * p.Fg[l] * 4);
  }
  p.part = off;
  off = al256(off + (size_t)p.S * p.n_params * 4);
  p.spart = off;
  off = al256(off + (size_t)2 * p.ntiles * 4 * sizeof(double));   // one entry per CTA
  p.total = off;
  p.ok = true;
  return p;
}

}  // namespace lw

bool loss_wide_fits(const LossArgs& a) { return lw::plan(a).ok; }

size_t loss_wide_workspace(const LossArgs& a) {
  const lw::Plan p = lw::plan(a);
  return p.ok ? p.total : 0;
}

cudaError_t launch_loss_wide(const LossArgs& a, void* ws, size_t ws_bytes, cudaStream_t s) {
  const lw::Plan p = lw::plan(a);
  if (!p.ok || ws_bytes < p.total) return cudaErrorInvalidValue;
  lw::Args A{};
  A.a = a;
  A.p = p;
  A.ws = static_cast<unsigned char*>(ws);
  int64_t elems = 0;
  for (int l = 0; l < p.L; ++l) elems += p.wf_elems[l] + p.wb_elems[l];
  int64_t blocks = (elems + 255) / 256;
  const int64_t cap = (int64_t)sm_count() * 4;
  if (blocks > cap) blocks = cap;
  lw::k_lw_prep<<<(unsigned)blocks, 256, 0, s>>>(A);
  // a cluster of two CTAs per 128-row tile
  cudaFuncSetAttribute(lw::k_lw_rows, cudaFuncAttributeMaxDynamicSharedMemorySize, p.smem);
  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3((unsigned)(2 * p.ntiles));
  lc.blockDim = dim3(lw::kThreads);
  lc.dynamicSmemBytes = (size_t)p.smem;
  lc.stream = s;
  // rows and dW are launched as programmatic dependents of the kernel before them: their
  // prologues overlap its tail and griddepcontrol.wait orders the data
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = 2;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[1].val.programmaticStreamSerializationAllowed = 1;
  lc.attrs = at;
  lc.numAttrs = 2;
  cudaError_t e = cudaLaunchKernelEx(&lc, lw::k_lw_rows, A);
  if (e != cudaSuccess) return e;
  cudaFuncSetAttribute(lw::k_lw_dw, cudaFuncAttributeMaxDynamicSharedMemorySize, p.dw_smem);
  lc.gridDim = dim3((unsigned)(p.mt_total * p.S));
  lc.blockDim = dim3(lw::kDwThreads);
  lc.dynamicSmemBytes = (size_t)p.dw_smem;
  lc.attrs = at + 1;
  lc.numAttrs = 1;
  e = cudaLaunchKernelEx(&lc, lw::k_lw_dw, A);
  if (e != cudaSuccess) return e;
  count_launches(3);
  launch_loss_reduce_n(reinterpret_cast<const float*>(A.ws + p.part), p.S, p.n_params,
                       reinterpret_cast<const double*>(A.ws + p.spart), (int)(2 * p.ntiles), a, s);
  return cudaGetLastError();
}

}  // namespace simx
