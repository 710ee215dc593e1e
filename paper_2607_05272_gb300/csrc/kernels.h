// kernels.h — launch interfaces between the C ABI (api.cu) and the kernels.
#pragma once
#include <cuda_runtime.h>

#include <cstdint>

#include "../../include/simx.h"
#include "sim.cuh"

namespace simx {

// Host-side count of kernel launches (every launcher adds its launches).
void count_launches(int n);
// SM count of the current device (grid sizes and lane choices scale with it).
int sm_count();

// The grid policy's forward on the tensor cores inside the fused step (rollout.cu): per
// layer l the weights as bf16 A operands of nmt[l] tiles of 128 outputs x Kp[l] inputs,
// the block's envs (padded to Bn columns) as the bf16 B operand, an FP32 accumulator in
// tensor memory.  Byte offsets are inside the kernel's dynamic shared memory.
struct TcPlan {
  int on;                     // 1: this launch runs the grid forward on the tensor cores
  int Bn;                     // MMA N: the block's envs rounded up to 16
  int Kp[SIMX_MAX_LAYERS];    // layer inputs rounded up to 16
  int nmt[SIMX_MAX_LAYERS];   // tiles of 128 outputs
  uint32_t w_off[SIMX_MAX_LAYERS];
  uint32_t x_off[2];          // the two activation operand buffers (Bn x Kx bf16)
  uint32_t bar_off;           // mbarrier (8 B) and tensor-memory base (4 B)
  int tcols;                  // tensor-memory columns allocated per block
};

struct RolloutArgs {
  simx_config cfg;
  DevState st;
  DevMlp mlp;
  uint32_t key0, key1;
  int policy_mode;
  uint32_t n_actions;
  const int32_t* ext;
  int H;
  int obs_dim;
  int64_t ld;
  float* obs;
  uint8_t* action;
  float* logp;
  float* value;
  float* reward;
  uint8_t* done;
  int64_t* trace;
  float* next_obs;
  int64_t next_ld;
  int maxd4;        // rows of each activation buffer (widest layer, multiple of 4)
  int apad;         // softmax scratch floats per env (multiple of 4)
  int G;            // lanes per env (8, 16 or 32)
  int threads;      // threads per block (64, 128 or 256)
  int bs_pad;       // activation row stride = envs per block + bs_pad (see act_stride_pad)
  int mlp_warp;     // 1: each warp runs the policy for its own envs (see mlp_forward_warp)
  TcPlan tc;        // grid policies: the tensor-core forward (tc.on = 0 otherwise)
  StagePlan stage;  // the forward with staged weights (stage.on = 0 otherwise)
  // trace replay (arrival_kind TRACE): gaps, types (or null), costs (or null), length
  const uint32_t* tr_gap;
  const uint8_t* tr_type;
  const uint32_t* tr_cost;
  uint32_t tr_n;
};

struct PolicyArgs {
  DevMlp mlp;
  const float* obs;
  int64_t ld, n;
  int mode;
  uint32_t key0, key1, step, env_base;
  float* logits;
  float* value;
  uint8_t* action;
  float* logp;
  int maxd4, apad;
  int G, threads;
};

// Padding of the block's activation rows: 4 (16-byte rows) when some layer takes the
// 4-env tiles of mlp_tiles (B envs shared by `threads` threads), else 1.  With 4 envs per block a stride of 8 floats put
// every output group of a warp's stores in one bank (an 8-way conflict); an odd stride
// spreads them over all 32.
int act_stride_pad(const DevMlp& m, int B, int threads);

cudaError_t launch_rollout(const RolloutArgs& a, cudaStream_t s);
// step_thread.cu: one thread per env for the policy-free modes
bool step_thread_supported(const RolloutArgs& a);
cudaError_t launch_step_thread(const RolloutArgs& a, cudaStream_t s);
cudaError_t launch_reset(const RolloutArgs& a, cudaStream_t s);
cudaError_t launch_observe(const RolloutArgs& a, cudaStream_t s);
cudaError_t launch_save(const DevState& st, int32_t cost_type, uint64_t words, uint32_t* out, cudaStream_t s);
cudaError_t launch_load(const DevState& st, int32_t cost_type, uint64_t words, const uint32_t* in, cudaStream_t s);
cudaError_t launch_stats(const DevState& st, unsigned long long* out, cudaStream_t s);
cudaError_t launch_repack(const float* W, const float* b, int N, int K, int Npad, float* Wt, float* bias, cudaStream_t s);
cudaError_t launch_policy_forward(const PolicyArgs& p, cudaStream_t s);
// Sets a.tc (and the activation rows a.maxd4 it needs) when the grid forward of this
// launch can run on the tensor cores; returns the dynamic shared memory of the launch.
size_t plan_tc_forward(RolloutArgs& a, int B);
// The rollout launch's forward plans (the tensor-core grid forward, else the staged
// weights), as launch_rollout makes them; returns the dynamic shared memory.
size_t plan_rollout(RolloutArgs& a);
int choose_lanes(int64_t envs);
int choose_threads(int64_t envs, int G);

// returns.cu
cudaError_t launch_returns_gae(const float* rew, const float* val, const uint8_t* done,
                               const float* last_val, int64_t T, int64_t E, int64_t ld,
                               float gamma, float lam, float* ret, float* adv, cudaStream_t s);
cudaError_t launch_baseline(const float* x, int64_t n, float* adv, float* mean_out, double* ws,
                            int nblocks, cudaStream_t s);
int baseline_blocks(int64_t n);

// loss.cu
struct LossArgs {
  int n_layers, has_value, n_actions;
  int dims[SIMX_MAX_LAYERS + 1];
  const float* W[SIMX_MAX_LAYERS];
  const float* b[SIMX_MAX_LAYERS];
  const float* obs;      // [T][D][E]
  const uint8_t* action; // [T][E]
  const float* logp_old; // [T][E]
  const float* ret;      // [T][E] (value target) or null
  const float* adv;      // [T][E]
  int64_t E;             // rows per step
  const int64_t* idx;    // minibatch rows or null
  int64_t n;
  int algo;
  float clip_eps, c_value, c_entropy;
  float* grad;           // flat gradient
  float* stats;          // [5]
  int precision;         // SIMX_PREC_FP32 (SIMT) or SIMX_PREC_TF32 (tensor cores where it fits)
  int act[SIMX_MAX_LAYERS];  // simx_act after layer l, -1 for the output layer
  int grid;                  // grid policy (the exact forward; straight-through gradient)
  int gx[SIMX_MAX_LAYERS];   // grid policy: input grid exponent of layer l
};
size_t loss_workspace_bytes(const LossArgs& a);
// loss_fused.cu
bool loss_fused_fits(const LossArgs& a);
size_t loss_fused_workspace(const LossArgs& a);
cudaError_t launch_loss_fused(const LossArgs& a, void* ws, size_t ws_bytes, cudaStream_t s);
void launch_loss_reduce(const float* part, int nb, int n_params, const double* spart,
                        const LossArgs& a, cudaStream_t s);
// the same with nbs statistics partials (nb gradient partials summed in order)
void launch_loss_reduce_n(const float* part, int nb, int n_params, const double* spart, int nbs,
                          const LossArgs& a, cudaStream_t s);
// fma_probe.cu
cudaError_t launch_fma_probe(int64_t iters, float* sink, double* flops, cudaStream_t s);

// optim.cu
size_t adam_workspace_bytes(int64_t n);
cudaError_t launch_adam(float* p, const float* g, float* m, float* v, const uint8_t* mask,
                        int64_t n, int64_t t, int64_t* d_t, float lr, float b1, float b2,
                        float eps, float max_norm, void* ws, cudaStream_t s);
size_t fma_probe_sink_floats();
// loss_tc.cu
bool loss_tc_fits(const LossArgs& a);
size_t loss_tc_workspace(const LossArgs& a);
cudaError_t launch_loss_tc(const LossArgs& a, void* ws, size_t ws_bytes, cudaStream_t s);
// loss_wide.cu
bool loss_wide_fits(const LossArgs& a);
size_t loss_wide_workspace(const LossArgs& a);
cudaError_t launch_loss_wide(const LossArgs& a, void* ws, size_t ws_bytes, cudaStream_t s);
cudaError_t launch_loss_grad(const LossArgs& a, void* ws, size_t ws_bytes, cudaStream_t s);

}  // namespace simx
