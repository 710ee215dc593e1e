/*
 * simx.h — C ABI of libsimx.so, the GB300 (sm_103a) batched rollout engine for
 * "Adaptive Inference Batching using Policy Gradients".
 *
 * The library runs thousands of independent copies of the paper's discrete-event
 * inference-serving simulator (Sec. 3.1, Sec. 3.2) in lockstep on one GPU, evaluates the
 * policy network of Sec. 4.2 fused into the step, and computes the REINFORCE returns,
 * GAE advantages and REINFORCE / PPO loss gradients of Sec. 4.3 over the rollout buffer.
 *
 * Conventions shared by every entry point
 *   - Every pointer argument whose name starts with d_ (and every pointer inside
 *     simx_mlp / simx_rollout) is DEVICE memory owned by the caller; the library
 *     never frees it.  Host pointers are marked "host".
 *   - `stream` is a cudaStream_t passed as void*; NULL is the legacy default stream.
 *     Calls are asynchronous on it; only sim_stats, sim_save, sim_load and
 *     simx_last_status synchronise.
 *   - Argument errors are detected on the host before any launch and returned as
 *     a simx_status; nothing throws across the ABI.  simx_last_error() returns a
 *     human-readable message for the last failure on the calling thread.
 *   - Device-side errors (time overflow, event-loop cap, invalid external action)
 *     never trap: they set a per-env status word, visible through
 *     simx_last_status() and sim_save().
 *   - Layouts are time-major: a [H][E] array holds step t of env e at t*ld + e and
 *     observations are [H][D][E] (feature d of env e at step t at (t*D + d)*ld + e).
 *   - Time inside the simulator is an unsigned 32-bit count of microseconds; any
 *     time that would reach 2^31 us sets SIMX_DEV_TIME_OVERFLOW.
 *
 * The meaning of every field below is the executable specification the oracle
 * (a separate single-threaded C program) implements independently.
 */
#ifndef SIMX_H
#define SIMX_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SIMX_ABI_VERSION 5u
#define SIMX_MAX_TYPES 2
#define SIMX_MAX_SERVERS 8
#define SIMX_MAX_BSIZES 8
#define SIMX_MAX_LAYERS 6
#define SIMX_MAX_WIDTH 256      /* widest hidden layer */
#define SIMX_MAX_OUT 257        /* widest output layer: actions + value row */
#define SIMX_MAX_OBS 64
#define SIMX_DIURNAL_MAX 128
#define SIMX_STATE_HEADER_WORDS 32
#define SIMX_TRACE_WIDTH 4

typedef enum {
  SIMX_OK = 0,
  SIMX_EINVAL = 1,     /* invalid argument or configuration (host-side check) */
  SIMX_ENOMEM = 2,     /* device or host allocation failed in sim_create */
  SIMX_ECUDA = 3,      /* a CUDA runtime call failed (message has the CUDA error) */
  SIMX_EOVERFLOW = 4,  /* an env raised a device status flag (see SIMX_DEV_*) */
  SIMX_ESTATE = 5      /* call out of order (e.g. step before reset) */
} simx_status;

/* Per-env device status bits (OR-ed into the env's status word). */
#define SIMX_DEV_TIME_OVERFLOW 1u   /* a simulated time reached 2^31 us */
#define SIMX_DEV_EVENT_CAP 2u       /* more than 2^20 arrival candidates in one decision */
#define SIMX_DEV_BAD_ACTION 4u      /* external action outside [0, n_actions): action 0 used */
#define SIMX_DEV_TC_TIMEOUT 8u      /* a wait for the tensor-core policy forward timed out */
#define SIMX_DEV_COPY_TIMEOUT 16u   /* a wait for a staged copy of the policy weights timed out */

/* Simulator mode (Sec. 3.1 "Multi-GPU Support"; Sec. 4.1 action space). */
typedef enum {
  SIMX_MODE_SINGLE = 0,  /* one server; a decision whenever it is free and work is queued;
                            action = (type to serve, batch size)                          */
  SIMX_MODE_ROUTE = 1    /* K servers; one decision per arriving request;
                            action = (target server, that server's batch size)            */
} simx_mode;

/* Arrival process (Sec. 3.2 workloads). */
typedef enum {
  SIMX_ARR_THINNED = 0,  /* Poisson candidate stream thinned by a 1- or 2-state modulating
                            chain: Poisson when n_mod_states = 1, MMPP when 2            */
  SIMX_ARR_DIURNAL = 1,  /* piecewise-constant rate per epoch: diurnal table x lognormal
                            burst factor; a synthetic stand-in for a trace               */
  SIMX_ARR_TRACE = 2     /* trace replay (Sec. 3.2 real-world traces): as THINNED, but the
                            gap before candidate j, and optionally its type and cost,
                            come from entry j mod n of the trace given by sim_set_trace  */
} simx_arrival_kind;

/* Action selection (Sec. 4.2 stochastic policy; Sec. 5.1 baselines). */
typedef enum {
  SIMX_POLICY_SAMPLE = 0,   /* categorical sample from softmax(logits)                   */
  SIMX_POLICY_ARGMAX = 1,   /* first index of the largest logit                          */
  SIMX_POLICY_STATIC = 2,   /* single mode: oldest-head type, batch bsizes[static_bi]     */
  SIMX_POLICY_RR = 3,       /* route mode: server t mod K, batch bsizes[static_bi]        */
  SIMX_POLICY_SQ = 4,       /* route mode: server with fewest queued requests             */
  SIMX_POLICY_RANDOM = 5,   /* uniform action from the POLICY Philox stream              */
  SIMX_POLICY_EXTERNAL = 6  /* sim_step_batched only: caller-supplied actions            */
} simx_policy_mode;

/*
 * Environment configuration (plain data, copied by sim_create).
 * Every numeric value enters the simulator exactly as given; nothing here is
 * recomputed by the library, so the same struct fed to the oracle fixes every bit.
 */
typedef struct simx_config {
  uint32_t abi_version;        /* must be SIMX_ABI_VERSION */
  uint32_t mode;               /* simx_mode */
  uint32_t n_envs;             /* E, 1 .. 2^24 */
  uint32_t n_servers;          /* K: 1 in SINGLE mode, 1..SIMX_MAX_SERVERS in ROUTE mode */
  uint32_t n_types;            /* request types (Sec. 3.1 model type m_i): 1 or 2 */
  uint32_t queue_cap;          /* FIFO capacity per (server, type); power of two <= 4096;
                                  arrivals to a full queue are dropped (Sec. 3.1 Queuing) */
  uint32_t episode_len;        /* done[t] = 1 when (global step + 1) % episode_len == 0 */
  uint32_t arrival_kind;       /* simx_arrival_kind */
  /* THINNED: candidates at i.i.d. exponential gaps, accepted with probability
     accept_thr[state] / 2^24 where state is the modulating chain's state */
  float    cand_mean_gap_us;   /* mean candidate gap (1e6 / max rate) */
  uint32_t n_mod_states;       /* 1 (Poisson) or 2 (two-state MMPP) */
  uint32_t accept_thr[2];      /* acceptance threshold per state, out of 2^24 */
  float    dwell_mean_us;      /* mean exponential dwell of the modulating chain */
  /* DIURNAL: rate(epoch) = diurnal_rate[(epoch + offset_env) % diurnal_len] * exp(sigma Z) */
  uint32_t epoch_us;           /* epoch length */
  uint32_t diurnal_len;        /* 1 .. SIMX_DIURNAL_MAX */
  float    diurnal_rate[SIMX_DIURNAL_MAX]; /* base arrival rate per epoch slot, requests/s */
  float    burst_sigma;        /* lognormal sigma of the per-epoch burst factor */
  /* request types and the execution model L = alpha + beta * n (Sec. 3.1) */
  uint32_t type0_thr;          /* P(type 0) * 2^24 */
  uint32_t alpha_us[SIMX_MAX_TYPES];
  uint32_t beta_us[SIMX_MAX_TYPES];
  int32_t  cost_type;          /* type whose batch time is alpha + the sum of per-request
                                  costs drawn at arrival (-1: none; beta then unused) */
  uint32_t cost_kind;          /* 0: Pareto(x_m = cost_scale_us, shape 1/pareto_inv_alpha);
                                  1: exponential with mean cost_scale_us */
  float    cost_scale_us;
  float    pareto_inv_alpha;
  /* reward (Sec. 4.1): r = n_dispatched - sum_type w_wait[type] * queueing_us */
  float    w_wait[SIMX_MAX_TYPES];
  /* actions (Sec. 4.1): a = major * n_bsizes + i, major = type (SINGLE) or server (ROUTE) */
  uint32_t n_bsizes;
  uint32_t bsizes[SIMX_MAX_BSIZES];
  uint32_t static_bi;          /* batch-size index of the policy-free baselines and the
                                  initial per-server batch size in ROUTE mode */
  /* observation (Sec. 4.1 state) */
  uint32_t obs_extra;          /* append the extra features (see obs layout below) */
  uint32_t obs_dim;            /* must equal simx_obs_dim(cfg) */
  float    t_window_us;        /* time normaliser T_window */
  float    rate_scale;         /* SINGLE: rate feature = n_arrivals * rate_scale / dt_us */
  float    rate_ref;           /* ROUTE: EWMA rate normaliser and its initial value */
  float    busy_norm_us;       /* ROUTE: busy-remaining normaliser */
  uint32_t phase_period_us;    /* ROUTE extra: diurnal phase period */
  /* workload variants (Sec. 3.1 K heterogeneous GPUs; Sec. 3.2 Extreme Burst) */
  uint32_t dwell_kind;         /* 0: exponential dwell of mean dwell_mean_us; 1: fixed dwell of
                                  round(dwell_mean_us) (a square wave between the two rates) */
  uint32_t srv_speed16[SIMX_MAX_SERVERS]; /* batch time factor of server k in 1/16 (0 means 16):
                                  L_k = (L * s_k + 8) / 16 in integer microseconds, 1 .. 255 */
  uint32_t action_layout;      /* 0: a = major * n_bsizes + i, batch bsizes[i];
                                  1 (SINGLE only; Sec. 4.1 action 0 = Wait): a = 0 waits (no
                                  dispatch; the next decision is at the next arrival), a >= 1 is
                                  type (a-1) / n_bsizes with batch ((a-1) % n_bsizes) + 1;
                                  n_bsizes <= 64, static batch static_bi + 1.  Actions:
                                  1 + T * n_bsizes (33 for T = 1, 65 for T = 2 at n_bsizes 32) */
} simx_config;

/* Activation after a hidden layer (simx_mlp.act). */
typedef enum { SIMX_ACT_TANH = 0, SIMX_ACT_IDENTITY = 1, SIMX_ACT_GELU = 2 } simx_act;

/*
 * Policy network (Sec. 4.2): an MLP.  Layer l maps dims[l] -> dims[l+1] with
 * z_j = (sum_k W_l[j][k] x_k, accumulated in fp32 by fused multiply-adds in k order
 * from k = 0) + b_l[j]; every layer but the last applies act[l]: tanh (the default, 0),
 * identity, or GELU in its tanh form, 0.5 z (1 + tanh(c (z + 0.044715 z^3))),
 * c = sqrt(2/pi), evaluated as u = fma(0.044715, (z*z)*z, z), t = tanh(c*u),
 * (0.5*z)*(1 + t) with the library's deterministic tanh.  The last layer has n_actions
 * rows followed by one value row when has_value.  The paper's network (projection,
 * 2-head attention over its single token, GELU policy and value heads) is such an MLP:
 * attention over one token is a linear map, and separate heads are one hidden layer with
 * zero blocks in the output layer.  W_l is row-major [dims[l+1]][dims[l]] fp32, device
 * memory.
 *
 * Grid policy (grid != 0; the exact policy forward): the input of layer l is first put
 * on the grid 2^-gx[l] (0 <= gx[l] <= 24) by Q(v, e) = clamp(rint(v 2^e), -255, 255) 2^-e,
 * ties to even, for finite v (infinities clamp; NaN is not an input): the observation
 * for l = 0, the activated hidden output of layer l - 1 otherwise; the output layer is
 * not rounded.  When the caller's weights lie on a grid
 * 2^-e_w with integer mantissas |m| <= 255, the biases on 2^-(gx[l] + e_w) with |m| <=
 * 2^16, and every fan-in is <= 256, each pre-activation is an exact fp32 value (the exact
 * dot product plus bias), identical under any summation order; the library does not read
 * the weights back to check this.  Grid policies run in rollout_collect, sim_step_batched
 * and policy_forward.  The loss-gradient entry points take them on their FP32 fused path
 * whatever the precision asked for: the forward rounds the observation and the hidden
 * outputs as above, the gradient passes every rounding unchanged (straight through:
 * dQ(a)/da = 1, the activation's derivative taken at the pre-activation), and the weight
 * gradients use the rounded layer inputs.  A grid policy too large for that path (its
 * per-tile activations and parameters must fit one SM's shared memory: c2 and c3 / c5
 * sizes do, c4's does not) is rejected with SIMX_EINVAL.
 */
typedef struct simx_mlp {
  int32_t n_layers;                     /* 1 .. SIMX_MAX_LAYERS */
  int32_t dims[SIMX_MAX_LAYERS + 1];
  const float* W[SIMX_MAX_LAYERS];
  const float* b[SIMX_MAX_LAYERS];
  int32_t has_value;
  int32_t act[SIMX_MAX_LAYERS];         /* simx_act after layer l < n_layers - 1 */
  int32_t grid;                         /* 0: plain fp32 policy; 1: grid policy */
  int32_t gx[SIMX_MAX_LAYERS];          /* grid policy: input grid exponent of layer l */
} simx_mlp;

/* Rollout buffer (device memory, caller-owned).  ld >= n_envs is the env stride. */
typedef struct simx_rollout {
  int64_t  ld;
  float*   obs;      /* [H][obs_dim][ld] observation at each decision */
  uint8_t* action;   /* [H][ld] action index */
  float*   logp;     /* [H][ld] log pi(a|s) (0 for policy-free modes); may be NULL */
  float*   value;    /* [H][ld] value head output; NULL unless has_value */
  float*   reward;   /* [H][ld] reward of the step */
  uint8_t* done;     /* [H][ld] segment end flag */
  int64_t* trace;    /* [H][SIMX_TRACE_WIDTH][ld] or NULL: decision time (us), requests
                        dispatched in the step, their summed queueing us, requests queued
                        after the decision */
} simx_rollout;

/* Loss selection for ppo_loss_grad (Sec. 4.3). */
typedef enum { SIMX_ALGO_REINFORCE = 0, SIMX_ALGO_PPO = 1 } simx_algo;

/* Arithmetic of the loss-gradient products (the paper fixes none; Sec. 4.3 trains in
   PyTorch's default fp32).  SIMX_PREC_FP32: FP32 fused multiply-adds on the CUDA cores
   (within 1e-5 of the fp64 definition).  SIMX_PREC_TF32: the matrix products on the
   tensor cores with TF32 inputs (rounded to nearest) and FP32 accumulation, within 1e-2;
   policies too wide for the tensor-core kernel (a layer wider than 128 outputs, or
   operands beyond one SM's shared memory) silently take the FP32 path. */
typedef enum { SIMX_PREC_FP32 = 0, SIMX_PREC_TF32 = 1 } simx_precision;

typedef struct simx_loss_params {
  int32_t algo;        /* simx_algo */
  float   clip_eps;    /* PPO clip range epsilon */
  float   c_value;     /* value-loss coefficient (used when the MLP has a value row) */
  float   c_entropy;   /* entropy bonus coefficient */
  int32_t precision;   /* simx_precision */
} simx_loss_params;

/* Aggregate counters over all envs (sim_stats). */
typedef struct simx_counters {
  uint64_t arrived, dropped, dispatched, batches, queued, sum_wait_us, decisions;
  uint32_t envs_flagged;     /* envs whose status word is non-zero */
  uint32_t status_or;        /* OR of all env status words */
} simx_counters;

typedef struct simx_ctx simx_ctx;

/* Observation width implied by a configuration (0 if the configuration is invalid):
   SINGLE: 2T + 6 (+6 with obs_extra); ROUTE: 3K + 1 (+3 with obs_extra). */
uint32_t simx_obs_dim(const simx_config* cfg);
/* Words of one env's canonical state image (sim_save layout). */
uint64_t simx_state_words(const simx_config* cfg);

/* Create a simulator context on `device`: validates cfg, allocates the SoA env state
   and FIFO rings in device memory (owned by the context).  *out is NULL on error. */
simx_status sim_create(const simx_config* cfg, int device, simx_ctx** out);
void sim_destroy(simx_ctx* ctx);

/*
 * Trace replay input (Sec. 3.2: the paper replays Azure Functions and BurstGPT traces;
 * no trace ships with this library, the caller supplies one in this format).
 *   d_gap_us [n]  : gap in integer us between request i - 1 and request i of the trace
 *                   (absolute timestamps t_i give gap_i = t_i - t_{i-1}; gap_0 is the
 *                   gap taken when the replay wraps from entry n - 1 back to entry 0);
 *   d_type [n]    : request type (values >= n_types count as n_types - 1), or NULL to
 *                   draw types as THINNED does (type0_thr);
 *   d_cost_us [n] : per-request cost in us for requests of cfg.cost_type, or NULL to
 *                   draw costs as THINNED does (cost_kind, cost_scale_us).
 * Env e replays the trace from entry o_e = floor(u * n / 2^32), u the third word of its
 * INIT draw, so envs see different windows of one trace; candidate j of an env uses
 * entry j mod n with its candidate counter starting at o_e (32-bit, wrapping).  The
 * thinning and the modulating chain of THINNED still apply on top (accept_thr[s] =
 * 2^24 keeps every entry).  Arrays are device memory owned by the caller and must stay
 * valid while the context uses them; the call records the pointers and copies nothing.
 * Required before sim_reset when cfg.arrival_kind == SIMX_ARR_TRACE, refused (EINVAL)
 * for other arrival kinds; 1 <= n < 2^31.  A new trace takes effect at the next reset.
 */
simx_status sim_set_trace(simx_ctx* ctx, const uint32_t* d_gap_us, const uint8_t* d_type,
                          const uint32_t* d_cost_us, uint32_t n);

/* Reset every env to time 0 with empty queues and idle servers, keyed by `seed`
   (Philox key), and advance each to its first decision point.  SIMX_ESTATE for a
   TRACE context without a trace. */
simx_status sim_reset(simx_ctx* ctx, uint64_t seed, void* stream);

/* Write the current observation of every env to d_obs [obs_dim][ld]. */
simx_status sim_observe(simx_ctx* ctx, float* d_obs, int64_t ld, void* stream);

/*
 * One decision step of every env (the gym-style step of Sec. 4.1).
 *   policy_mode == SIMX_POLICY_EXTERNAL: d_actions [E] int32 chosen by the caller;
 *   otherwise the internal policy (pol required for SAMPLE/ARGMAX).
 * Outputs (any may be NULL): d_obs [obs_dim][ld] next observation, d_reward [E],
 * d_done [E], d_action [E] u8 action taken, d_logp [E].
 */
simx_status sim_step_batched(simx_ctx* ctx, const int32_t* d_actions, const simx_mlp* pol,
                             int policy_mode, float* d_obs, int64_t ld, float* d_reward,
                             uint8_t* d_done, uint8_t* d_action, float* d_logp, void* stream);

/*
 * Collect `horizon` decision steps of every env into `out` in one persistent launch:
 * observation, fused policy forward, action, reward, done (Sec. 4.1, Sec. 4.2).
 * Equivalent, bit for bit, to `horizon` calls of sim_step_batched.  The context repacks
 * the policy into a buffer of its own, grown when a larger policy is passed: a CUDA graph
 * that captured a call stays valid while no larger policy is passed to the context.
 */
simx_status rollout_collect(simx_ctx* ctx, const simx_mlp* pol, int policy_mode,
                            int32_t horizon, const simx_rollout* out, void* stream);

/*
 * The launch that rollout_collect and sim_step_batched take for this context, policy and
 * mode (host only: no device work; the lane and block choice follows the device's SM
 * count).  host_out[6] receives: [0] kernel, 0 = the fused step with the policy forward
 * (one group of lanes per env), 1 = the thread-per-env step of the policy-free modes;
 * [1] lanes per env (1 for the thread-per-env step); [2] threads per block; [3] 1 when
 * each warp runs the policy forward for its own envs, 0 for the block-wide forward;
 * [4] 1 when a grid policy's forward runs on the tensor cores (tcgen05, bf16 operands
 * exact on the grid, FP32 accumulation: the FP32 path's bits), 0 otherwise; [5] 1 when
 * the block-wide FP32 forward streams its weights through shared memory (bulk copies
 * into two stages; the same fma chains and bits), 0 otherwise.
 * It exists so that tests and benchmarks can state which instantiation they exercise.
 * SIMX_EINVAL for a NULL argument, an unknown mode or a policy that rollout_collect
 * would refuse.
 */
simx_status simx_launch_shape(simx_ctx* ctx, const simx_mlp* pol, int policy_mode,
                              int32_t* host_out);

/*
 * Batched policy forward (Sec. 4.2) for n observation columns d_obs [dims[0]][ld].
 * Column i is env (env_base + i) at global decision step `step`, which fixes its
 * POLICY Philox counter, so this reproduces the actions the rollout drew.
 * Outputs (any may be NULL): d_logits [n_actions][ld], d_value [ld], d_action [ld] u8,
 * d_logp [ld].  policy_mode: SAMPLE or ARGMAX.
 * The policy is repacked into a buffer the library keeps per device: calls on one device
 * must not overlap on the GPU, and a call with a larger policy replaces the buffer (a
 * CUDA graph that captured an earlier call would then use freed memory).  For concurrent
 * streams or graph capture use policy_forward_ws.
 */
simx_status policy_forward(const simx_mlp* pol, const float* d_obs, int64_t ld, int64_t n,
                           int policy_mode, uint64_t seed, uint32_t step, uint32_t env_base,
                           float* d_logits, float* d_value, uint8_t* d_action, float* d_logp,
                           void* stream);

/* policy_forward with a caller-owned device workspace of policy_forward_workspace_size(pol)
   bytes (16-byte aligned) for the repacked policy: no state shared between calls, so calls
   may run on concurrent streams and inside captured CUDA graphs (the workspace must
   outlive the graph).  SIMX_EINVAL for a short, misaligned or NULL workspace. */
size_t policy_forward_workspace_size(const simx_mlp* pol);
simx_status policy_forward_ws(const simx_mlp* pol, const float* d_obs, int64_t ld, int64_t n,
                              int policy_mode, uint64_t seed, uint32_t step, uint32_t env_base,
                              float* d_logits, float* d_value, uint8_t* d_action, float* d_logp,
                              void* d_workspace, size_t workspace_bytes, void* stream);

/*
 * Returns and advantages over a [T][E] buffer (Sec. 4.3):
 *   lam < 0 : REINFORCE returns G_t = r_t + gamma (1 - d_t) G_{t+1}, G_T = last_value
 *             (d_ret gets G; d_adv may be NULL);
 *   lam >= 0: GAE  delta_t = r_t + gamma (1 - d_t) V_{t+1} - V_t, V_T = last_value,
 *             A_t = delta_t + gamma lam (1 - d_t) A_{t+1}, R_t = A_t + V_t.
 * d_val is required for GAE; d_last_val [E] may be NULL (zeros).  ld >= E.  T == 0 or
 * E == 0 is an empty problem: SIMX_OK, nothing touched (its buffers may be NULL).
 */
simx_status compute_returns_gae(const float* d_rew, const float* d_val, const uint8_t* d_done,
                                const float* d_last_val, int64_t T, int64_t E, int64_t ld,
                                float gamma, float lam, float* d_ret, float* d_adv,
                                void* stream);

/*
 * Mean-return baseline (Sec. 4.3 REINFORCE with a baseline): mean = (1/n) sum x_i,
 * accumulated in fp64; d_adv_out[i] = x_i - mean (fp32); d_mean_out[0] = mean (fp32).
 * d_workspace must hold returns_baseline_workspace_size(n) bytes.
 */
size_t returns_baseline_workspace_size(int64_t n);
simx_status returns_baseline(const float* d_x, int64_t n, float* d_adv_out, float* d_mean_out,
                             void* d_workspace, size_t workspace_bytes, void* stream);

/*
 * Loss and gradient over a minibatch (Sec. 4.3).  Row r of the rollout is
 * (t = r / E, e = r % E) with E = n_rows_per_step; the minibatch is rows d_idx[0..n)
 * (d_idx == NULL: rows 0..n-1).  With pi = softmax(logits):
 *   REINFORCE: L = -mean(adv * log pi(a))
 *   PPO      : rho = exp(log pi(a) - logp_old),
 *              L = -mean(min(rho adv, clip(rho, 1-eps, 1+eps) adv))
 *   both     : + c_value mean((V - ret)^2) (value row only) - c_entropy mean(H[pi]).
 * d_grad [n_params] fp32 is overwritten with dL/dtheta in the order W0,b0,W1,b1,...;
 * d_stats [5] = {L, policy term, mean (V-ret)^2, mean entropy, clip fraction}.
 * d_workspace must hold ppo_loss_grad_workspace_size(pol, n) bytes (the size depends on
 * pol's layer widths and activations, not on its weights).
 */
size_t ppo_loss_grad_workspace_size(const simx_mlp* pol, int64_t n);
simx_status ppo_loss_grad(const simx_mlp* pol, const simx_rollout* buf, int64_t n_rows_per_step,
                          const float* d_ret, const float* d_adv, const int64_t* d_idx, int64_t n,
                          const simx_loss_params* params, float* d_grad, float* d_stats,
                          void* d_workspace, size_t workspace_bytes, void* stream);

/*
 * Allocation-free variant of ppo_loss_grad.  The paper has no counterpart: this is a
 * service of the library for callers that cannot allocate device memory themselves,
 * for instance a plain C host program with no device allocator of its own, or an
 * application that fixes its device-memory budget before it starts.  Instead of a
 * caller workspace it uses a buffer of SIMX_NOALLOC_SCRATCH_BYTES built into the
 * library (a file-scope device array that every GPU which loads the library holds
 * until the process exits); it calls no cudaMalloc or cudaFree.
 *   - Arguments and results are those of ppo_loss_grad.
 *   - A minibatch whose workspace (ppo_loss_grad_workspace_size) exceeds the buffer is
 *     rejected with SIMX_EINVAL and a message giving both sizes.
 *   - The first call on a device looks up the buffer's device address (with that
 *     device current) and keeps it for the device's context; make that first call
 *     before any stream capture.  A device reset (cudaDeviceReset) ends the context
 *     and may move the buffer: the first call in the new context looks the address
 *     up again, so after a reset that call, too, belongs before any capture.
 *   - Each device has its own copy of the buffer, and every call on that device uses
 *     it: calls on the same device that overlap on the GPU (different streams, or
 *     host threads without ordering between them) race and must be ordered by the
 *     caller.  Calls on different devices do not share scratch.  Nothing needs to
 *     start at zero: each call writes all scratch it reads.
 */
#define SIMX_NOALLOC_SCRATCH_BYTES (64u << 20)
simx_status ppo_loss_grad_noalloc(const simx_mlp* pol, const simx_rollout* buf,
                                  int64_t n_rows_per_step, const float* d_ret, const float* d_adv,
                                  const int64_t* d_idx, int64_t n, const simx_loss_params* params,
                                  float* d_grad, float* d_stats, void* stream);

/*
 * Optimiser step of the training loop (Sec. 4.3 trains REINFORCE and PPO; the paper
 * names no optimiser, so this is Adam, Kingma & Ba 2015).  On a flat fp32 parameter
 * vector in the gradient's order (W0, b0, W1, b1, ...; a policy whose W_l, b_l are views
 * into it updates in place):
 *   s   = min(1, max_grad_norm / ||g||_2)  when max_grad_norm > 0, else 1;
 *   m   = beta1 m + (1 - beta1) s g;   v = beta2 v + (1 - beta2) (s g)^2;
 *   p  -= (lr / (1 - beta1^t)) m / (sqrt(v) / sqrt(1 - beta2^t) + eps),
 * for every i with d_mask == NULL or d_mask[i] != 0 (masked entries keep p, m and v:
 * the zero blocks of a block-diagonal head stay zero).  m and v start at zero.
 * ||g||_2 is taken over the unmasked entries.
 * The step number: t >= 1 from the host when d_t is NULL; otherwise d_t is a device
 * int64 counter that the step increments before use (t = ++*d_t, on the stream), so a
 * captured CUDA graph of training steps advances it on every replay.
 * All arrays are device memory of n entries (mask: bytes), owned by the caller;
 * d_workspace holds simx_adam_workspace_size(n) bytes (used when clipping or with d_t).
 * SIMX_EINVAL for n < 1, t < 1 without d_t, NULL arrays, a short workspace or a
 * parameter outside lr >= 0, 0 <= beta < 1, eps > 0.
 */
typedef struct simx_adam_params {
  float lr, beta1, beta2, eps;
  float max_grad_norm;  /* <= 0: no clipping */
} simx_adam_params;
size_t simx_adam_workspace_size(int64_t n);
simx_status simx_adam_step(float* d_params, const float* d_grad, float* d_m, float* d_v,
                           const uint8_t* d_mask, int64_t n, int64_t t, int64_t* d_t,
                           const simx_adam_params* params, void* d_workspace,
                           size_t workspace_bytes, void* stream);

/* Aggregate counters (synchronises the context's last stream). host_out: host. */
simx_status sim_stats(simx_ctx* ctx, simx_counters* host_out);

/* Canonical state images (synchronising).  host_buf: host, n_envs * simx_state_words
   u32 words; env e's image starts at word e * simx_state_words(cfg). */
simx_status sim_save(simx_ctx* ctx, uint32_t* host_buf, uint64_t n_words);
simx_status sim_load(simx_ctx* ctx, const uint32_t* host_buf, uint64_t n_words);

/* OR of all env status words (synchronising).  Returns SIMX_EOVERFLOW if non-zero. */
simx_status simx_last_status(simx_ctx* ctx, uint32_t* device_code);

/* Number of kernels this library has launched in the process so far (all devices);
   a tracing aid: the difference across a region counts the region's launches. */
uint64_t simx_launches(void);

/* FP32 fused multiply-add probe (no counterpart in the paper: the denominator of the FP32
   roofline fractions).  Launches, on `stream`, one block of 256 threads per quarter warp
   slot (4 blocks per SM), each thread running 16 independent FMA chains `iters` long, and
   stores one float per thread into d_sink (device, at least simx_fma_probe_sink_floats()
   floats).  host_flops receives the FLOPs the launch performs (2 per FMA); the caller
   times the launch on the stream.  SIMX_EINVAL for iters < 1 or a NULL pointer. */
simx_status simx_fma_probe(int64_t iters, float* d_sink, double* host_flops, void* stream);
size_t simx_fma_probe_sink_floats(void);

const char* simx_strerror(simx_status s);
const char* simx_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* SIMX_H */
