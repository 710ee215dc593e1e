/*
 * oracle.h — the reference (test infrastructure only) for the rollout engine.
 *
 * A plain, slow, single-threaded CPU implementation of the discrete-event
 * inference-serving simulator of "Adaptive Inference Batching using Policy
 * Gradients" (Sec. 3.1 dynamics, Sec. 3.2 workloads, Sec. 4.1 MDP) and its policy
 * (Sec. 4.2), written from the paper and its resolved readings.  Only the test
 * suite, the package's smoke check and the benchmark's CPU-baseline leg may load
 * it.  It shares no code with the CUDA library.
 */
#ifndef ORACLE_H
#define ORACLE_H
#include <stdint.h>

#define ORC_MAX_TYPES 2
#define ORC_MAX_SERVERS 8
#define ORC_MAX_BSIZES 8
#define ORC_MAX_LAYERS 6
#define ORC_DIURNAL_MAX 128
#define ORC_HEADER_WORDS 32

enum { ORC_SINGLE = 0, ORC_ROUTE = 1 };
enum { ORC_ARR_THINNED = 0, ORC_ARR_DIURNAL = 1, ORC_ARR_TRACE = 2 };
enum { ORC_SAMPLE = 0, ORC_ARGMAX = 1, ORC_STATIC = 2, ORC_RR = 3, ORC_SQ = 4,
       ORC_RANDOM = 5, ORC_EXTERNAL = 6 };

/* Philox streams (third counter word). */
enum { ORC_STREAM_ARRIVAL = 1, ORC_STREAM_POLICY = 2, ORC_STREAM_SWITCH = 3,
       ORC_STREAM_INIT = 4, ORC_STREAM_EPOCH = 5 };

/* Same field list and meaning as the library's configuration record. */
typedef struct {
  uint32_t abi_version, mode, n_envs, n_servers, n_types, queue_cap, episode_len, arrival_kind;
  float cand_mean_gap_us;
  uint32_t n_mod_states;
  uint32_t accept_thr[2];
  float dwell_mean_us;
  uint32_t epoch_us, diurnal_len;
  float diurnal_rate[ORC_DIURNAL_MAX];
  float burst_sigma;
  uint32_t type0_thr;
  uint32_t alpha_us[ORC_MAX_TYPES];
  uint32_t beta_us[ORC_MAX_TYPES];
  int32_t cost_type;
  uint32_t cost_kind;
  float cost_scale_us, pareto_inv_alpha;
  float w_wait[ORC_MAX_TYPES];
  uint32_t n_bsizes;
  uint32_t bsizes[ORC_MAX_BSIZES];
  uint32_t static_bi;
  uint32_t obs_extra, obs_dim;
  float t_window_us, rate_scale, rate_ref, busy_norm_us;
  uint32_t phase_period_us;
  uint32_t dwell_kind;                      /* 0 exponential dwell, 1 fixed dwell (square wave) */
  uint32_t srv_speed16[ORC_MAX_SERVERS];    /* batch time factor of each server, in 1/16 (0: 16) */
  uint32_t action_layout;                   /* 0: major x table index; 1: Wait + sizes 1..n */
  /* Trace replay (arrival_kind TRACE, Sec. 3.2): host arrays of trace_len entries; the
     gap before each request, its type (or NULL: drawn), its cost (or NULL: drawn). */
  const uint32_t* trace_gap;
  const uint8_t* trace_type;
  const uint32_t* trace_cost;
  uint32_t trace_len;
} orc_config;

/* Host-memory MLP (row-major W[l] of dims[l+1] x dims[l]). */
typedef struct {
  int32_t n_layers;
  int32_t dims[ORC_MAX_LAYERS + 1];
  const float* W[ORC_MAX_LAYERS];
  const float* b[ORC_MAX_LAYERS];
  int32_t has_value;
  int32_t act[ORC_MAX_LAYERS];   /* after layer l < n_layers - 1: 0 tanh, 1 identity, 2 GELU */
  /* Grid policy (the exact policy forward; Sec. 4.2 network on a fixed-point grid): when
     grid != 0 the input of layer l is put on the grid 2^-gx[l] by orc_gridq (the
     observation for l = 0, the activated hidden output otherwise) and every pre-activation
     is the exact dot product plus bias, rounded once to fp32.  With weights on a grid
     2^-e_w (|mantissa| <= 255), biases on 2^-(gx[l] + e_w) (|mantissa| <= 2^16) and
     dims[l] <= 256 that value is exact, so any summation order reproduces it. */
  int32_t grid;
  int32_t gx[ORC_MAX_LAYERS];
} orc_mlp;

typedef struct orc_env orc_env;

/* Per-step outputs of one env. */
typedef struct {
  float* obs;        /* [obs_dim] observation at the decision */
  float* logits;     /* [n_actions] (policy modes SAMPLE/ARGMAX), may be NULL */
  int32_t action;
  float logp, value, reward;
  uint8_t done;
  int64_t trace[4];  /* decision time, dispatched, summed queueing us, queued after decision */
} orc_step_out;

#ifdef __cplusplus
extern "C" {
#endif
/* Primitives, exported for the pin tests. */
void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);
float orc_detlog(float x);
float orc_detexp(float x);
float orc_dettanh(float x);
float orc_detgelu(float x);
/* Grid rounding Q(v, e) = clamp(rint(v 2^e), -255, 255) 2^-e, ties to even. */
float orc_gridq(float v, int32_t e);
void orc_gridq_n(const float* v, int64_t n, int32_t e, float* out);
float orc_detcos2pi(float u);
float orc_normal(uint32_t w0, uint32_t w1);
uint32_t orc_duration(float x);

uint32_t orc_obs_dim(const orc_config* c);
uint64_t orc_state_words(const orc_config* c);

orc_env* orc_env_new(const orc_config* c, uint32_t env_id, uint64_t seed);
void orc_env_free(orc_env* e);
void orc_env_reset(orc_env* e);
void orc_env_observe(const orc_env* e, float* obs);
/* One decision step.  ext_action is used when mode == ORC_EXTERNAL. */
void orc_env_step(orc_env* e, const orc_mlp* m, int mode, int32_t ext_action, orc_step_out* o);
void orc_env_export(const orc_env* e, uint32_t* words);
void orc_env_import(orc_env* e, const uint32_t* words);
uint32_t orc_env_status(const orc_env* e);
/* Test hook: attach a host array of cap (time, state) pairs that the env fills, from its
   next reset on, with the modulating chain's state at time 0 and the time and new state
   of every switch it processes (n_mod_states = 2 only); NULL detaches.  The count of
   pairs written is orc_env_switch_log_count.  The simulation does not read the log. */
void orc_env_switch_log(orc_env* e, uint32_t* pairs, uint32_t cap);
uint32_t orc_env_switch_log_count(const orc_env* e);
/* Exact finite-horizon Little identity pieces up to time t_end (>= every event):
   *area = integral of the total queue length over [0, t_end] accumulated event by
   event; *waits = summed queueing time of dispatched requests plus (t_end - arrival)
   of every request still queued. */
void orc_env_little(const orc_env* e, uint32_t t_end, uint64_t* area, uint64_t* waits);

/* Vectorised primitives for the pin tests. */
void orc_map(int fn, const float* x, float* y, int64_t n);
void orc_philox_n(uint32_t idx0, uint32_t env, uint32_t stream, uint64_t seed, int64_t n,
                  uint32_t* out);
void orc_samplers(const orc_config* c, int kind, float scale, const uint32_t* w, int64_t n,
                  float* out);

/* Policy forward on one observation: logits/value, sampled or argmax action, logp. */
void orc_policy(const orc_mlp* m, const float* obs, int mode, uint64_t seed, uint32_t step,
                uint32_t env_id, float* logits, float* value, int32_t* action, float* logp);

/*
 * Convenience driver: reset envs env_ids[0..n), run H steps each, write the rollout in
 * the library's time-major layouts ([H][D][n] obs, [H][n] others, [H][4][n] trace) and
 * the final canonical states [n][state_words].  Any output pointer may be NULL.
 */
int orc_rollout(const orc_config* c, const orc_mlp* m, uint64_t seed, int mode,
                const uint32_t* env_ids, int64_t n, int32_t H, float* obs, int32_t* action,
                float* logp, float* value, float* reward, uint8_t* done, int64_t* trace,
                uint32_t* final_state);
#ifdef __cplusplus
}
#endif
#endif
