// api.cu — the C ABI of libsimx.so (declared in include/simx.h): argument
// validation on the host, device state ownership, and kernel launches.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <atomic>
#include <cstring>
#include <mutex>
#include <string>

#include "../../include/simx.h"
#include "kernels.h"

using namespace simx;

static std::atomic<uint64_t> g_launches{0};
void simx::count_launches(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }

// SM count of the current device, looked up once per device (152 on a GB300).  Without a
// usable device (a host that only builds or sizes workspaces) the GB300's count is taken.
static std::atomic<int> g_sms[64];
int simx::sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 152;
  int n = g_sms[dev].load(std::memory_order_relaxed);
  if (n > 0) return n;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    return 152;
  }
  g_sms[dev].store(n, std::memory_order_relaxed);
  return n;
}

namespace {

thread_local std::string g_err;

simx_status fail(simx_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_err = buf;
  return s;
}

simx_status cuda_fail(cudaError_t e, const char* what) {
  return fail(SIMX_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool pow2(uint32_t x) { return x && !(x & (x - 1)); }

uint32_t n_actions_of(const simx_config& c) {
  return (c.mode == SIMX_MODE_SINGLE ? c.n_types : c.n_servers) * c.n_bsizes +
         (c.action_layout == 1 ? 1u : 0u);
}

uint32_t obs_dim_of(const simx_config& c) {
  if (c.mode == SIMX_MODE_SINGLE) return 2u * c.n_types + 6u + (c.obs_extra ? 6u : 0u);
  return 3u * c.n_servers + 1u + (c.obs_extra ? 3u : 0u);
}

bool finite_pos(float x) { return std::isfinite(x) && x > 0.0f; }

simx_status validate_config(const simx_config* c) {
  if (!c) return fail(SIMX_EINVAL, "config is NULL");
  if (c->abi_version != SIMX_ABI_VERSION) return fail(SIMX_EINVAL, "abi_version %u != %u", c->abi_version, SIMX_ABI_VERSION);
  if (c->mode > SIMX_MODE_ROUTE) return fail(SIMX_EINVAL, "mode %u", c->mode);
  if (c->n_envs < 1 || c->n_envs > (1u << 24)) return fail(SIMX_EINVAL, "n_envs %u outside [1, 2^24]", c->n_envs);
  if (c->n_types < 1 || c->n_types > SIMX_MAX_TYPES) return fail(SIMX_EINVAL, "n_types %u", c->n_types);
  if (c->mode == SIMX_MODE_SINGLE && c->n_servers != 1) return fail(SIMX_EINVAL, "SINGLE mode needs n_servers = 1");
  if (c->n_servers < 1 || c->n_servers > SIMX_MAX_SERVERS) return fail(SIMX_EINVAL, "n_servers %u", c->n_servers);
  for (uint32_t k = 0; k < SIMX_MAX_SERVERS; ++k)
    if (c->srv_speed16[k] > 255) return fail(SIMX_EINVAL, "srv_speed16[%u] = %u (at most 255)", k, c->srv_speed16[k]);
  if (!pow2(c->queue_cap) || c->queue_cap > 4096) return fail(SIMX_EINVAL, "queue_cap %u must be a power of two <= 4096", c->queue_cap);
  if (c->episode_len < 1) return fail(SIMX_EINVAL, "episode_len must be >= 1");
  if (c->arrival_kind == SIMX_ARR_THINNED || c->arrival_kind == SIMX_ARR_TRACE) {
    if (c->arrival_kind == SIMX_ARR_THINNED && !finite_pos(c->cand_mean_gap_us))
      return fail(SIMX_EINVAL, "cand_mean_gap_us must be > 0");
    if (c->n_mod_states < 1 || c->n_mod_states > 2) return fail(SIMX_EINVAL, "n_mod_states %u", c->n_mod_states);
    for (uint32_t i = 0; i < c->n_mod_states; ++i)
      if (c->accept_thr[i] > (1u << 24)) return fail(SIMX_EINVAL, "accept_thr[%u] > 2^24", i);
    if (c->n_mod_states == 2 && !finite_pos(c->dwell_mean_us)) return fail(SIMX_EINVAL, "dwell_mean_us must be > 0");
    if (c->dwell_kind > 1) return fail(SIMX_EINVAL, "dwell_kind %u", c->dwell_kind);
    if (c->n_mod_states == 2 && c->dwell_kind == 1 && !(c->dwell_mean_us >= 0.5f))
      return fail(SIMX_EINVAL, "a fixed dwell must be at least 1 us");
  } else if (c->arrival_kind == SIMX_ARR_DIURNAL) {
    if (c->mode != SIMX_MODE_ROUTE) return fail(SIMX_EINVAL, "DIURNAL arrivals need ROUTE mode");
    if (c->epoch_us < 1) return fail(SIMX_EINVAL, "epoch_us must be >= 1");
    if (c->diurnal_len < 1 || c->diurnal_len > SIMX_DIURNAL_MAX) return fail(SIMX_EINVAL, "diurnal_len %u", c->diurnal_len);
    for (uint32_t i = 0; i < c->diurnal_len; ++i)
      if (!finite_pos(c->diurnal_rate[i])) return fail(SIMX_EINVAL, "diurnal_rate[%u] must be > 0", i);
    if (!std::isfinite(c->burst_sigma)) return fail(SIMX_EINVAL, "burst_sigma");
  } else {
    return fail(SIMX_EINVAL, "arrival_kind %u", c->arrival_kind);
  }
  if (c->type0_thr > (1u << 24)) return fail(SIMX_EINVAL, "type0_thr > 2^24");
  if (c->cost_type < -1 || c->cost_type >= (int32_t)c->n_types) return fail(SIMX_EINVAL, "cost_type %d", c->cost_type);
  if (c->cost_type >= 0) {
    if (c->cost_kind > 1) return fail(SIMX_EINVAL, "cost_kind %u", c->cost_kind);
    if (!finite_pos(c->cost_scale_us)) return fail(SIMX_EINVAL, "cost_scale_us must be > 0");
    if (c->cost_kind == 0 && !finite_pos(c->pareto_inv_alpha)) return fail(SIMX_EINVAL, "pareto_inv_alpha must be > 0");
  }
  if (c->action_layout > 1) return fail(SIMX_EINVAL, "action_layout %u", c->action_layout);
  if (c->action_layout == 1) {  // Wait + batch sizes 1 .. n_bsizes (no table)
    if (c->mode != SIMX_MODE_SINGLE) return fail(SIMX_EINVAL, "the Wait action layout is single-server only");
    if (c->n_bsizes < 1 || c->n_bsizes > 64) return fail(SIMX_EINVAL, "n_bsizes %u (1 .. 64 with the Wait layout)", c->n_bsizes);
  } else {
    if (c->n_bsizes < 1 || c->n_bsizes > SIMX_MAX_BSIZES) return fail(SIMX_EINVAL, "n_bsizes %u", c->n_bsizes);
    for (uint32_t i = 0; i < c->n_bsizes; ++i)
      if (c->bsizes[i] < 1) return fail(SIMX_EINVAL, "bsizes[%u] must be >= 1", i);
  }
  if (c->static_bi >= c->n_bsizes) return fail(SIMX_EINVAL, "static_bi %u >= n_bsizes", c->static_bi);
  if (n_actions_of(*c) > 255) return fail(SIMX_EINVAL, "more than 255 actions");
  if (c->obs_dim != obs_dim_of(*c)) return fail(SIMX_EINVAL, "obs_dim %u != %u implied by the configuration", c->obs_dim, obs_dim_of(*c));
  if (!finite_pos(c->t_window_us)) return fail(SIMX_EINVAL, "t_window_us must be > 0");
  if (c->mode == SIMX_MODE_ROUTE) {
    if (!finite_pos(c->rate_ref)) return fail(SIMX_EINVAL, "rate_ref must be > 0");
    if (!finite_pos(c->busy_norm_us)) return fail(SIMX_EINVAL, "busy_norm_us must be > 0");
    if (c->obs_extra && c->phase_period_us < 1) return fail(SIMX_EINVAL, "phase_period_us must be >= 1");
  } else if (!std::isfinite(c->rate_scale)) {
    return fail(SIMX_EINVAL, "rate_scale");
  }
  return SIMX_OK;
}

int round_up(int x, int m) { return (x + m - 1) / m * m; }

// Shared-memory geometry of the env kernels: activation rows (widest layer) and
// softmax scratch per env, both rounded to float4.
void act_layout(int maxdim, int n_actions, int& maxd4, int& apad) {
  maxd4 = round_up(maxdim, 4);
  apad = round_up(n_actions > 0 ? n_actions : 1, 4);
}

simx_status validate_mlp(const simx_mlp* m, uint32_t obs_dim, uint32_t n_actions) {
  if (!m) return fail(SIMX_EINVAL, "policy is NULL");
  if (m->n_layers < 1 || m->n_layers > SIMX_MAX_LAYERS) return fail(SIMX_EINVAL, "n_layers %d", m->n_layers);
  if (obs_dim && (uint32_t)m->dims[0] != obs_dim) return fail(SIMX_EINVAL, "policy input %d != obs_dim %u", m->dims[0], obs_dim);
  if (m->dims[0] < 1 || m->dims[0] > SIMX_MAX_OBS) return fail(SIMX_EINVAL, "policy input width %d", m->dims[0]);
  for (int l = 1; l < m->n_layers; ++l)
    if (m->dims[l] < 1 || m->dims[l] > SIMX_MAX_WIDTH) return fail(SIMX_EINVAL, "hidden width %d", m->dims[l]);
  const int out = m->dims[m->n_layers];
  const int A = out - (m->has_value ? 1 : 0);
  if (out < 1 || out > SIMX_MAX_OUT || A < 1 || A > 255) return fail(SIMX_EINVAL, "output width %d", out);
  if (n_actions && (uint32_t)A != n_actions) return fail(SIMX_EINVAL, "policy has %d actions, environment %u", A, n_actions);
  for (int l = 0; l < m->n_layers; ++l)
    if (!m->W[l] || !m->b[l]) return fail(SIMX_EINVAL, "layer %d weights are NULL", l);
  for (int l = 0; l + 1 < m->n_layers; ++l)
    if (m->act[l] < SIMX_ACT_TANH || m->act[l] > SIMX_ACT_GELU) return fail(SIMX_EINVAL, "act[%d] = %d", l, m->act[l]);
  if (m->grid != 0 && m->grid != 1) return fail(SIMX_EINVAL, "grid = %d", m->grid);
  if (m->grid)
    for (int l = 0; l < m->n_layers; ++l) {
      if (m->gx[l] < 0 || m->gx[l] > 24) return fail(SIMX_EINVAL, "gx[%d] = %d (0 .. 24)", l, m->gx[l]);
      if (m->dims[l] > 256) return fail(SIMX_EINVAL, "grid policy fan-in %d above 256", m->dims[l]);
    }
  return SIMX_OK;
}

// Device copy of a policy in the kernels' layout; grown on demand.
struct Packed {
  float* buf = nullptr;
  size_t cap = 0;
  int device = -1;
};

simx_status pack_mlp(const simx_mlp* m, Packed& P, DevMlp& out, cudaStream_t s) {
  size_t need = 0;
  int npad[SIMX_MAX_LAYERS + 1];
  for (int l = 0; l < m->n_layers; ++l) {
    npad[l + 1] = round_up(m->dims[l + 1], 4);
    need += (size_t)m->dims[l] * npad[l + 1] + npad[l + 1];
  }
  if (need > P.cap) {
    if (P.buf) cudaFree(P.buf);
    P.buf = nullptr;
    P.cap = 0;
    cudaError_t e = cudaMalloc(&P.buf, need * sizeof(float));
    if (e != cudaSuccess) return cuda_fail(e, "cudaMalloc(policy repack)");
    P.cap = need;
  }
  std::memset(&out, 0, sizeof(out));
  float* p = P.buf;
  for (int l = 0; l < m->n_layers; ++l) {
    const int K = m->dims[l], N = m->dims[l + 1];
    float* Wt = p;
    float* bias = p + (size_t)K * npad[l + 1];
    cudaError_t e = launch_repack(m->W[l], m->b[l], N, K, npad[l + 1], Wt, bias, s);
    if (e != cudaSuccess) return cuda_fail(e, "repack");
    out.Wt[l] = Wt;
    out.bias[l] = bias;
    out.act[l] = (l + 1 < m->n_layers) ? m->act[l] : -1;  // -1: no activation (output layer)
    p = bias + npad[l + 1];
  }
  for (int l = 0; l <= m->n_layers; ++l) {
    out.dims[l] = m->dims[l];
    out.npad[l] = l ? npad[l] : m->dims[0];
  }
  out.n_layers = m->n_layers;
  out.has_value = m->has_value ? 1 : 0;
  out.grid = m->grid ? 1 : 0;
  for (int l = 0; l < m->n_layers; ++l) out.gx[l] = m->grid ? m->gx[l] : 0;
  out.n_actions = m->dims[m->n_layers] - out.has_value;
  return SIMX_OK;
}

int mlp_maxdim(const simx_mlp* m) {
  int mx = 0;
  for (int l = 0; l <= m->n_layers; ++l) mx = m->dims[l] > mx ? m->dims[l] : mx;
  return mx;
}

std::mutex g_pf_mu;
Packed g_pf_pack[64];  // per-device policy repack buffers for policy_forward

}  // namespace

struct Trace {
  const uint32_t* gap = nullptr;
  const uint8_t* type = nullptr;
  const uint32_t* cost = nullptr;
  uint32_t n = 0;
};

struct simx_ctx {
  simx_config cfg;
  int device = 0;
  Trace trace_next, trace;  // set by sim_set_trace; taken over by sim_reset
  DevState st{};
  uint32_t key0 = 0, key1 = 0;
  bool seeded = false;
  Packed pack;
  uint32_t* img = nullptr;
  unsigned long long* stats = nullptr;
  cudaStream_t last = nullptr;
  void* mem[8] = {};
};

extern "C" {

const char* simx_strerror(simx_status s) {
  switch (s) {
    case SIMX_OK: return "ok";
    case SIMX_EINVAL: return "invalid argument";
    case SIMX_ENOMEM: return "out of memory";
    case SIMX_ECUDA: return "CUDA error";
    case SIMX_EOVERFLOW: return "device status flag raised (time overflow, event cap, bad action or a bounded wait timed out)";
    case SIMX_ESTATE: return "call out of order";
  }
  return "unknown status";
}

const char* simx_last_error(void) { return g_err.c_str(); }

uint64_t simx_launches(void) { return g_launches.load(std::memory_order_relaxed); }

simx_status simx_fma_probe(int64_t iters, float* d_sink, double* host_flops, void* stream) {
  if (iters < 1 || !d_sink || !host_flops) return fail(SIMX_EINVAL, "fma probe: iters %lld", (long long)iters);
  const cudaError_t e = launch_fma_probe(iters, d_sink, host_flops, (cudaStream_t)stream);
  if (e != cudaSuccess) return fail(SIMX_ECUDA, "fma probe: %s", cudaGetErrorString(e));
  return SIMX_OK;
}

size_t simx_fma_probe_sink_floats(void) { return fma_probe_sink_floats(); }

size_t simx_adam_workspace_size(int64_t n) { return n < 1 ? 0 : adam_workspace_bytes(n); }

simx_status simx_adam_step(float* d_params, const float* d_grad, float* d_m, float* d_v,
                           const uint8_t* d_mask, int64_t n, int64_t t, int64_t* d_t,
                           const simx_adam_params* p, void* d_workspace, size_t workspace_bytes,
                           void* stream) {
  if (!d_params || !d_grad || !d_m || !d_v || !p) return fail(SIMX_EINVAL, "adam: NULL array or params");
  if (n < 1 || (!d_t && t < 1)) return fail(SIMX_EINVAL, "adam: n %lld, t %lld", (long long)n, (long long)t);
  if (!(p->lr >= 0.0f) || !(p->beta1 >= 0.0f && p->beta1 < 1.0f) ||
      !(p->beta2 >= 0.0f && p->beta2 < 1.0f) || !(p->eps > 0.0f) || !std::isfinite(p->lr) ||
      std::isnan(p->max_grad_norm))
    return fail(SIMX_EINVAL, "adam: lr %g beta1 %g beta2 %g eps %g", p->lr, p->beta1, p->beta2, p->eps);
  if ((p->max_grad_norm > 0.0f || d_t) && (!d_workspace || workspace_bytes < adam_workspace_bytes(n)))
    return fail(SIMX_EINVAL, "adam: workspace of %zu bytes needed", adam_workspace_bytes(n));
  const cudaError_t e = launch_adam(d_params, d_grad, d_m, d_v, d_mask, n, t, d_t, p->lr, p->beta1,
                                    p->beta2, p->eps, p->max_grad_norm, d_workspace,
                                    (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "adam launch");
  return SIMX_OK;
}

uint32_t simx_obs_dim(const simx_config* cfg) {
  if (!cfg || cfg->mode > SIMX_MODE_ROUTE || cfg->n_types < 1 || cfg->n_types > SIMX_MAX_TYPES ||
      cfg->n_servers < 1 || cfg->n_servers > SIMX_MAX_SERVERS)
    return 0;
  return obs_dim_of(*cfg);
}

uint64_t simx_state_words(const simx_config* c) {
  if (!c) return 0;
  const uint64_t K = c->n_servers, T = c->n_types, cap = c->queue_cap;
  uint64_t w = SIMX_STATE_HEADER_WORDS + 2 * K + K * T + K * T * cap;
  if (c->cost_type >= 0) w += K * cap;
  return w;
}

simx_status sim_create(const simx_config* cfg, int device, simx_ctx** out) {
  if (!out) return fail(SIMX_EINVAL, "out is NULL");
  *out = nullptr;
  simx_status v = validate_config(cfg);
  if (v != SIMX_OK) return v;
  int ndev = 0;
  cudaError_t e = cudaGetDeviceCount(&ndev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDeviceCount");
  if (device < 0 || device >= ndev) return fail(SIMX_EINVAL, "device %d of %d", device, ndev);
  e = cudaSetDevice(device);
  if (e != cudaSuccess) return cuda_fail(e, "cudaSetDevice");
  simx_ctx* c = new (std::nothrow) simx_ctx();
  if (!c) return fail(SIMX_ENOMEM, "host allocation");
  c->cfg = *cfg;
  c->device = device;
  const uint64_t E = cfg->n_envs, K = cfg->n_servers, T = cfg->n_types, cap = cfg->queue_cap;
  const size_t sizes[6] = {
      (size_t)F_COUNT * E * 4, (size_t)2 * K * E * 4, (size_t)K * T * E * 4, (size_t)K * T * E * 4,
      (size_t)E * K * T * cap * 4, cfg->cost_type >= 0 ? (size_t)E * K * cap * 4 : 0};
  for (int i = 0; i < 6; ++i) {
    if (!sizes[i]) continue;
    e = cudaMalloc(&c->mem[i], sizes[i]);
    if (e != cudaSuccess) {
      sim_destroy(c);
      cudaGetLastError();
      return fail(SIMX_ENOMEM, "cudaMalloc(%zu bytes): %s", sizes[i], cudaGetErrorString(e));
    }
    cudaMemset(c->mem[i], 0, sizes[i]);
  }
  e = cudaMalloc(&c->stats, 16 * sizeof(unsigned long long));
  if (e != cudaSuccess) {
    sim_destroy(c);
    return fail(SIMX_ENOMEM, "cudaMalloc(stats)");
  }
  c->st.hdr = (uint32_t*)c->mem[0];
  c->st.srv = (uint32_t*)c->mem[1];
  c->st.qh = (uint32_t*)c->mem[2];
  c->st.qc = (uint32_t*)c->mem[3];
  c->st.ring = (uint32_t*)c->mem[4];
  c->st.cost = (uint32_t*)c->mem[5];
  c->st.E = (uint32_t)E;
  c->st.K = (uint32_t)K;
  c->st.T = (uint32_t)T;
  c->st.cap = (uint32_t)cap;
  e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    sim_destroy(c);
    return cuda_fail(e, "sim_create");
  }
  *out = c;
  return SIMX_OK;
}

void sim_destroy(simx_ctx* c) {
  if (!c) return;
  cudaSetDevice(c->device);
  for (void* p : c->mem)
    if (p) cudaFree(p);
  if (c->pack.buf) cudaFree(c->pack.buf);
  if (c->img) cudaFree(c->img);
  if (c->stats) cudaFree(c->stats);
  delete c;
}

static void base_args(simx_ctx* c, RolloutArgs& a) {
  std::memset(&a, 0, sizeof(a));
  a.cfg = c->cfg;
  a.st = c->st;
  a.key0 = c->key0;
  a.key1 = c->key1;
  a.n_actions = n_actions_of(c->cfg);
  a.obs_dim = (int)c->cfg.obs_dim;
  a.ld = c->cfg.n_envs;
  a.next_ld = c->cfg.n_envs;
  a.G = choose_lanes(c->cfg.n_envs);
  a.threads = choose_threads(c->cfg.n_envs, a.G);
  act_layout((int)c->cfg.obs_dim, (int)a.n_actions, a.maxd4, a.apad);
  a.bs_pad = 4;
  a.tr_gap = c->trace.gap;
  a.tr_type = c->trace.type;
  a.tr_cost = c->trace.cost;
  a.tr_n = c->trace.n;
}

simx_status sim_set_trace(simx_ctx* c, const uint32_t* d_gap_us, const uint8_t* d_type,
                          const uint32_t* d_cost_us, uint32_t n) {
  if (!c || !d_gap_us) return fail(SIMX_EINVAL, "ctx or d_gap_us is NULL");
  if (c->cfg.arrival_kind != SIMX_ARR_TRACE) return fail(SIMX_EINVAL, "arrival_kind is not TRACE");
  if (n < 1 || n >= (1u << 31)) return fail(SIMX_EINVAL, "trace length %u outside [1, 2^31)", n);
  c->trace_next.gap = d_gap_us;
  c->trace_next.type = d_type;
  c->trace_next.cost = d_cost_us;
  c->trace_next.n = n;
  return SIMX_OK;
}

simx_status sim_reset(simx_ctx* c, uint64_t seed, void* stream) {
  if (!c) return fail(SIMX_EINVAL, "ctx is NULL");
  cudaSetDevice(c->device);
  if (c->cfg.arrival_kind == SIMX_ARR_TRACE && !c->trace_next.gap)
    return fail(SIMX_ESTATE, "TRACE arrivals need sim_set_trace before sim_reset");
  c->trace = c->trace_next;
  c->key0 = (uint32_t)seed;
  c->key1 = (uint32_t)(seed >> 32);
  RolloutArgs a;
  base_args(c, a);
  cudaError_t e = launch_reset(a, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "reset launch");
  c->seeded = true;
  c->last = (cudaStream_t)stream;
  return SIMX_OK;
}

simx_status sim_observe(simx_ctx* c, float* d_obs, int64_t ld, void* stream) {
  if (!c || !d_obs) return fail(SIMX_EINVAL, "ctx or d_obs is NULL");
  if (!c->seeded) return fail(SIMX_ESTATE, "sim_reset has not been called");
  if (ld < (int64_t)c->cfg.n_envs) return fail(SIMX_EINVAL, "ld %lld < n_envs", (long long)ld);
  cudaSetDevice(c->device);
  RolloutArgs a;
  base_args(c, a);
  a.next_obs = d_obs;
  a.next_ld = ld;
  cudaError_t e = launch_observe(a, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "observe launch");
  c->last = (cudaStream_t)stream;
  return SIMX_OK;
}

// k_rollout's forward: warp-local for narrow policies at 16 or 32 lanes per env in SINGLE
// mode (each warp then loads every weight row, which wide layers cannot afford); the
// kernel has that variant only there.
static int mlp_warp_of(bool route, int G, const simx_mlp* pol) {
  return (!route && G >= 16 && mlp_maxdim(pol) <= 64) ? 1 : 0;
}

static simx_status prepare_policy(simx_ctx* c, const simx_mlp* pol, int mode, RolloutArgs& a,
                                  cudaStream_t s) {
  const bool route = c->cfg.mode == SIMX_MODE_ROUTE;
  switch (mode) {
    case SIMX_POLICY_SAMPLE:
    case SIMX_POLICY_ARGMAX: {
      simx_status v = validate_mlp(pol, c->cfg.obs_dim, a.n_actions);
      if (v != SIMX_OK) return v;
      v = pack_mlp(pol, c->pack, a.mlp, s);
      if (v != SIMX_OK) return v;
      act_layout(mlp_maxdim(pol), (int)a.n_actions, a.maxd4, a.apad);
      a.mlp_warp = mlp_warp_of(route, a.G, pol);
      a.bs_pad = a.mlp_warp ? act_stride_pad(a.mlp, 32 / a.G, 32)
                            : act_stride_pad(a.mlp, a.threads / a.G, a.threads);
      break;
    }
    case SIMX_POLICY_STATIC:
      if (route) return fail(SIMX_EINVAL, "STATIC is a SINGLE-mode baseline");
      break;
    case SIMX_POLICY_RR:
    case SIMX_POLICY_SQ:
      if (!route) return fail(SIMX_EINVAL, "RR and SQ are ROUTE-mode baselines");
      break;
    case SIMX_POLICY_RANDOM:
      break;
    default:
      return fail(SIMX_EINVAL, "policy_mode %d", mode);
  }
  a.policy_mode = mode;
  return SIMX_OK;
}

simx_status sim_step_batched(simx_ctx* c, const int32_t* d_actions, const simx_mlp* pol,
                             int policy_mode, float* d_obs, int64_t ld, float* d_reward,
                             uint8_t* d_done, uint8_t* d_action, float* d_logp, void* stream) {
  if (!c) return fail(SIMX_EINVAL, "ctx is NULL");
  if (!c->seeded) return fail(SIMX_ESTATE, "sim_reset has not been called");
  if (d_obs && ld < (int64_t)c->cfg.n_envs) return fail(SIMX_EINVAL, "ld %lld < n_envs", (long long)ld);
  cudaSetDevice(c->device);
  RolloutArgs a;
  base_args(c, a);
  const cudaStream_t s = (cudaStream_t)stream;
  if (policy_mode == SIMX_POLICY_EXTERNAL) {
    if (!d_actions) return fail(SIMX_EINVAL, "EXTERNAL mode needs d_actions");
    a.policy_mode = SIMX_POLICY_EXTERNAL;
    a.ext = d_actions;
  } else {
    simx_status v = prepare_policy(c, pol, policy_mode, a, s);
    if (v != SIMX_OK) return v;
  }
  a.H = 1;
  a.ld = c->cfg.n_envs;
  a.reward = d_reward;
  a.done = d_done;
  a.action = d_action;
  a.logp = d_logp;
  a.next_obs = d_obs;
  a.next_ld = d_obs ? ld : c->cfg.n_envs;
  cudaError_t e = step_thread_supported(a) ? launch_step_thread(a, s) : launch_rollout(a, s);
  if (e != cudaSuccess) return cuda_fail(e, "step launch");
  c->last = s;
  return SIMX_OK;
}

simx_status rollout_collect(simx_ctx* c, const simx_mlp* pol, int policy_mode, int32_t horizon,
                            const simx_rollout* out, void* stream) {
  if (!c || !out) return fail(SIMX_EINVAL, "ctx or out is NULL");
  if (!c->seeded) return fail(SIMX_ESTATE, "sim_reset has not been called");
  if (horizon < 0) return fail(SIMX_EINVAL, "horizon %d", horizon);
  if (out->ld < (int64_t)c->cfg.n_envs) return fail(SIMX_EINVAL, "rollout ld %lld < n_envs", (long long)out->ld);
  if (!out->obs || !out->action || !out->reward || !out->done)
    return fail(SIMX_EINVAL, "rollout obs, action, reward and done are required");
  if (policy_mode == SIMX_POLICY_EXTERNAL) return fail(SIMX_EINVAL, "EXTERNAL actions are a sim_step_batched mode");
  if (horizon == 0) return SIMX_OK;
  cudaSetDevice(c->device);
  RolloutArgs a;
  base_args(c, a);
  const cudaStream_t s = (cudaStream_t)stream;
  simx_status v = prepare_policy(c, pol, policy_mode, a, s);
  if (v != SIMX_OK) return v;
  if (out->value && !(pol && pol->has_value) && (policy_mode == SIMX_POLICY_SAMPLE || policy_mode == SIMX_POLICY_ARGMAX))
    return fail(SIMX_EINVAL, "value buffer given but the policy has no value row");
  a.H = horizon;
  a.ld = out->ld;
  a.obs = out->obs;
  a.action = out->action;
  a.logp = out->logp;
  a.value = out->value;
  a.reward = out->reward;
  a.done = out->done;
  a.trace = out->trace;
  cudaError_t e = step_thread_supported(a) ? launch_step_thread(a, s) : launch_rollout(a, s);
  if (e != cudaSuccess) return cuda_fail(e, "rollout launch");
  c->last = s;
  return SIMX_OK;
}

simx_status simx_launch_shape(simx_ctx* c, const simx_mlp* pol, int policy_mode,
                              int32_t* host_out) {
  if (!c || !host_out) return fail(SIMX_EINVAL, "ctx or host_out is NULL");
  const bool route = c->cfg.mode == SIMX_MODE_ROUTE;
  const bool net = policy_mode == SIMX_POLICY_SAMPLE || policy_mode == SIMX_POLICY_ARGMAX;
  if (policy_mode < 0 || policy_mode > SIMX_POLICY_EXTERNAL) return fail(SIMX_EINVAL, "policy_mode %d", policy_mode);
  if (net) {
    simx_status v = validate_mlp(pol, c->cfg.obs_dim, n_actions_of(c->cfg));
    if (v != SIMX_OK) return v;
  }
  cudaSetDevice(c->device);
  RolloutArgs a;
  base_args(c, a);
  a.policy_mode = policy_mode;
  const bool thread = step_thread_supported(a);
  host_out[0] = thread ? 1 : 0;
  host_out[1] = thread ? 1 : a.G;
  host_out[2] = thread ? 128 : a.threads;
  host_out[3] = (!thread && net) ? mlp_warp_of(route, a.G, pol) : 0;
  host_out[4] = 0;
  host_out[5] = 0;
  if (!thread && net) {  // the launch's forward plans (no repack needed)
    a.mlp_warp = host_out[3];
    a.mlp.n_layers = pol->n_layers;
    for (int l = 0; l <= pol->n_layers; ++l) {
      a.mlp.dims[l] = pol->dims[l];
      a.mlp.npad[l] = l ? round_up(pol->dims[l], 4) : pol->dims[0];
    }
    a.mlp.grid = pol->grid;
    act_layout(mlp_maxdim(pol), (int)a.n_actions, a.maxd4, a.apad);
    a.bs_pad = a.mlp_warp ? act_stride_pad(a.mlp, 32 / a.G, 32)
                          : act_stride_pad(a.mlp, a.threads / a.G, a.threads);
    plan_rollout(a);
    host_out[4] = a.tc.on;
    host_out[5] = a.stage.on;
  }
  return SIMX_OK;
}

// Floats of a policy repacked in the kernels' layout (pack_mlp).
static size_t packed_floats(const simx_mlp* m) {
  size_t need = 0;
  for (int l = 0; l < m->n_layers; ++l) {
    const int np = round_up(m->dims[l + 1], 4);
    need += (size_t)m->dims[l] * np + np;
  }
  return need;
}

// policy_forward with the repack buffer P (the library's per-device one, or a caller's).
static simx_status policy_forward_into(Packed& P, const simx_mlp* pol, const float* d_obs,
                                       int64_t ld, int64_t n, int policy_mode, uint64_t seed,
                                       uint32_t step, uint32_t env_base, float* d_logits,
                                       float* d_value, uint8_t* d_action, float* d_logp,
                                       cudaStream_t s) {
  PolicyArgs p;
  std::memset(&p, 0, sizeof(p));
  p.G = choose_lanes(n);
  p.threads = choose_threads(n, p.G);
  simx_status v = pack_mlp(pol, P, p.mlp, s);
  if (v != SIMX_OK) return v;
  act_layout(mlp_maxdim(pol), p.mlp.n_actions, p.maxd4, p.apad);
  p.obs = d_obs;
  p.ld = ld;
  p.n = n;
  p.mode = policy_mode;
  p.key0 = (uint32_t)seed;
  p.key1 = (uint32_t)(seed >> 32);
  p.step = step;
  p.env_base = env_base;
  p.logits = d_logits;
  p.value = d_value;
  p.action = d_action;
  p.logp = d_logp;
  cudaError_t e = launch_policy_forward(p, s);
  if (e != cudaSuccess) return cuda_fail(e, "policy_forward launch");
  return SIMX_OK;
}

static simx_status policy_forward_check(const simx_mlp* pol, const float* d_obs, int64_t ld,
                                        int64_t n, int policy_mode, const float* d_value) {
  if (!d_obs) return fail(SIMX_EINVAL, "d_obs is NULL");
  if (n < 0 || ld < n) return fail(SIMX_EINVAL, "n %lld, ld %lld", (long long)n, (long long)ld);
  if (policy_mode != SIMX_POLICY_SAMPLE && policy_mode != SIMX_POLICY_ARGMAX)
    return fail(SIMX_EINVAL, "policy_forward supports SAMPLE and ARGMAX");
  simx_status v = validate_mlp(pol, 0, 0);
  if (v != SIMX_OK) return v;
  if (d_value && !pol->has_value) return fail(SIMX_EINVAL, "d_value given but the policy has no value row");
  return SIMX_OK;
}

simx_status policy_forward(const simx_mlp* pol, const float* d_obs, int64_t ld, int64_t n,
                           int policy_mode, uint64_t seed, uint32_t step, uint32_t env_base,
                           float* d_logits, float* d_value, uint8_t* d_action, float* d_logp,
                           void* stream) {
  simx_status v = policy_forward_check(pol, d_obs, ld, n, policy_mode, d_value);
  if (v != SIMX_OK || n == 0) return v;
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return fail(SIMX_EINVAL, "device %d", dev);
  std::lock_guard<std::mutex> lk(g_pf_mu);
  return policy_forward_into(g_pf_pack[dev], pol, d_obs, ld, n, policy_mode, seed, step, env_base,
                             d_logits, d_value, d_action, d_logp, (cudaStream_t)stream);
}

size_t policy_forward_workspace_size(const simx_mlp* pol) {
  if (!pol || pol->n_layers < 1 || pol->n_layers > SIMX_MAX_LAYERS) return 0;
  return packed_floats(pol) * sizeof(float);
}

simx_status policy_forward_ws(const simx_mlp* pol, const float* d_obs, int64_t ld, int64_t n,
                              int policy_mode, uint64_t seed, uint32_t step, uint32_t env_base,
                              float* d_logits, float* d_value, uint8_t* d_action, float* d_logp,
                              void* d_workspace, size_t workspace_bytes, void* stream) {
  simx_status v = policy_forward_check(pol, d_obs, ld, n, policy_mode, d_value);
  if (v != SIMX_OK || n == 0) return v;
  const size_t need = packed_floats(pol) * sizeof(float);
  if (!d_workspace || workspace_bytes < need || (reinterpret_cast<uintptr_t>(d_workspace) & 15))
    return fail(SIMX_EINVAL, "workspace of %zu bytes (16-byte aligned) needed, %zu given", need,
                workspace_bytes);
  Packed P;  // the caller's buffer: large enough, so pack_mlp neither frees nor allocates
  P.buf = static_cast<float*>(d_workspace);
  P.cap = workspace_bytes / sizeof(float);
  return policy_forward_into(P, pol, d_obs, ld, n, policy_mode, seed, step, env_base, d_logits,
                             d_value, d_action, d_logp, (cudaStream_t)stream);
}

simx_status compute_returns_gae(const float* d_rew, const float* d_val, const uint8_t* d_done,
                                const float* d_last_val, int64_t T, int64_t E, int64_t ld,
                                float gamma, float lam, float* d_ret, float* d_adv, void* stream) {
  if (T < 0 || E < 0 || ld < E) return fail(SIMX_EINVAL, "T %lld, E %lld, ld %lld", (long long)T, (long long)E, (long long)ld);
  if (T == 0 || E == 0) return SIMX_OK;  // nothing to compute (empty buffers may be NULL)
  if (!d_rew || !d_done || !d_ret) return fail(SIMX_EINVAL, "rewards, dones and returns are required");
  if (!std::isfinite(gamma)) return fail(SIMX_EINVAL, "gamma");
  if (lam >= 0.0f && (!d_val || !d_adv)) return fail(SIMX_EINVAL, "GAE needs values and an advantage buffer");
  cudaError_t e = launch_returns_gae(d_rew, d_val, d_done, d_last_val, T, E, ld, gamma, lam, d_ret,
                                     d_adv, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "returns launch");
  return SIMX_OK;
}

size_t returns_baseline_workspace_size(int64_t n) {
  return (size_t)baseline_blocks(n) * sizeof(double);
}

simx_status returns_baseline(const float* d_x, int64_t n, float* d_adv_out, float* d_mean_out,
                             void* d_workspace, size_t workspace_bytes, void* stream) {
  if (!d_x || n < 1) return fail(SIMX_EINVAL, "need n >= 1 returns");
  const int nb = baseline_blocks(n);
  if (!d_workspace || workspace_bytes < (size_t)nb * sizeof(double))
    return fail(SIMX_EINVAL, "workspace of %zu bytes needed", (size_t)nb * sizeof(double));
  cudaError_t e = launch_baseline(d_x, n, d_adv_out, d_mean_out, (double*)d_workspace, nb,
                                  (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "baseline launch");
  return SIMX_OK;
}

static simx_status loss_args(const simx_mlp* pol, const simx_rollout* buf, int64_t E,
                             const float* d_ret, const float* d_adv, const int64_t* d_idx,
                             int64_t n, const simx_loss_params* p, float* d_grad, float* d_stats,
                             LossArgs& a) {
  simx_status v = validate_mlp(pol, 0, 0);
  if (v != SIMX_OK) return v;
  if (n < 1) return fail(SIMX_EINVAL, "minibatch of %lld rows", (long long)n);
  if (!buf || !buf->obs || !buf->action) return fail(SIMX_EINVAL, "rollout obs and action are required");
  if (!p) return fail(SIMX_EINVAL, "loss params are NULL");
  if (p->algo != SIMX_ALGO_REINFORCE && p->algo != SIMX_ALGO_PPO) return fail(SIMX_EINVAL, "algo %d", p->algo);
  if (p->algo == SIMX_ALGO_PPO && !buf->logp) return fail(SIMX_EINVAL, "PPO needs logp_old");
  if (p->precision != SIMX_PREC_FP32 && p->precision != SIMX_PREC_TF32)
    return fail(SIMX_EINVAL, "precision %d", p->precision);
  if (!d_adv || !d_grad || !d_stats) return fail(SIMX_EINVAL, "adv, grad and stats are required");
  if (pol->has_value && !d_ret) return fail(SIMX_EINVAL, "a value row needs return targets");
  if (E < 1 || buf->ld != E) return fail(SIMX_EINVAL, "n_rows_per_step %lld must equal the rollout ld %lld", (long long)E, (long long)buf->ld);
  std::memset(&a, 0, sizeof(a));
  a.n_layers = pol->n_layers;
  a.has_value = pol->has_value ? 1 : 0;
  for (int l = 0; l <= pol->n_layers; ++l) a.dims[l] = pol->dims[l];
  for (int l = 0; l < pol->n_layers; ++l) {
    a.W[l] = pol->W[l];
    a.b[l] = pol->b[l];
    a.act[l] = (l + 1 < pol->n_layers) ? pol->act[l] : -1;
  }
  a.n_actions = pol->dims[pol->n_layers] - a.has_value;
  a.obs = buf->obs;
  a.action = buf->action;
  a.logp_old = buf->logp;
  a.ret = d_ret;
  a.adv = d_adv;
  a.E = E;
  a.idx = d_idx;
  a.n = n;
  a.algo = p->algo;
  a.clip_eps = p->clip_eps;
  a.c_value = p->c_value;
  a.c_entropy = p->c_entropy;
  a.precision = p->precision;
  a.grad = d_grad;
  a.stats = d_stats;
  a.grid = pol->grid ? 1 : 0;
  for (int l = 0; l < pol->n_layers; ++l) a.gx[l] = pol->grid ? pol->gx[l] : 0;
  if (a.grid && !loss_fused_fits(a))
    return fail(SIMX_EINVAL, "grid policy too large for the fused FP32 loss (its only path)");
  return SIMX_OK;
}

size_t ppo_loss_grad_workspace_size(const simx_mlp* pol, int64_t n) {
  if (!pol || pol->n_layers < 1 || pol->n_layers > SIMX_MAX_LAYERS || n < 1) return 0;
  LossArgs a;
  std::memset(&a, 0, sizeof(a));
  a.n_layers = pol->n_layers;
  for (int l = 0; l <= pol->n_layers; ++l) a.dims[l] = pol->dims[l];
  for (int l = 0; l < pol->n_layers; ++l) a.act[l] = (l + 1 < pol->n_layers) ? pol->act[l] : -1;
  a.grid = pol->grid ? 1 : 0;
  a.n = n;
  return loss_workspace_bytes(a);
}

simx_status ppo_loss_grad(const simx_mlp* pol, const simx_rollout* buf, int64_t n_rows_per_step,
                          const float* d_ret, const float* d_adv, const int64_t* d_idx, int64_t n,
                          const simx_loss_params* params, float* d_grad, float* d_stats,
                          void* d_workspace, size_t workspace_bytes, void* stream) {
  LossArgs a;
  simx_status v = loss_args(pol, buf, n_rows_per_step, d_ret, d_adv, d_idx, n, params, d_grad,
                            d_stats, a);
  if (v != SIMX_OK) return v;
  const size_t need = loss_workspace_bytes(a);
  if (!d_workspace || workspace_bytes < need)
    return fail(SIMX_EINVAL, "workspace of %zu bytes needed, %zu given", need, workspace_bytes);
  cudaError_t e = launch_loss_grad(a, d_workspace, workspace_bytes, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "loss launch");
  return SIMX_OK;
}

// ---------------------------------------------------------------------------
// Allocation-free loss gradient: the scratch is this file-scope device array.  Host
// code may not use its name as a device address (it is a host-side stand-in), so the
// address is looked up with cudaGetSymbolAddress, with the device current, on the first
// call on each device.  The address belongs to the device's context: after a device
// reset the module is loaded again and the array may move, so the cached address is
// kept together with the context's unique id and looked up again when that id changes.
// ---------------------------------------------------------------------------
static __device__ __align__(256) unsigned char g_noalloc_scratch[SIMX_NOALLOC_SCRATCH_BYTES];
static std::mutex g_noalloc_mu;
struct NoallocSlot {
  unsigned long long ctx_id;  // unique id of the context the address was found in
  void* ptr;
};
static NoallocSlot g_noalloc[64] = {};

// Unique id of the current context (cuCtxGetId, reached through the runtime's driver
// entry points so that the library links no driver library); false when there is no
// current context or the driver lacks the call.  Called with g_noalloc_mu held.
static bool current_ctx_id(unsigned long long* id) {
  static bool tried = false;
  static void* get_cur = nullptr;
  static void* get_id = nullptr;
  if (!tried) {
    tried = true;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &get_cur, 12000, cudaEnableDefault, &q) !=
            cudaSuccess || q != cudaDriverEntryPointSuccess)
      get_cur = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &get_id, 12000, cudaEnableDefault, &q) !=
            cudaSuccess || q != cudaDriverEntryPointSuccess)
      get_id = nullptr;
    cudaGetLastError();
  }
  if (!get_cur || !get_id) return false;
  CUcontext ctx = nullptr;
  if (reinterpret_cast<CUresult (*)(CUcontext*)>(get_cur)(&ctx) != CUDA_SUCCESS || !ctx) return false;
  return reinterpret_cast<CUresult (*)(CUcontext, unsigned long long*)>(get_id)(ctx, id) == CUDA_SUCCESS;
}

static simx_status noalloc_scratch(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= 64) return fail(SIMX_EINVAL, "device %d", dev);
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  NoallocSlot& slot = g_noalloc[dev];
  unsigned long long id = 0;
  const bool known = current_ctx_id(&id);
  if (!slot.ptr || !known || id != slot.ctx_id) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p) return cuda_fail(e, "cudaGetSymbolAddress(scratch)");
    slot.ptr = p;
    slot.ctx_id = current_ctx_id(&id) ? id : 0;
  }
  *out = slot.ptr;
  return SIMX_OK;
}

simx_status ppo_loss_grad_noalloc(const simx_mlp* pol, const simx_rollout* buf,
                                  int64_t n_rows_per_step, const float* d_ret, const float* d_adv,
                                  const int64_t* d_idx, int64_t n, const simx_loss_params* params,
                                  float* d_grad, float* d_stats, void* stream) {
  LossArgs a;
  simx_status v = loss_args(pol, buf, n_rows_per_step, d_ret, d_adv, d_idx, n, params, d_grad,
                            d_stats, a);
  if (v != SIMX_OK) return v;
  const size_t need = loss_workspace_bytes(a);
  if (need > SIMX_NOALLOC_SCRATCH_BYTES)
    return fail(SIMX_EINVAL, "this minibatch needs %zu bytes of scratch; the allocation-free entry "
                "point holds %zu (use ppo_loss_grad with a workspace)", need,
                (size_t)SIMX_NOALLOC_SCRATCH_BYTES);
  void* ws = nullptr;
  v = noalloc_scratch(&ws);
  if (v != SIMX_OK) return v;
  cudaError_t e = launch_loss_grad(a, ws, SIMX_NOALLOC_SCRATCH_BYTES, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "loss launch");
  return SIMX_OK;
}

static simx_status gather_stats(simx_ctx* c, unsigned long long host[9]) {
  cudaSetDevice(c->device);
  cudaError_t e = cudaStreamSynchronize(c->last);
  if (e != cudaSuccess) return cuda_fail(e, "synchronise");
  e = cudaMemset(c->stats, 0, 16 * sizeof(unsigned long long));
  if (e != cudaSuccess) return cuda_fail(e, "memset");
  e = launch_stats(c->st, c->stats, nullptr);
  if (e != cudaSuccess) return cuda_fail(e, "stats launch");
  e = cudaMemcpy(host, c->stats, 9 * sizeof(unsigned long long), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "stats copy");
  return SIMX_OK;
}

simx_status sim_stats(simx_ctx* c, simx_counters* out) {
  if (!c || !out) return fail(SIMX_EINVAL, "ctx or out is NULL");
  unsigned long long h[9];
  simx_status v = gather_stats(c, h);
  if (v != SIMX_OK) return v;
  out->arrived = h[0];
  out->dropped = h[1];
  out->dispatched = h[2];
  out->batches = h[3];
  out->queued = h[4];
  out->sum_wait_us = h[5];
  out->decisions = h[6];
  out->envs_flagged = (uint32_t)h[7];
  out->status_or = (uint32_t)h[8];
  return SIMX_OK;
}

simx_status simx_last_status(simx_ctx* c, uint32_t* code) {
  if (!c) return fail(SIMX_EINVAL, "ctx is NULL");
  unsigned long long h[9];
  simx_status v = gather_stats(c, h);
  if (v != SIMX_OK) return v;
  if (code) *code = (uint32_t)h[8];
  if (h[8]) return fail(SIMX_EOVERFLOW, "device status 0x%x in %llu envs", (unsigned)h[8], h[7]);
  return SIMX_OK;
}

static simx_status ensure_img(simx_ctx* c, uint64_t words) {
  if (c->img) return SIMX_OK;
  cudaError_t e = cudaMalloc(&c->img, words * sizeof(uint32_t));
  if (e != cudaSuccess) {
    c->img = nullptr;
    return fail(SIMX_ENOMEM, "cudaMalloc(state image of %llu words)", (unsigned long long)words);
  }
  return SIMX_OK;
}

simx_status sim_save(simx_ctx* c, uint32_t* host_buf, uint64_t n_words) {
  if (!c || !host_buf) return fail(SIMX_EINVAL, "ctx or buffer is NULL");
  const uint64_t sw = simx_state_words(&c->cfg), need = sw * c->cfg.n_envs;
  if (n_words < need) return fail(SIMX_EINVAL, "buffer of %llu words, %llu needed", (unsigned long long)n_words, (unsigned long long)need);
  cudaSetDevice(c->device);
  cudaError_t e = cudaStreamSynchronize(c->last);
  if (e != cudaSuccess) return cuda_fail(e, "synchronise");
  simx_status v = ensure_img(c, need);
  if (v != SIMX_OK) return v;
  e = launch_save(c->st, c->cfg.cost_type, sw, c->img, nullptr);
  if (e != cudaSuccess) return cuda_fail(e, "save launch");
  e = cudaMemcpy(host_buf, c->img, need * sizeof(uint32_t), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "save copy");
  return SIMX_OK;
}

simx_status sim_load(simx_ctx* c, const uint32_t* host_buf, uint64_t n_words) {
  if (!c || !host_buf) return fail(SIMX_EINVAL, "ctx or buffer is NULL");
  const uint64_t sw = simx_state_words(&c->cfg), need = sw * c->cfg.n_envs;
  if (n_words < need) return fail(SIMX_EINVAL, "buffer of %llu words, %llu needed", (unsigned long long)n_words, (unsigned long long)need);
  if (!c->seeded) return fail(SIMX_ESTATE, "sim_load needs the Philox key of a prior sim_reset");
  const uint32_t cap = c->cfg.queue_cap;
  for (uint64_t e = 0; e < c->cfg.n_envs; ++e) {  // queue lengths must fit the rings
    const uint32_t* q = host_buf + e * sw + SIMX_STATE_HEADER_WORDS + 2 * c->cfg.n_servers;
    for (uint32_t i = 0; i < c->cfg.n_servers * c->cfg.n_types; ++i)
      if (q[i] > cap) return fail(SIMX_EINVAL, "env %llu: queue length %u > capacity %u", (unsigned long long)e, q[i], cap);
  }
  cudaSetDevice(c->device);
  cudaError_t e = cudaStreamSynchronize(c->last);
  if (e != cudaSuccess) return cuda_fail(e, "synchronise");
  simx_status v = ensure_img(c, need);
  if (v != SIMX_OK) return v;
  e = cudaMemcpy(c->img, host_buf, need * sizeof(uint32_t), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return cuda_fail(e, "load copy");
  e = launch_load(c->st, c->cfg.cost_type, sw, c->img, nullptr);
  if (e != cudaSuccess) return cuda_fail(e, "load launch");
  e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(e, "load");
  return SIMX_OK;
}

}  // extern "C"
