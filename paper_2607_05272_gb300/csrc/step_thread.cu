// step_thread.cu — the simulator step with one thread per environment, for the
// policy-free modes (Sec. 5.1 baselines Static, Random, Round-Robin, Shortest-Queue,
// and caller-supplied actions).
//
// Without the policy network a step is a short sequence of integer event work per
// env, so each env gets one thread: the structure-of-arrays state is read and
// written with one coalesced access per field for 32 envs, the K servers are
// unrolled into registers (K in {1, 2, 4, 8}), arrivals are drawn one candidate at
// a time, and the records are written coalesced across envs.  The event semantics are
// those of the lane-group kernel (rollout.cu) and of the oracle, step for step.
#include <cstdint>

#include "kernels.h"

namespace simx {

namespace {

template <int K>
struct TEnv {
  uint32_t now, tg, cj, cT, swi, swT, mst, ep, epo, pt, pty, pc;
  uint32_t narr, ndrop, ndisp, nbat, tld, prev, nlast, tlast, na0, na1, nd0, nd1, status, events;
  uint64_t swait;
  float lmw, rate, ep_factor;
  uint32_t ep_cached;
  uint32_t busy[K], bsize[K], qh0[K], qh1[K], qc0[K], qc1[K];
};

__device__ __forceinline__ uint32_t t_add(uint32_t a, uint64_t b, uint32_t& status) {
  const uint64_t s = (uint64_t)a + b;
  if (s >= kTimeLimit) {
    status |= kStTime;
    return kTimeLimit;
  }
  return (uint32_t)s;
}

struct Ctx {
  const RolloutArgs& A;
  uint32_t env;
  uint32_t* ring;  // this env's rings [K][T][cap]
  uint32_t* cost;  // this env's cost rings [K][cap] or null
};

__device__ __forceinline__ uint32_t t_type(const simx_config& c, uint32_t w1) {
  return (c.n_types > 1 && (w1 >> 8) >= c.type0_thr) ? 1u : 0u;
}

__device__ __forceinline__ uint32_t t_cost(const simx_config& c, uint32_t w3) {
  const float E = expo1(w3);
  if (c.cost_kind == 0) return duration_us(__fmul_rn(c.cost_scale_us, det_exp(__fmul_rn(c.pareto_inv_alpha, E))));
  return duration_us(__fmul_rn(c.cost_scale_us, E));
}

template <int K>
__device__ __forceinline__ bool t_count(TEnv<K>& s) {
  if (++s.events > kEventCap) {
    s.status |= kStEvent;
    return true;
  }
  return false;
}

template <int K>
__device__ void t_switches(const Ctx& x, TEnv<K>& s, uint32_t limit) {
  if (x.A.cfg.n_mod_states < 2) return;
  while (s.swT <= limit) {
    if (t_count(s)) return;
    s.mst ^= 1u;
    s.swi += 1u;
    if (x.A.cfg.dwell_kind == 1) {  // fixed dwell: a square wave
      s.swT = t_add(s.swT, duration_us(x.A.cfg.dwell_mean_us), s.status);
    } else {
      const U4 w = philox(s.swi, x.env, kStreamSwitch, 0u, x.A.key0, x.A.key1);
      s.swT = t_add(s.swT, duration_us(__fmul_rn(x.A.cfg.dwell_mean_us, expo1(w.x))), s.status);
    }
  }
}

// Candidate s.cj: its Philox words and its time (a drawn gap, or under trace replay,
// TR, entry cj mod n of the trace).  TR is a template parameter so that the generated-
// arrival kernels carry none of the trace code.
template <int K, bool TR>
__device__ __forceinline__ uint32_t t_cand(const Ctx& x, TEnv<K>& s, U4& w) {
  w = philox(s.cj, x.env, kStreamArrival, 0u, x.A.key0, x.A.key1);
  const uint32_t gap = TR ? x.A.tr_gap[s.cj % x.A.tr_n]
                          : duration_us(__fmul_rn(x.A.cfg.cand_mean_gap_us, expo1(w.x)));
  return t_add(s.cT, gap, s.status);
}

// Type and cost of candidate j: the trace's when it has them, else drawn.
template <bool TR>
__device__ __forceinline__ uint32_t t_cand_type(const RolloutArgs& A, uint32_t j, uint32_t w1) {
  if (TR && A.tr_type) {
    const uint32_t t = A.tr_type[j % A.tr_n];
    return t < A.cfg.n_types ? t : A.cfg.n_types - 1u;
  }
  return t_type(A.cfg, w1);
}

template <bool TR>
__device__ __forceinline__ uint32_t t_cand_cost(const RolloutArgs& A, uint32_t j, uint32_t w3) {
  return (TR && A.tr_cost) ? A.tr_cost[j % A.tr_n] : t_cost(A.cfg, w3);
}

// SINGLE mode: an accepted candidate joins its type's FIFO or is dropped.
template <int K, bool TR>
__device__ bool t_consume(const Ctx& x, TEnv<K>& s, const U4& w, uint32_t T) {
  const simx_config& c = x.A.cfg;
  if (!((w.z >> 8) < c.accept_thr[s.mst])) return false;
  const uint32_t ty = t_cand_type<TR>(x.A, s.cj, w.y);
  const uint32_t cap = c.queue_cap;
  s.narr += 1u;
  if (ty) s.na1 += 1u; else s.na0 += 1u;
  const uint32_t q = ty ? s.qc1[0] : s.qc0[0];
  if (q < cap) {
    const uint32_t slot = ((ty ? s.qh1[0] : s.qh0[0]) + q) & (cap - 1u);
    x.ring[ty * cap + slot] = T;
    if ((int32_t)ty == c.cost_type) x.cost[slot] = t_cand_cost<TR>(x.A, s.cj, w.w);
    if (ty) s.qc1[0] += 1u; else s.qc0[0] += 1u;
  } else {
    s.ndrop += 1u;
    if (ty) s.nd1 += 1u; else s.nd0 += 1u;
  }
  return true;
}

template <int K, bool TR>
__device__ void t_advance(const Ctx& x, TEnv<K>& s, uint32_t target) {
  for (;;) {
    U4 w;
    const uint32_t T = t_cand<K, TR>(x, s, w);
    if (T > target) break;
    if (t_count(s)) return;
    t_switches(x, s, T);
    t_consume<K, TR>(x, s, w, T);
    s.cj += 1u;
    s.cT = T;
  }
  t_switches(x, s, target);
}

template <int K, bool TR>
__device__ void t_jump(const Ctx& x, TEnv<K>& s) {
  for (;;) {
    U4 w;
    const uint32_t T = t_cand<K, TR>(x, s, w);
    if (t_count(s)) return;
    t_switches(x, s, T);
    const bool acc = t_consume<K, TR>(x, s, w, T);
    s.cj += 1u;
    s.cT = T;
    if (acc) {
      s.now = T;
      t_advance<K, TR>(x, s, T);
      return;
    }
  }
}

// ROUTE mode: the next arrival into the pending slot.
template <int K, bool TR>
__device__ void t_next_arrival(const Ctx& x, TEnv<K>& s) {
  const simx_config& c = x.A.cfg;
  for (;;) {
    if (t_count(s)) return;
    U4 w;
    if (TR || c.arrival_kind != SIMX_ARR_DIURNAL) {  // THINNED or TRACE
      const uint32_t T = t_cand<K, TR>(x, s, w);
      t_switches(x, s, T);
      const bool acc = (w.z >> 8) < c.accept_thr[s.mst];
      const uint32_t j = s.cj;
      s.cj += 1u;
      s.cT = T;
      if (!acc) continue;
      s.pty = t_cand_type<TR>(x.A, j, w.y);
      s.pc = ((int32_t)s.pty == c.cost_type) ? t_cand_cost<TR>(x.A, j, w.w) : 0u;
      s.pt = T;
      s.narr += 1u;
      return;
    }
    if (s.ep_cached != s.ep) {
      const U4 we = philox(s.ep, x.env, kStreamEpoch, 0u, x.A.key0, x.A.key1);
      s.ep_factor = det_exp(__fmul_rn(c.burst_sigma, normal01(we.x, we.y)));
      s.ep_cached = s.ep;
    }
    const float rate = __fmul_rn(c.diurnal_rate[(s.ep + s.epo) % c.diurnal_len], s.ep_factor);
    const float mean = __fdiv_rn(1.0e6f, rate);
    w = philox(s.cj, x.env, kStreamArrival, 0u, x.A.key0, x.A.key1);
    const uint32_t gap = duration_us(__fmul_rn(mean, expo1(w.x)));
    s.cj += 1u;
    const uint64_t end = (uint64_t)(s.ep + 1u) * (uint64_t)c.epoch_us;
    if ((uint64_t)s.cT + gap < end) {
      s.cT = t_add(s.cT, gap, s.status);
      s.pt = s.cT;
      s.pty = t_type(c, w.y);
      s.pc = ((int32_t)s.pty == c.cost_type) ? t_cost(c, w.w) : 0u;
      s.narr += 1u;
      return;
    }
    if (end >= kTimeLimit) {
      s.status |= kStTime;
      s.cT = kTimeLimit;
    } else {
      s.cT = (uint32_t)end;
    }
    s.ep += 1u;
  }
}

// Batch time L on server k scaled by its speed s/16, rounded to the nearest microsecond.
__device__ __forceinline__ uint64_t t_speed(const simx_config& c, int k, uint64_t L) {
  const uint64_t s = c.srv_speed16[k] ? c.srv_speed16[k] : 16u;
  return (L * s + 8u) >> 4;
}

// ROUTE mode: one server's queue state, selected out of the register arrays by unrolled
// selects so that the batch start below is emitted once per call site instead of once per
// server (the K-fold copies made the kernel's instruction fetch its largest stall).
struct Srv {
  uint32_t busy, bsize, qh0, qc0, qh1, qc1;
};

template <int K>
__device__ __forceinline__ Srv srv_get(const TEnv<K>& s, int i) {
  Srv r{s.busy[0], s.bsize[0], s.qh0[0], s.qc0[0], s.qh1[0], s.qc1[0]};
#pragma unroll
  for (int k = 1; k < K; ++k)
    if (i == k) r = Srv{s.busy[k], s.bsize[k], s.qh0[k], s.qc0[k], s.qh1[k], s.qc1[k]};
  return r;
}

template <int K>
__device__ __forceinline__ void srv_put(TEnv<K>& s, int i, const Srv& r) {
#pragma unroll
  for (int k = 0; k < K; ++k)
    if (i == k) {
      s.busy[k] = r.busy;
      s.bsize[k] = r.bsize;
      s.qh0[k] = r.qh0;
      s.qc0[k] = r.qc0;
      s.qh1[k] = r.qh1;
      s.qc1[k] = r.qc1;
    }
}

// ROUTE mode: server i (state r) starts a batch at time st (the oldest-head type, tie:
// type 0).
template <int K>
__device__ __forceinline__ void t_start(const Ctx& x, TEnv<K>& s, Srv& r, int i, uint32_t st,
                                        uint32_t& stn, uint64_t& w0, uint64_t& w1) {
  const simx_config& c = x.A.cfg;
  const uint32_t cap = c.queue_cap, T = c.n_types;
  uint32_t* rs = x.ring + (size_t)i * T * cap;
  uint32_t h;
  if (r.qc0 > 0u && r.qc1 > 0u) {
    h = rs[cap + r.qh1] < rs[r.qh0] ? 1u : 0u;
  } else if (r.qc0 > 0u) {
    h = 0u;
  } else if (r.qc1 > 0u) {
    h = 1u;
  } else {
    return;
  }
  const uint32_t qn = h ? r.qc1 : r.qc0;
  const uint32_t head = h ? r.qh1 : r.qh0;
  const uint32_t n = r.bsize < qn ? r.bsize : qn;
  const bool costed = (int32_t)h == c.cost_type;
  uint64_t W = 0, csum = 0;
  for (uint32_t j = 0; j < n; ++j) {
    const uint32_t slot = (head + j) & (cap - 1u);
    W += (uint64_t)(st - rs[h * cap + slot]);
    if (costed) csum += x.cost[(size_t)i * cap + slot];
  }
  if (h) {
    r.qh1 = (head + n) & (cap - 1u);
    r.qc1 -= n;
  } else {
    r.qh0 = (head + n) & (cap - 1u);
    r.qc0 -= n;
  }
  const uint64_t L = costed ? (uint64_t)c.alpha_us[h] + csum
                            : (uint64_t)c.alpha_us[h] + (uint64_t)c.beta_us[h] * n;
  r.busy = t_add(st, t_speed(c, i, L), s.status);
  stn += n;
  if (h) w1 += W; else w0 += W;
  s.ndisp += n;
  s.swait += W;
  s.nbat += 1u;
}

template <int K>
__device__ __forceinline__ uint32_t t_queued(const TEnv<K>& s) {
  uint32_t q = 0;
#pragma unroll
  for (int i = 0; i < K; ++i) q += s.qc0[i] + s.qc1[i];
  return q;
}

// Observation (Sec. 4.1; the layouts of rollout.cu) into obs[d * ld].
// q / cap for a power-of-two capacity: multiplying by the exact reciprocal 2^-k gives
// the bits of the IEEE division (no rounding either way for these small integers).
__device__ __forceinline__ float over_cap(uint32_t q, float inv_cap) {
  return __fmul_rn(__uint2float_rn(q), inv_cap);
}

template <bool ROUTE, int K>
__device__ void t_observe(const Ctx& x, const TEnv<K>& s, float* o, int64_t ld) {
  const simx_config& c = x.A.cfg;
  const float fcap = __uint2float_rn(c.queue_cap);
  const float inv_cap = __fdiv_rn(1.0f, fcap);
  int i = 0;
  if (!ROUTE) {
    const uint32_t T = c.n_types, cap = c.queue_cap;
    const bool ne0 = s.qc0[0] > 0u, ne1 = T > 1 && s.qc1[0] > 0u;
    const uint32_t h0 = ne0 ? x.ring[s.qh0[0]] : 0u, h1 = ne1 ? x.ring[cap + s.qh1[0]] : 0u;
    const uint32_t head = ne0 ? ((ne1 && h1 < h0) ? 1u : 0u) : (ne1 ? 1u : kNone);
    uint32_t dt = s.now - s.prev;
    if (dt < 1u) dt = 1u;
    const float fdt = __uint2float_rn(dt), tw = c.t_window_us;
    o[(i++) * ld] = over_cap(s.qc0[0], inv_cap);
    if (T > 1) o[(i++) * ld] = over_cap(s.qc1[0], inv_cap);
    o[(i++) * ld] = __fdiv_rn(__uint2float_rn(s.now - s.tld), tw);
    o[(i++) * ld] = head == 0u ? 1.0f : 0.0f;
    o[(i++) * ld] = head == 1u ? 1.0f : 0.0f;
    o[(i++) * ld] = 0.0f;
    o[(i++) * ld] = __fdiv_rn(__fmul_rn(__uint2float_rn(s.na0 + s.na1), c.rate_scale), fdt);
    o[(i++) * ld] = __fdiv_rn(__uint2float_rn(s.nlast), 32.0f);
    o[(i++) * ld] = ne0 ? __fdiv_rn(__uint2float_rn(s.now - h0), tw) : 0.0f;
    if (T > 1) o[(i++) * ld] = ne1 ? __fdiv_rn(__uint2float_rn(s.now - h1), tw) : 0.0f;
    if (c.obs_extra) {
      o[(i++) * ld] = __fdiv_rn(__fmul_rn(__uint2float_rn(s.na0), c.rate_scale), fdt);
      o[(i++) * ld] = __fdiv_rn(__fmul_rn(__uint2float_rn(s.na1), c.rate_scale), fdt);
      o[(i++) * ld] = s.tlast == 0u ? 1.0f : 0.0f;
      o[(i++) * ld] = s.tlast == 1u ? 1.0f : 0.0f;
      o[(i++) * ld] = __fdiv_rn(__uint2float_rn(s.nd0 + s.nd1), 32.0f);
      o[(i++) * ld] = __fdiv_rn(s.lmw, tw);
    }
    return;
  } else {
#pragma unroll
  for (int k = 0; k < K; ++k) {
    o[(i++) * ld] = over_cap(s.qc0[k], inv_cap);
    o[(i++) * ld] = over_cap(c.n_types > 1 ? s.qc1[k] : 0u, inv_cap);
    const uint32_t rem = s.busy[k] > s.now ? s.busy[k] - s.now : 0u;
    o[(i++) * ld] = __fdiv_rn(__uint2float_rn(rem), c.busy_norm_us);
  }
  o[(i++) * ld] = __fdiv_rn(s.rate, c.rate_ref);
  if (c.obs_extra) {
    o[(i++) * ld] = s.pty == 0u ? 1.0f : 0.0f;
    o[(i++) * ld] = s.pty == 1u ? 1.0f : 0.0f;
    const uint32_t ph = (s.now + s.epo * c.epoch_us) % c.phase_period_us;
    o[(i++) * ld] = __fdiv_rn(__uint2float_rn(ph), __uint2float_rn(c.phase_period_us));
  }
  }
}

template <bool ROUTE, int K>
__device__ int t_action(const Ctx& x, TEnv<K>& s) {
  const RolloutArgs& A = x.A;
  const simx_config& c = A.cfg;
  const int mode = A.policy_mode;
  if (mode == SIMX_POLICY_EXTERNAL) {
    const int32_t a = A.ext[x.env];
    if (a < 0 || (uint32_t)a >= A.n_actions) {
      s.status |= kStAction;
      return 0;
    }
    return a;
  }
  if (mode == SIMX_POLICY_RANDOM) {
    const U4 w = philox(s.tg, x.env, kStreamPolicy, 0u, A.key0, A.key1);
    return (int)(((uint64_t)(w.y >> 8) * A.n_actions) >> 24);
  }
  if (!ROUTE) {  // STATIC
    uint32_t h = 0;
    const uint32_t cap = c.queue_cap;
    if (s.qc0[0] > 0u && c.n_types > 1 && s.qc1[0] > 0u) h = x.ring[cap + s.qh1[0]] < x.ring[s.qh0[0]] ? 1u : 0u;
    else if (s.qc0[0] == 0u && c.n_types > 1 && s.qc1[0] > 0u) h = 1u;
    return (int)((c.action_layout == 1 ? 1u : 0u) + h * c.n_bsizes + c.static_bi);
  }
  if (mode == SIMX_POLICY_RR) return (int)((s.tg % c.n_servers) * c.n_bsizes + c.static_bi);
  int best = 0;
  uint32_t bq = 0xFFFFFFFFu;
#pragma unroll
  for (int k = 0; k < K; ++k) {
    const uint32_t q = s.qc0[k] + s.qc1[k];
    if (q < bq) {
      bq = q;
      best = k;
    }
  }
  return best * (int)c.n_bsizes + (int)c.static_bi;
}

// MINB resident 128-thread blocks per SM bound the registers (4: 128).  The latency of
// one env-step is a long dependent chain, so the step rate is the number of resident
// threads over that latency: more residency beats more registers.
template <bool ROUTE, int K, int MINB, bool TR>
__global__ void __launch_bounds__(128, MINB) k_step_thread(const __grid_constant__ RolloutArgs A) {
  // Programmatic dependent launch: the next step's blocks may be scheduled as soon as every
  // block of this one has started; each waits here until the previous grid has completed
  // and its stores are visible, before it reads or writes any state.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const uint32_t env = blockIdx.x * blockDim.x + threadIdx.x;
  if (env >= A.st.E) return;
  const DevState& st = A.st;
  const simx_config& c = A.cfg;
  const uint32_t E = st.E, T = c.n_types, cap = c.queue_cap;
  Ctx x{A, env, st.ring + (size_t)env * K * T * cap, st.cost ? st.cost + (size_t)env * K * cap : nullptr};
  TEnv<K> s;
  const uint32_t* h = st.hdr;
  s.now = h[F_NOW * E + env];
  s.tg = h[F_TG * E + env];
  s.cj = h[F_CJ * E + env];
  s.cT = h[F_CT * E + env];
  s.swi = h[F_SWI * E + env];
  s.swT = h[F_SWT * E + env];
  s.mst = h[F_MST * E + env];
  s.ep = h[F_EP * E + env];
  s.epo = h[F_EPO * E + env];
  s.pt = h[F_PT * E + env];
  s.pty = h[F_PTY * E + env];
  s.pc = h[F_PC * E + env];
  s.narr = h[F_NARR * E + env];
  s.ndrop = h[F_NDROP * E + env];
  s.ndisp = h[F_NDISP * E + env];
  s.nbat = h[F_NBAT * E + env];
  s.swait = (uint64_t)h[F_SWLO * E + env] | ((uint64_t)h[F_SWHI * E + env] << 32);
  s.tld = h[F_TLD * E + env];
  s.prev = h[F_PREV * E + env];
  s.nlast = h[F_NLAST * E + env];
  s.tlast = h[F_TLAST * E + env];
  s.lmw = __uint_as_float(h[F_LMW * E + env]);
  s.rate = __uint_as_float(h[F_RATE * E + env]);
  s.na0 = h[F_NA0 * E + env];
  s.na1 = h[F_NA1 * E + env];
  s.nd0 = h[F_ND0 * E + env];
  s.nd1 = h[F_ND1 * E + env];
  s.status = h[F_STATUS * E + env];
  s.events = 0;
  s.ep_cached = kNone;
  s.ep_factor = 0.0f;
#pragma unroll
  for (int k = 0; k < K; ++k) {
    s.busy[k] = st.srv[(0 * K + k) * E + env];
    s.bsize[k] = st.srv[(1 * K + k) * E + env];
    s.qh0[k] = st.qh[(k * T + 0) * E + env];
    s.qc0[k] = st.qc[(k * T + 0) * E + env];
    s.qh1[k] = T > 1 ? st.qh[(k * T + 1) * E + env] : 0u;
    s.qc1[k] = T > 1 ? st.qc[(k * T + 1) * E + env] : 0u;
  }

  for (int t = 0; t < A.H; ++t) {
    if (A.obs) t_observe<ROUTE, K>(x, s, A.obs + (int64_t)t * A.obs_dim * A.ld + env, A.ld);
    const int a = t_action<ROUTE, K>(x, s);
    uint32_t kk, b;
    if (c.action_layout == 1) {  // a = 0: Wait (batch 0); a >= 1: type, batch 1 .. n_bsizes
      kk = a == 0 ? 0u : (uint32_t)(a - 1) / c.n_bsizes;
      b = a == 0 ? 0u : (uint32_t)(a - 1) % c.n_bsizes + 1u;
    } else {
      kk = (uint32_t)a / c.n_bsizes;
      b = c.bsizes[(uint32_t)a % c.n_bsizes];
    }
    const bool frozen = s.status != 0;
    const uint32_t now = ROUTE ? s.pt : s.now;
    uint32_t n_step = 0, qafter;
    uint64_t w_step = 0;
    float reward;
    if (!ROUTE) {
      uint32_t n = 0;
      uint64_t W = 0, csum = 0;
      if (!frozen) {
        const uint32_t q = kk ? s.qc1[0] : s.qc0[0];
        const uint32_t head = kk ? s.qh1[0] : s.qh0[0];
        n = b < q ? b : q;
        for (uint32_t j = 0; j < n; ++j) {
          const uint32_t slot = (head + j) & (cap - 1u);
          W += (uint64_t)(now - x.ring[kk * cap + slot]);
          if ((int32_t)kk == c.cost_type) csum += x.cost[slot];
        }
        if (kk) {
          s.qh1[0] = (head + n) & (cap - 1u);
          s.qc1[0] -= n;
        } else {
          s.qh0[0] = (head + n) & (cap - 1u);
          s.qc0[0] -= n;
        }
        if (n > 0) {
          const uint64_t L = ((int32_t)kk == c.cost_type)
                                 ? (uint64_t)c.alpha_us[kk] + csum
                                 : (uint64_t)c.alpha_us[kk] + (uint64_t)c.beta_us[kk] * n;
          s.busy[0] = t_add(now, t_speed(c, 0, L), s.status);
          s.nlast = n;
          s.tlast = kk;
          s.tld = now;
          s.lmw = __fdiv_rn(__ull2float_rn(W), __uint2float_rn(n));
          s.nbat += 1u;
        }
        s.ndisp += n;
        s.swait += W;
      }
      reward = __fsub_rn(__uint2float_rn(n), __fmul_rn(c.w_wait[kk], __ull2float_rn(W)));
      n_step = n;
      w_step = W;
      qafter = t_queued(s);
      s.prev = now;
      s.na0 = s.na1 = s.nd0 = s.nd1 = 0u;
      s.tg += 1u;
      if (!frozen) {
        s.events = 0;
        if (n > 0) {
          const uint32_t next = s.busy[0];
          t_advance<K, TR>(x, s, next);
          s.now = next;
          if (t_queued(s) == 0u) t_jump<K, TR>(x, s);
        } else {
          t_jump<K, TR>(x, s);
        }
      }
    } else {
      const uint32_t mt = s.pty;
      uint32_t stn = 0;
      uint64_t w0 = 0, w1 = 0;
      if (!frozen) {
        s.events = 0;
        bool go = false;
#pragma unroll
        for (int k = 0; k < K; ++k) {
          if ((uint32_t)k != kk) continue;
          const uint32_t q = mt ? s.qc1[k] : s.qc0[k];
          if (q < cap) {
            const uint32_t slot = ((mt ? s.qh1[k] : s.qh0[k]) + q) & (cap - 1u);
            x.ring[((size_t)k * T + mt) * cap + slot] = now;
            if ((int32_t)mt == c.cost_type) x.cost[(size_t)k * cap + slot] = s.pc;
            if (mt) s.qc1[k] += 1u; else s.qc0[k] += 1u;
          } else {
            s.ndrop += 1u;
            if (mt) s.nd1 += 1u; else s.nd0 += 1u;
          }
          s.bsize[k] = b;
          go = s.busy[k] <= now;
        }
        if (go) {  // the routed-to server is free: it starts a batch now
          Srv r = srv_get<K>(s, (int)kk);
          t_start<K>(x, s, r, (int)kk, now, stn, w0, w1);
          srv_put<K>(s, (int)kk, r);
        }
        qafter = t_queued(s);
        t_next_arrival<K, TR>(x, s);
        uint32_t gap = s.pt - now;
        if (gap < 1u) gap = 1u;
        const float inst = __fdiv_rn(1.0e6f, __uint2float_rn(gap));
        s.rate = __fadd_rn(s.rate, __fmul_rn(0.0625f, __fsub_rn(inst, s.rate)));
        // every server free by the next arrival starts batches, server by server in
        // index order (one copy of the batch start for all servers)
        for (;;) {
          int k = -1;  // the lowest-index server free by then with requests queued
#pragma unroll
          for (int j = K - 1; j >= 0; --j)
            if (s.busy[j] <= s.pt && (s.qc0[j] + s.qc1[j]) > 0u) k = j;
          if (k < 0) break;
          Srv r = srv_get<K>(s, k);
          t_start<K>(x, s, r, k, r.busy, stn, w0, w1);
          srv_put<K>(s, k, r);
        }
        s.now = s.pt;
      } else {
        qafter = t_queued(s);
      }
      reward = __fsub_rn(__uint2float_rn(stn),
                         __fadd_rn(__fmul_rn(c.w_wait[0], __ull2float_rn(w0)),
                                   __fmul_rn(c.w_wait[1], __ull2float_rn(w1))));
      n_step = stn;
      w_step = w0 + w1;
      s.prev = now;
      s.tg += 1u;
    }
    const int64_t o = (int64_t)t * A.ld + env;
    if (A.action) A.action[o] = (uint8_t)a;
    if (A.logp) A.logp[o] = 0.0f;
    if (A.value) A.value[o] = 0.0f;
    if (A.reward) A.reward[o] = reward;
    if (A.done) A.done[o] = (uint8_t)((s.tg % c.episode_len) == 0u);
    if (A.trace) {
      int64_t* tr = A.trace + (int64_t)t * SIMX_TRACE_WIDTH * A.ld + env;
      tr[0] = now;
      tr[A.ld] = n_step;
      tr[2 * A.ld] = (int64_t)w_step;
      tr[3 * A.ld] = qafter;
    }
  }
  if (A.next_obs) t_observe<ROUTE, K>(x, s, A.next_obs + env, A.next_ld);

  uint32_t* hw = st.hdr;
  hw[F_NOW * E + env] = s.now;
  hw[F_TG * E + env] = s.tg;
  hw[F_CJ * E + env] = s.cj;
  hw[F_CT * E + env] = s.cT;
  hw[F_SWI * E + env] = s.swi;
  hw[F_SWT * E + env] = s.swT;
  hw[F_MST * E + env] = s.mst;
  hw[F_EP * E + env] = s.ep;
  hw[F_EPO * E + env] = s.epo;
  hw[F_PT * E + env] = s.pt;
  hw[F_PTY * E + env] = s.pty;
  hw[F_PC * E + env] = s.pc;
  hw[F_NARR * E + env] = s.narr;
  hw[F_NDROP * E + env] = s.ndrop;
  hw[F_NDISP * E + env] = s.ndisp;
  hw[F_NBAT * E + env] = s.nbat;
  hw[F_SWLO * E + env] = (uint32_t)s.swait;
  hw[F_SWHI * E + env] = (uint32_t)(s.swait >> 32);
  hw[F_TLD * E + env] = s.tld;
  hw[F_PREV * E + env] = s.prev;
  hw[F_NLAST * E + env] = s.nlast;
  hw[F_TLAST * E + env] = s.tlast;
  hw[F_LMW * E + env] = __float_as_uint(s.lmw);
  hw[F_RATE * E + env] = __float_as_uint(s.rate);
  hw[F_NA0 * E + env] = s.na0;
  hw[F_NA1 * E + env] = s.na1;
  hw[F_ND0 * E + env] = s.nd0;
  hw[F_ND1 * E + env] = s.nd1;
  hw[F_STATUS * E + env] = s.status;
#pragma unroll
  for (int k = 0; k < K; ++k) {
    st.srv[(0 * K + k) * E + env] = s.busy[k];
    st.srv[(1 * K + k) * E + env] = s.bsize[k];
    st.qh[(k * T + 0) * E + env] = s.qh0[k];
    st.qc[(k * T + 0) * E + env] = s.qc0[k];
    if (T > 1) {
      st.qh[(k * T + 1) * E + env] = s.qh1[k];
      st.qc[(k * T + 1) * E + env] = s.qc1[k];
    }
  }
}

// 4 resident blocks per SM (128 registers): one wave of 77,824 envs; from 262,144 envs 5
// (96 registers; 6 would spill the server state of the router).  Launched with programmatic stream serialization
// so that back-to-back steps (a graph of sim_step_batched calls) overlap one step's block
// launch with the previous step's tail; the kernel's griddepcontrol.wait keeps the order.
template <bool ROUTE, int K>
cudaError_t step_thread_t(const RolloutArgs& a, cudaStream_t s) {
  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3((a.st.E + 127) / 128);
  lc.blockDim = dim3(128);
  lc.dynamicSmemBytes = 0;
  lc.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  lc.attrs = at;
  lc.numAttrs = 1;
  // from 262,144 envs (several waves) five resident blocks per SM (96 registers, no
  // spills) beat four: 124.8 against 126.8 us per step at 1,048,576 envs; below that the
  // single wave of four blocks with 128 registers is faster (8.6 against 10.2 us at 65,536)
  const bool tr = a.cfg.arrival_kind == SIMX_ARR_TRACE;
  cudaError_t e;
  if (a.st.E >= 262144u)
    e = tr ? cudaLaunchKernelEx(&lc, k_step_thread<ROUTE, K, 5, true>, a)
           : cudaLaunchKernelEx(&lc, k_step_thread<ROUTE, K, 5, false>, a);
  else
    e = tr ? cudaLaunchKernelEx(&lc, k_step_thread<ROUTE, K, 4, true>, a)
           : cudaLaunchKernelEx(&lc, k_step_thread<ROUTE, K, 4, false>, a);
  count_launches(1);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

bool step_thread_supported(const RolloutArgs& a) {
  const int m = a.policy_mode;
  if (m == SIMX_POLICY_SAMPLE || m == SIMX_POLICY_ARGMAX) return false;
  const uint32_t K = a.cfg.n_servers;
  return K == 1 || K == 2 || K == 4 || K == 8;
}

cudaError_t launch_step_thread(const RolloutArgs& a, cudaStream_t s) {
  const bool route = a.cfg.mode == SIMX_MODE_ROUTE;
  switch (a.cfg.n_servers) {
    case 1: return route ? step_thread_t<true, 1>(a, s) : step_thread_t<false, 1>(a, s);
    case 2: return route ? step_thread_t<true, 2>(a, s) : cudaErrorInvalidValue;
    case 4: return route ? step_thread_t<true, 4>(a, s) : cudaErrorInvalidValue;
    case 8: return route ? step_thread_t<true, 8>(a, s) : cudaErrorInvalidValue;
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace simx
