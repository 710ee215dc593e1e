// rollout.cu — the batched discrete-event inference-serving simulator of
// "Adaptive Inference Batching using Policy Gradients" (Sec. 3.1 dynamics, Sec. 3.2
// workloads, Sec. 4.1 MDP) with the policy of Sec. 4.2 fused into the step.
//
// One lane group (G = 8 lanes) per environment, four environments per warp.  A
// launch runs H decision steps of every environment with its state in registers:
// rollout_collect uses H = horizon; sim_step_batched uses H = 1.
#include <cstdint>
#include <cstdlib>
#include <cstring>

#include "kernels.h"
#include "sim.cuh"
#include "tc_common.cuh"

namespace simx {

// Env kernels run blocks of 64, 128 or 256 threads (chosen per launch); an env is a
// group of G lanes (G = 8, 16 or 32, also chosen per launch), so a block holds
// blockDim.x / G envs.  At least 2 resident 256-thread blocks (16 warps) per SM caps
// registers at 128 per thread.
constexpr int kMaxThreads = 256;
#ifndef SIMX_MIN_BLOCKS
#define SIMX_MIN_BLOCKS 2
#endif
#ifndef SIMX_MIN_BLOCKS_32
#define SIMX_MIN_BLOCKS_32 SIMX_MIN_BLOCKS
#endif
// Resident 256-thread blocks per SM the register allocation must allow (one env per
// warp needs more warps resident than narrower groups do).
template <int G>
constexpr int min_blocks() { return G == 32 ? SIMX_MIN_BLOCKS_32 : SIMX_MIN_BLOCKS; }

// Two values indexed by a runtime 0/1 through selects, so that the structs below
// stay in registers (a dynamically indexed array would be placed in local memory).
struct Pair {
  uint32_t v0, v1;
  __device__ __forceinline__ uint32_t operator[](uint32_t i) const { return i ? v1 : v0; }
  __device__ __forceinline__ void set(uint32_t i, uint32_t x) {
    if (i) v1 = x; else v0 = x;
  }
  __device__ __forceinline__ void add(uint32_t i, uint32_t x) {
    if (i) v1 += x; else v0 += x;
  }
};

struct Scal {
  uint32_t now, tg, cj, cT, swi, swT, mst, ep, epo, pt, pty, pc;
  uint32_t narr, ndrop, ndisp, nbat;
  uint64_t swait;
  uint32_t tld, prev, nlast, tlast;
  float lmw, rate;
  Pair na, nd;
  uint32_t status, events;
  uint32_t ep_cached;
  float ep_factor;
};

// Per-environment queue state: SINGLE mode keeps it replicated in every lane;
// ROUTE mode keeps server gl's in lane gl.
struct Srv {
  uint32_t busy, bsize;
  Pair qh, qc;
};

__device__ __forceinline__ uint32_t add_time(uint32_t a, uint64_t b, uint32_t& status) {
  const uint64_t s = (uint64_t)a + b;
  if (s >= kTimeLimit) {
    status |= kStTime;
    return kTimeLimit;
  }
  return (uint32_t)s;
}

__device__ __forceinline__ uint32_t req_cost(const simx_config& c, uint32_t w3) {
  const float E = expo1(w3);
  if (c.cost_kind == 0) return duration_us(__fmul_rn(c.cost_scale_us, det_exp(__fmul_rn(c.pareto_inv_alpha, E))));
  return duration_us(__fmul_rn(c.cost_scale_us, E));
}

__device__ __forceinline__ uint32_t req_type(const simx_config& c, uint32_t w1) {
  return (c.n_types > 1 && (w1 >> 8) >= c.type0_thr) ? 1u : 0u;
}

// Type and cost of candidate j with Philox words w1, w3: under trace replay (TR) the
// trace's when it has them, else drawn.  TR is a template parameter of the kernels
// because the trace lookups, even untaken, slowed the candidate loop of generated-
// arrival workloads by up to a sixth.
template <bool TR>
__device__ __forceinline__ uint32_t cand_type(const RolloutArgs& A, uint32_t j, uint32_t w1) {
  if (TR && A.tr_type) {
    const uint32_t t = A.tr_type[j % A.tr_n];
    return t < A.cfg.n_types ? t : A.cfg.n_types - 1u;
  }
  return req_type(A.cfg, w1);
}

template <bool TR>
__device__ __forceinline__ uint32_t cand_cost(const RolloutArgs& A, uint32_t j, uint32_t w3) {
  if (TR && A.tr_cost) return A.tr_cost[j % A.tr_n];
  return req_cost(A.cfg, w3);
}

// Batch time of `n` requests of `type` on server k: alpha + beta n (or alpha + the sum
// of the requests' costs for the cost type), times the server's speed s/16, rounded to
// the nearest microsecond in integers.
__device__ __forceinline__ uint64_t service_us(const simx_config& c, uint32_t k, uint32_t type,
                                               uint32_t n, uint64_t csum) {
  const uint64_t L = ((int32_t)type == c.cost_type)
                         ? (uint64_t)c.alpha_us[type] + csum
                         : (uint64_t)c.alpha_us[type] + (uint64_t)c.beta_us[type] * n;
  const uint64_t s = c.srv_speed16[k] ? c.srv_speed16[k] : 16u;
  return (L * s + 8u) >> 4;
}

// Action a -> (major, batch size) (Sec. 4.1): layout 0, major a / n_bsizes and batch
// bsizes[a % n_bsizes]; layout 1, a = 0 is Wait (batch 0) and a >= 1 is major
// (a - 1) / n_bsizes with batch ((a - 1) % n_bsizes) + 1.
__device__ __forceinline__ void decode_action(const simx_config& c, uint32_t a, uint32_t& major,
                                              uint32_t& b) {
  if (c.action_layout == 1) {
    major = a == 0u ? 0u : (a - 1u) / c.n_bsizes;
    b = a == 0u ? 0u : (a - 1u) % c.n_bsizes + 1u;
  } else {
    major = a / c.n_bsizes;
    b = c.bsizes[a % c.n_bsizes];
  }
}

// Initial per-server batch size: the static one.
__device__ __forceinline__ uint32_t static_bsize(const simx_config& c) {
  return c.action_layout == 1 ? c.static_bi + 1u : c.bsizes[c.static_bi];
}

// Time of the modulating chain's switch number i, given switch i-1 at t: an exponential
// dwell drawn from the SWITCH stream, or the fixed dwell of a square wave.
__device__ __forceinline__ uint32_t switch_time(const RolloutArgs& A, uint32_t env, uint32_t i,
                                                uint32_t t, uint32_t& status) {
  if (A.cfg.dwell_kind == 1) return add_time(t, duration_us(A.cfg.dwell_mean_us), status);
  const U4 w = philox(i, env, kStreamSwitch, 0u, A.key0, A.key1);
  return add_time(t, duration_us(__fmul_rn(A.cfg.dwell_mean_us, expo1(w.x))), status);
}

// G consecutive candidates from (cand_j, cand_T): lane gl holds candidate cj + gl with
// its Philox block; times are the prefix sums of integer gaps (exact in any order).  The
// gap is drawn, or read from entry j mod n of a replayed trace.
template <int G, bool TR>
__device__ __forceinline__ void gen_chunk(const RolloutArgs& A, const Grp<G>& g, uint32_t env,
                                          const Scal& s, uint32_t& T, bool& over, U4& w) {
  const uint32_t j = s.cj + g.gl;
  w = philox(j, env, kStreamArrival, 0u, A.key0, A.key1);
  const uint32_t gap = TR ? A.tr_gap[j % A.tr_n]
                          : duration_us(__fmul_rn(A.cfg.cand_mean_gap_us, expo1(w.x)));
  const uint64_t t64 = (uint64_t)s.cT + g.scan_incl(gap);
  over = t64 >= kTimeLimit;
  T = over ? kTimeLimit : (uint32_t)t64;
}

// SINGLE mode: consume every candidate with time <= target; accepted ones join
// their type's FIFO (or are dropped when it is full); switches <= target apply.
template <int G, bool TR>
__device__ void advance_single(const RolloutArgs& A, const Grp<G>& g, uint32_t env, Scal& s,
                               Srv& q, uint32_t* ringb, uint32_t* costb, uint32_t target) {
  const simx_config& c = A.cfg;
  const uint32_t cap = c.queue_cap;
  for (;;) {
    uint32_t T;
    bool over;
    U4 w;
    gen_chunk<G, TR>(A, g, env, s, T, over, w);
    const bool cons = T <= target;
    const int m = __popc(g.ballot(cons));
    const int peek = m < G ? m : G - 1;
    if (g.ballot(over && (int)g.gl <= peek)) s.status |= kStTime;
    if (m == 0) break;
    const uint32_t Tlast = g.shfl(T, m - 1);
    uint32_t st = s.mst;
    if (c.n_mod_states == 2) {
      while (s.swT <= Tlast) {
        if (T >= s.swT) st ^= 1u;
        s.mst ^= 1u;
        s.swi += 1u;
        s.swT = switch_time(A, env, s.swi, s.swT, s.status);
        if (++s.events > kEventCap) {
          s.status |= kStEvent;
          return;
        }
      }
    }
    const bool acc = cons && ((w.z >> 8) < c.accept_thr[st]);
    const uint32_t type = cand_type<TR>(A, s.cj + g.gl, w.y);
    const uint32_t cst = (acc && (int32_t)type == c.cost_type) ? cand_cost<TR>(A, s.cj + g.gl, w.w) : 0u;
    for (uint32_t t = 0; t < c.n_types; ++t) {
      const bool mine = acc && type == t;
      const uint32_t bt = g.ballot(mine);
      const uint32_t cnt = __popc(bt);
      if (cnt == 0) continue;
      const uint32_t room = cap - q.qc[t];
      if (mine) {
        const uint32_t rank = __popc(bt & ((1u << g.gl) - 1u));
        if (rank < room) {
          const uint32_t slot = (q.qh[t] + q.qc[t] + rank) & (cap - 1u);
          ringb[t * cap + slot] = T;
          if ((int32_t)t == c.cost_type) costb[slot] = cst;
        }
      }
      const uint32_t adm = cnt < room ? cnt : room;
      q.qc.add(t, adm);
      s.na.add(t, cnt);
      s.nd.add(t, cnt - adm);
      s.narr += cnt;
      s.ndrop += cnt - adm;
    }
    s.cj += (uint32_t)m;
    s.cT = Tlast;
    s.events += (uint32_t)m;
    if (s.events > kEventCap) {
      s.status |= kStEvent;
      return;
    }
    if (m < G) break;
  }
  if (c.n_mod_states == 2) {
    while (s.swT <= target) {
      s.mst ^= 1u;
      s.swi += 1u;
      s.swT = switch_time(A, env, s.swi, s.swT, s.status);
      if (++s.events > kEventCap) {
        s.status |= kStEvent;
        return;
      }
    }
  }
}

// Walk the modulating chain over a chunk without committing: per-lane state at
// each candidate time, the chain's state after switches <= Tmax and their count.
template <int G>
__device__ __forceinline__ void tentative_states(const RolloutArgs& A, uint32_t env, const Scal& s,
                                                 uint32_t T, uint32_t Tmax, uint32_t& st,
                                                 uint32_t& ms, uint32_t& si, uint32_t& sT,
                                                 uint32_t& tflag, uint32_t& nsw) {
  st = s.mst;
  ms = s.mst;
  si = s.swi;
  sT = s.swT;
  tflag = 0;
  nsw = 0;
  if (A.cfg.n_mod_states != 2) return;
  while (sT <= Tmax && nsw <= kEventCap) {
    if (T >= sT) st ^= 1u;
    ms ^= 1u;
    si += 1u;
    sT = switch_time(A, env, si, sT, tflag);
    nsw += 1u;
  }
}

// SINGLE mode: advance to the next accepted arrival and take in all candidates up
// to its time (the next decision point when nothing is queued).
template <int G, bool TR>
__device__ void jump_single(const RolloutArgs& A, const Grp<G>& g, uint32_t env, Scal& s,
                            Srv& q, uint32_t* ringb, uint32_t* costb) {
  const simx_config& c = A.cfg;
  for (;;) {
    uint32_t T;
    bool over;
    U4 w;
    gen_chunk<G, TR>(A, g, env, s, T, over, w);
    const uint32_t Tmax = g.shfl(T, G - 1);
    uint32_t st, ms, si, sT, tflag, nsw;
    tentative_states<G>(A, env, s, T, Tmax, st, ms, si, sT, tflag, nsw);
    const bool acc = (w.z >> 8) < c.accept_thr[st];
    const uint32_t bm = g.ballot(acc);
    if (bm) {
      const uint32_t Tf = g.shfl(T, __ffs(bm) - 1);
      advance_single<G, TR>(A, g, env, s, q, ringb, costb, Tf);
      s.now = Tf;
      return;
    }
    if (g.ballot(over)) s.status |= kStTime;
    s.status |= tflag;
    s.mst = ms;
    s.swi = si;
    s.swT = sT;
    s.cj += G;
    s.cT = Tmax;
    s.events += G + nsw;
    if (s.events > kEventCap) {
      s.status |= kStEvent;
      return;
    }
  }
}

// ROUTE mode: draw the next request arrival into the pending slot.
template <int G, bool TR>
__device__ void next_arrival(const RolloutArgs& A, const Grp<G>& g, uint32_t env, Scal& s) {
  const simx_config& c = A.cfg;
  if (TR || c.arrival_kind != SIMX_ARR_DIURNAL) {  // THINNED or TRACE
    for (;;) {
      uint32_t T;
      bool over;
      U4 w;
      gen_chunk<G, TR>(A, g, env, s, T, over, w);
      const uint32_t Tmax = g.shfl(T, G - 1);
      uint32_t st, ms, si, sT, tflag, nsw;
      tentative_states<G>(A, env, s, T, Tmax, st, ms, si, sT, tflag, nsw);
      const bool acc = (w.z >> 8) < c.accept_thr[st];
      const uint32_t bm = g.ballot(acc);
      if (bm) {
        const int f = __ffs(bm) - 1;
        const uint32_t Tf = g.shfl(T, f);
        const uint32_t wy = g.shfl(w.y, f), ww = g.shfl(w.w, f);
        if (g.ballot(over && (int)g.gl <= f)) s.status |= kStTime;
        if (c.n_mod_states == 2) {
          while (s.swT <= Tf) {
            s.mst ^= 1u;
            s.swi += 1u;
            s.swT = switch_time(A, env, s.swi, s.swT, s.status);
            if (++s.events > kEventCap) {
              s.status |= kStEvent;
              return;
            }
          }
        }
        const uint32_t jf = s.cj + (uint32_t)f;
        s.cj += (uint32_t)f + 1u;
        s.cT = Tf;
        s.events += (uint32_t)f + 1u;
        s.pt = Tf;
        s.pty = cand_type<TR>(A, jf, wy);
        s.pc = ((int32_t)s.pty == c.cost_type) ? cand_cost<TR>(A, jf, ww) : 0u;
        s.narr += 1u;
        if (s.events > kEventCap) s.status |= kStEvent;
        return;
      }
      if (g.ballot(over)) s.status |= kStTime;
      s.status |= tflag;
      s.mst = ms;
      s.swi = si;
      s.swT = sT;
      s.cj += G;
      s.cT = Tmax;
      s.events += G + nsw;
      if (s.events > kEventCap) {
        s.status |= kStEvent;
        return;
      }
    }
  } else {
    // DIURNAL: constant rate inside a 500 ms epoch; a gap crossing the epoch end is
    // discarded and redrawn from the epoch end at the next epoch's rate.  Every lane
    // of the group computes the same values.
    for (;;) {
      if (++s.events > kEventCap) {
        s.status |= kStEvent;
        return;
      }
      if (s.ep_cached != s.ep) {
        const U4 we = philox(s.ep, env, kStreamEpoch, 0u, A.key0, A.key1);
        s.ep_factor = det_exp(__fmul_rn(c.burst_sigma, normal01(we.x, we.y)));
        s.ep_cached = s.ep;
      }
      const float rate = __fmul_rn(c.diurnal_rate[(s.ep + s.epo) % c.diurnal_len], s.ep_factor);
      const float mean = __fdiv_rn(1.0e6f, rate);
      const U4 w = philox(s.cj, env, kStreamArrival, 0u, A.key0, A.key1);
      const uint32_t gap = duration_us(__fmul_rn(mean, expo1(w.x)));
      s.cj += 1u;
      const uint64_t end = (uint64_t)(s.ep + 1u) * (uint64_t)c.epoch_us;
      if ((uint64_t)s.cT + gap < end) {
        s.cT = add_time(s.cT, gap, s.status);
        s.pt = s.cT;
        s.pty = req_type(c, w.y);
        s.pc = ((int32_t)s.pty == c.cost_type) ? req_cost(c, w.w) : 0u;
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
}

// ROUTE mode, executed by the lane that owns the server: start a batch at time
// st from the queue whose head arrived first (tie: type 0).
__device__ __forceinline__ void try_start(const simx_config& c, uint32_t srv, uint32_t* ringS,
                                          uint32_t* costS, Srv& L, uint32_t st, uint32_t& stn,
                                          uint64_t& w0, uint64_t& w1, uint32_t& nbat,
                                          uint32_t& status) {
  const uint32_t cap = c.queue_cap;
  uint32_t h;
  if (L.qc[0] > 0 && L.qc[1] > 0) {
    const uint32_t h0 = ringS[L.qh[0]], h1 = ringS[cap + L.qh[1]];
    h = (h1 < h0) ? 1u : 0u;
  } else if (L.qc[0] > 0) {
    h = 0;
  } else if (L.qc[1] > 0) {
    h = 1;
  } else {
    return;
  }
  const uint32_t n = L.bsize < L.qc[h] ? L.bsize : L.qc[h];
  const bool costed = (int32_t)h == c.cost_type;
  uint64_t W = 0, csum = 0;
  for (uint32_t i = 0; i < n; ++i) {
    const uint32_t slot = (L.qh[h] + i) & (cap - 1u);
    W += (uint64_t)(st - ringS[h * cap + slot]);
    if (costed) csum += costS[slot];
  }
  L.qh.set(h, (L.qh[h] + n) & (cap - 1u));
  L.qc.set(h, L.qc[h] - n);
  L.busy = add_time(st, service_us(c, srv, h, n, csum), status);
  stn += n;
  if (h) w1 += W; else w0 += W;
  nbat += 1u;
}

__device__ __forceinline__ float fdiv_u(uint32_t a, float b) {
  return __fdiv_rn(__uint2float_rn(a), b);
}

// Observation (Sec. 4.1 state), written to o[0..D).
// SINGLE: every feature is (num * mul) / den with mul = 1 except for the rate
// features, so one lane per feature evaluates it without branches; multiplying by
// 1.0f is exact, so each value has the bits of the plain formula.  Layout for T types:
// [q_t / cap]_T, (now - t_last) / T_w, head-type one-hot (2), server busy (0),
// arrivals * rate_scale / dt, n_last / 32, [head-of-line wait_t / T_w]_T, and with
// obs_extra: type-0 and type-1 arrival rates, last batch type one-hot (2),
// drops / 32, last batch mean wait / T_w.
// ROUTE: lane k writes server k's three features, lane 0 the rest.
template <int G>
__device__ void observe_single(const simx_config& c, const Grp<G>& g, const Scal& s,
                               const Srv& q, const uint32_t* ringb, float* o, int B) {
  const int T = (int)c.n_types;
  const uint32_t cap = c.queue_cap;
  const bool ne0 = q.qc[0] > 0u, ne1 = T > 1 && q.qc[1] > 0u;
  const uint32_t h0 = ne0 ? ringb[q.qh[0]] : 0u;
  const uint32_t h1 = ne1 ? ringb[cap + q.qh[1]] : 0u;
  const uint32_t head = ne0 ? ((ne1 && h1 < h0) ? 1u : 0u) : (ne1 ? 1u : kNone);
  uint32_t dt = s.now - s.prev;
  if (dt < 1u) dt = 1u;
  const float fdt = __uint2float_rn(dt), fcap = __uint2float_rn(cap), tw = c.t_window_us;
  const float rs = c.rate_scale;
  const int D = 2 * T + 6 + (c.obs_extra ? 6 : 0);
  for (int d = (int)g.gl; d < D; d += G) {
    float num = 0.0f, mul = 1.0f, den = 1.0f;
    const int r = d - T;  // position after the queue lengths
    if (d < T) {
      num = __uint2float_rn(d ? q.qc[1] : q.qc[0]);
      den = fcap;
    } else if (r == 0) {
      num = __uint2float_rn(s.now - s.tld);
      den = tw;
    } else if (r == 1 || r == 2) {
      num = head == (uint32_t)(r - 1) ? 1.0f : 0.0f;
    } else if (r == 3) {
      num = 0.0f;  // server status: always free at a SINGLE-mode decision
    } else if (r == 4) {
      num = __uint2float_rn(s.na[0] + s.na[1]);
      mul = rs;
      den = fdt;
    } else if (r == 5) {
      num = __uint2float_rn(s.nlast);
      den = 32.0f;
    } else if (r < 6 + T) {
      const bool one = (r - 6) != 0;
      const bool ne = one ? ne1 : ne0;
      num = ne ? __uint2float_rn(s.now - (one ? h1 : h0)) : 0.0f;
      den = tw;
    } else {
      const int x = r - 6 - T;
      if (x == 0 || x == 1) {
        num = __uint2float_rn(x ? s.na[1] : s.na[0]);
        mul = rs;
        den = fdt;
      } else if (x == 2 || x == 3) {
        num = s.tlast == (uint32_t)(x - 2) ? 1.0f : 0.0f;
      } else if (x == 4) {
        num = __uint2float_rn(s.nd[0] + s.nd[1]);
        den = 32.0f;
      } else {
        num = s.lmw;
        den = tw;
      }
    }
    o[d * B] = __fdiv_rn(__fmul_rn(num, mul), den);
  }
  g.sync();
}

template <int G>
__device__ void observe_route(const simx_config& c, const Grp<G>& g, const Scal& s,
                              const Srv& L, float* o, int B) {
  const uint32_t K = c.n_servers;
  if (g.gl < K) {
    const float fcap = __uint2float_rn(c.queue_cap);
    o[(3 * g.gl + 0) * B] = fdiv_u(L.qc[0], fcap);
    o[(3 * g.gl + 1) * B] = fdiv_u(c.n_types > 1 ? L.qc[1] : 0u, fcap);
    const uint32_t rem = L.busy > s.now ? L.busy - s.now : 0u;
    o[(3 * g.gl + 2) * B] = fdiv_u(rem, c.busy_norm_us);
  }
  if (g.gl == 0) {
    o[(3 * K) * B] = __fdiv_rn(s.rate, c.rate_ref);
    if (c.obs_extra) {
      o[(3 * K + 1) * B] = (s.pty == 0) ? 1.0f : 0.0f;
      o[(3 * K + 2) * B] = (s.pty == 1) ? 1.0f : 0.0f;
      const uint32_t ph = (s.now + s.epo * c.epoch_us) % c.phase_period_us;
      o[(3 * K + 3) * B] = __fdiv_rn(__uint2float_rn(ph), __uint2float_rn(c.phase_period_us));
    }
  }
  g.sync();
}

__device__ __forceinline__ void load_scal(const DevState& st, uint32_t e, Scal& s) {
  const uint32_t E = st.E;
  const uint32_t* h = st.hdr;
  s.now = h[F_NOW * E + e];
  s.tg = h[F_TG * E + e];
  s.cj = h[F_CJ * E + e];
  s.cT = h[F_CT * E + e];
  s.swi = h[F_SWI * E + e];
  s.swT = h[F_SWT * E + e];
  s.mst = h[F_MST * E + e];
  s.ep = h[F_EP * E + e];
  s.epo = h[F_EPO * E + e];
  s.pt = h[F_PT * E + e];
  s.pty = h[F_PTY * E + e];
  s.pc = h[F_PC * E + e];
  s.narr = h[F_NARR * E + e];
  s.ndrop = h[F_NDROP * E + e];
  s.ndisp = h[F_NDISP * E + e];
  s.nbat = h[F_NBAT * E + e];
  s.swait = (uint64_t)h[F_SWLO * E + e] | ((uint64_t)h[F_SWHI * E + e] << 32);
  s.tld = h[F_TLD * E + e];
  s.prev = h[F_PREV * E + e];
  s.nlast = h[F_NLAST * E + e];
  s.tlast = h[F_TLAST * E + e];
  s.lmw = __uint_as_float(h[F_LMW * E + e]);
  s.rate = __uint_as_float(h[F_RATE * E + e]);
  s.na = Pair{h[F_NA0 * E + e], h[F_NA1 * E + e]};
  s.nd = Pair{h[F_ND0 * E + e], h[F_ND1 * E + e]};
  s.status = h[F_STATUS * E + e];
  s.events = 0;
  s.ep_cached = kNone;
  s.ep_factor = 0.0f;
}

__device__ __forceinline__ void store_scal(const DevState& st, uint32_t e, const Scal& s) {
  const uint32_t E = st.E;
  uint32_t* h = st.hdr;
  h[F_NOW * E + e] = s.now;
  h[F_TG * E + e] = s.tg;
  h[F_CJ * E + e] = s.cj;
  h[F_CT * E + e] = s.cT;
  h[F_SWI * E + e] = s.swi;
  h[F_SWT * E + e] = s.swT;
  h[F_MST * E + e] = s.mst;
  h[F_EP * E + e] = s.ep;
  h[F_EPO * E + e] = s.epo;
  h[F_PT * E + e] = s.pt;
  h[F_PTY * E + e] = s.pty;
  h[F_PC * E + e] = s.pc;
  h[F_NARR * E + e] = s.narr;
  h[F_NDROP * E + e] = s.ndrop;
  h[F_NDISP * E + e] = s.ndisp;
  h[F_NBAT * E + e] = s.nbat;
  h[F_SWLO * E + e] = (uint32_t)s.swait;
  h[F_SWHI * E + e] = (uint32_t)(s.swait >> 32);
  h[F_TLD * E + e] = s.tld;
  h[F_PREV * E + e] = s.prev;
  h[F_NLAST * E + e] = s.nlast;
  h[F_TLAST * E + e] = s.tlast;
  h[F_LMW * E + e] = __float_as_uint(s.lmw);
  h[F_RATE * E + e] = __float_as_uint(s.rate);
  h[F_NA0 * E + e] = s.na[0];
  h[F_NA1 * E + e] = s.na[1];
  h[F_ND0 * E + e] = s.nd[0];
  h[F_ND1 * E + e] = s.nd[1];
  h[F_STATUS * E + e] = s.status;
}

__device__ __forceinline__ void load_srv(const DevState& st, uint32_t e, uint32_t k, Srv& L) {
  const uint32_t E = st.E, K = st.K, T = st.T;
  L.busy = st.srv[(0 * K + k) * E + e];
  L.bsize = st.srv[(1 * K + k) * E + e];
  for (uint32_t t = 0; t < 2; ++t) {
    L.qh.set(t, t < T ? st.qh[(k * T + t) * E + e] : 0u);
    L.qc.set(t, t < T ? st.qc[(k * T + t) * E + e] : 0u);
  }
}

__device__ __forceinline__ void store_srv(const DevState& st, uint32_t e, uint32_t k, const Srv& L) {
  const uint32_t E = st.E, K = st.K, T = st.T;
  st.srv[(0 * K + k) * E + e] = L.busy;
  st.srv[(1 * K + k) * E + e] = L.bsize;
  for (uint32_t t = 0; t < T; ++t) {
    st.qh[(k * T + t) * E + e] = L.qh[t];
    st.qc[(k * T + t) * E + e] = L.qc[t];
  }
}

// Action of a baseline (Sec. 5.1) or an external caller; the policy case is
// handled by the block-wide MLP in the kernel.
template <int G, bool ROUTE>
__device__ int baseline_action(const RolloutArgs& A, const Grp<G>& g, uint32_t env, Scal& s,
                               const Srv& L, const uint32_t* ringb) {
  const simx_config& c = A.cfg;
  const int mode = A.policy_mode;
  if (mode == SIMX_POLICY_EXTERNAL) {
    const int32_t a = A.ext[env];
    if (a < 0 || (uint32_t)a >= A.n_actions) {
      s.status |= kStAction;
      return 0;
    }
    return a;
  }
  if (mode == SIMX_POLICY_RANDOM) {
    const U4 w = philox(s.tg, env, kStreamPolicy, 0u, A.key0, A.key1);
    return (int)(((uint64_t)(w.y >> 8) * A.n_actions) >> 24);
  }
  if (!ROUTE) {  // STATIC: the type whose head arrived first, batch bsizes[static_bi]
    uint32_t h = 0;
    if (L.qc[0] > 0 && c.n_types > 1 && L.qc[1] > 0) {
      h = ringb[c.queue_cap + L.qh[1]] < ringb[L.qh[0]] ? 1u : 0u;
    } else if (L.qc[0] == 0 && c.n_types > 1 && L.qc[1] > 0) {
      h = 1u;
    }
    return (int)((c.action_layout == 1 ? 1u : 0u) + h * c.n_bsizes + c.static_bi);
  }
  if (mode == SIMX_POLICY_RR) return (int)((s.tg % c.n_servers) * c.n_bsizes + c.static_bi);
  // SQ: server with the fewest queued requests (first such)
  uint32_t q = g.gl < c.n_servers ? (L.qc[0] + L.qc[1]) : 0xFFFFFFFFu;
  uint32_t key = (q << 4) | g.gl;  // q <= 2 * 4096 fits in 28 bits
  if (g.gl >= c.n_servers) key = 0xFFFFFFFFu;
#pragma unroll
  for (int d = G / 2; d > 0; d >>= 1) key = min(key, __shfl_xor_sync(g.mask, key, d, G));
  return (int)((key & 15u) * c.n_bsizes + c.static_bi);
}

template <int G>
__device__ __forceinline__ void write_obs(const Grp<G>& g, const float* o, int B, int D, float* dst,
                                          int64_t ld, uint32_t e) {
  if (!dst) return;
  for (int d = (int)g.gl; d < D; d += G) dst[(int64_t)d * ld + e] = o[d * B];
}

// ---------------------------------------------------------------------------------
// The grid policy's forward on the tensor cores (the exact policy forward).  On the
// grid every input, weight and hidden output is an integer multiple of its grid unit
// with a mantissa of at most 255, so each is exact in bf16, every product is exact in
// fp32, and every partial sum of a pre-activation stays below 2^24 product units: the
// tensor core's FP32 accumulation gives the exact dot product, the bits the FP32 FMA
// chains give.  Per layer: the block's envs are the N columns of one tcgen05.mma chain
// per tile of 128 outputs (kind::f16, bf16 operands, K = 16 per instruction), the
// weights the A operand resident in shared memory for the launch; threads then read the
// accumulator (lane = output, column = env), add the bias in FP32, apply the activation
// and the grid rounding, and write the next layer's operand, or the logits and value
// into the activation buffer the sampler reads.
// ---------------------------------------------------------------------------------
namespace tcf {

using namespace tcx;

constexpr long long kWaitCycles = 2000000000LL;  // bound on the MMA wait (about 1 s)

// Byte offset of (row i, k) in a K-major bf16 operand whose rows hold Kp values: core
// matrices of 8 rows x 8 values (16 bytes), K-adjacent ones 128 bytes apart.
__device__ __forceinline__ uint32_t boff(int i, int k, int Kp) {
  return (uint32_t)(((i >> 3) * (Kp >> 3) + (k >> 3)) * 128 + (i & 7) * 16 + (k & 7) * 2);
}

// bf16 bits of a value exact in bf16 (on the grid), which is its fp32 bits' upper half.
__device__ __forceinline__ uint16_t bf16_bits(float v) { return (uint16_t)(__float_as_uint(v) >> 16); }

// Once per launch: the weights of every layer into shared memory as bf16 A tiles (zero
// padded), the mbarrier, and (warp 0) the tensor memory of the block.
__device__ void setup(const RolloutArgs& A, unsigned char* sm, uint32_t* tbase) {
  const DevMlp& m = A.mlp;
  const TcPlan& P = A.tc;
  for (int l = 0; l < m.n_layers; ++l) {
    const int K = m.dims[l], N = m.dims[l + 1], Kp = P.Kp[l], Np = m.npad[l + 1];
    const int rows = 128 * P.nmt[l];
    uint16_t* w = reinterpret_cast<uint16_t*>(sm + P.w_off[l]);
    for (int i = threadIdx.x; i < rows * Kp; i += blockDim.x) {
      const int j = i / Kp, k = i % Kp;
      const float v = (j < N && k < K) ? m.Wt[l][(size_t)k * Np + j] : 0.0f;
      w[boff(j, k, Kp) / 2] = bf16_bits(v);
    }
  }
  uint64_t* bar = reinterpret_cast<uint64_t*>(sm + P.bar_off);
  if (threadIdx.x == 0) {
    mbar_init(bar, 1);
    mbar_fence_init();
  }
  if (threadIdx.x < 32) tm_alloc(tbase, (uint32_t)P.tcols);
  fence_async_smem();
  fence_before();
  __syncthreads();
  fence_after();
}

__device__ void teardown(const RolloutArgs& A, uint32_t tmem) {
  fence_before();
  __syncthreads();
  if (threadIdx.x < 32) {
    fence_after();
    tm_dealloc(tmem, (uint32_t)A.tc.tcols);
  }
}

// Returns the buffer holding the last layer (X1: logits rows 0..A-1, value row A) with
// row stride ld, or sets *timed_out when an MMA wait ran out (the result is then void).
__device__ float* forward(const RolloutArgs& A, unsigned char* sm, uint32_t tmem, float* X0,
                          float* X1, int B, int ld, uint32_t& phase, bool& timed_out) {
  const DevMlp& m = A.mlp;
  const TcPlan& P = A.tc;
  const int tid = threadIdx.x, nthr = blockDim.x, warp = tid >> 5, lane = tid & 31;
  const int Bn = P.Bn, L = m.n_layers;
  uint64_t* bar = reinterpret_cast<uint64_t*>(sm + P.bar_off);
  // the observation on its grid as the first B operand (padding columns and rows zero)
  __syncthreads();
  {
    const int D = m.dims[0], Kp = P.Kp[0];
    uint16_t* xb = reinterpret_cast<uint16_t*>(sm + P.x_off[0]);
    for (int i = tid; i < Bn * Kp; i += nthr) {
      const int e = i % Bn, k = i / Bn;
      const float v = (e < B && k < D) ? grid_q(X0[k * ld + e], m.gx[0]) : 0.0f;
      xb[boff(e, k, Kp) / 2] = bf16_bits(v);
    }
  }
  const int quarter = warp & 3, part = warp >> 2, nsplit = nthr >> 7;   // warps per lane quarter
  for (int l = 0; l < L; ++l) {
    const int Kp = P.Kp[l], N = m.dims[l + 1];
    const bool last = l + 1 == L;
    fence_async_smem();
    fence_before();
    __syncthreads();
    fence_after();
    if (tid == 0) {
      const uint32_t id = idesc_bf16(128, Bn);
      const uint32_t xa = su32(sm + P.x_off[l & 1]);
      const uint32_t sbo = (uint32_t)(Kp >> 3) * 128u;
      for (int mt = 0; mt < P.nmt[l]; ++mt) {
        const uint32_t wa = su32(sm + P.w_off[l]) + (uint32_t)mt * 128u * (uint32_t)Kp * 2u;
        for (int ks = 0; ks < Kp / 16; ++ks)
          mma_bf16(tmem + (uint32_t)(mt * Bn), sdesc(wa + (uint32_t)ks * 256u, 128, sbo),
                   sdesc(xa + (uint32_t)ks * 256u, 128, sbo), id, ks > 0 ? 1u : 0u);
      }
      commit(bar);
    }
    if (!mbar_wait(bar, phase, kWaitCycles)) timed_out = true;
    phase ^= 1u;
    __syncwarp();
    fence_after();
    // epilogue: lane = output j of tile mt, 16 env columns per warp
    const int Kn = last ? 0 : P.Kp[l + 1];
    const int gq = last ? -1 : m.gx[l + 1];
    const int act = last ? -1 : m.act[l];
    const float* bias = m.bias[l];
    uint16_t* xn = reinterpret_cast<uint16_t*>(sm + P.x_off[(l + 1) & 1]);
    for (int mt = 0; mt < P.nmt[l]; ++mt) {
      const int j = 128 * mt + 32 * quarter + lane;
      for (int c0 = 16 * part; c0 < Bn; c0 += 16 * nsplit) {
        uint32_t u[16];
        tm_ld16_nw(tmem + ((uint32_t)(32 * quarter) << 16) + (uint32_t)(mt * Bn + c0), u);
        tm_wait();
        reg_fence16(u);
        const float bj = j < N ? bias[j] : 0.0f;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int e = c0 + i;
          const float z = __fadd_rn(__uint_as_float(u[i]), bj);
          if (last) {
            if (j < N && e < B) X1[j * ld + e] = z;
          } else if (j < Kn) {
            float y = 0.0f;
            if (j < N && e < B) {
              y = z;
              if (act == 0) y = det_tanh(y);
              else if (act == 2) y = det_gelu(y);
              y = grid_q(y, gq);
            }
            xn[boff(e, j, Kn) / 2] = bf16_bits(y);
          }
        }
      }
    }
  }
  __syncthreads();
  return X1;
}

}  // namespace tcf

// The rollout / step kernel.  A block of blockDim.x threads owns B = blockDim.x / G
// envs, one per G-lane group.  Shared memory: two activation buffers X0, X1 of
// maxd4 x B floats (feature-major) and a softmax scratch of apad floats per env.
// Every lane stays alive to the end (groups past the last env do no work) so that
// warps reconverge at each phase and the block can run the MLP together.
template <bool ROUTE, int G, bool TR, bool WARP, bool GRID>
__global__ void __launch_bounds__(kMaxThreads, min_blocks<G>())
k_rollout(const __grid_constant__ RolloutArgs A) {
  extern __shared__ float smem[];
  const Grp<G> g;
  const int B = (int)blockDim.x / G;
  const int Bs = B + A.bs_pad;  // row stride of the activation buffers
  const uint32_t slot = threadIdx.x / G;
  const uint32_t env_raw = blockIdx.x * (uint32_t)B + slot;
  const bool live = env_raw < A.st.E;
  const uint32_t env = live ? env_raw : 0u;
  float* X0 = smem;
  float* X1 = smem + (size_t)A.maxd4 * Bs;
  float* scratch = smem + (size_t)2 * A.maxd4 * Bs + (size_t)slot * A.apad;
  float* ocol = X0 + slot;
  const simx_config& c = A.cfg;
  const DevState& st = A.st;
  const uint32_t K = c.n_servers, T = c.n_types, cap = c.queue_cap;
  uint32_t* ringb = st.ring + (size_t)env * K * T * cap;
  uint32_t* costb = st.cost ? st.cost + (size_t)env * K * cap : nullptr;
  const bool use_mlp = A.policy_mode == SIMX_POLICY_SAMPLE || A.policy_mode == SIMX_POLICY_ARGMAX;

  Scal s{};
  Srv L{0u, 0u, Pair{0u, 0u}, Pair{0u, 0u}};
  if (live) {
    load_scal(st, env, s);
    if (ROUTE) {
      if (g.gl < K) load_srv(st, env, g.gl, L);
    } else {
      load_srv(st, env, 0, L);
    }
  }
  uint32_t* ringS = ROUTE ? ringb + (size_t)(g.gl < K ? g.gl : 0) * T * cap : ringb;
  uint32_t* costS = (ROUTE && costb) ? costb + (size_t)(g.gl < K ? g.gl : 0) * cap : costb;
  const int D = A.obs_dim;
  // grid policies on the tensor cores: weights, barrier and tensor memory for the launch
  unsigned char* tsm = reinterpret_cast<unsigned char*>(smem);
  uint32_t tc_phase = 0u;
  bool tc_timeout = false;
  const bool tc = GRID && !WARP && A.tc.on && use_mlp;
  uint32_t* tc_tbase = reinterpret_cast<uint32_t*>(tsm + A.tc.bar_off + 8);
  if (tc) tcf::setup(A, tsm, tc_tbase);
  const uint32_t tc_tmem = tc ? *tc_tbase : 0u;
  // fp32 policies with staged weights: the launch's pipeline of weight chunks (not
  // instantiated for 32 lanes per env, whose blocks hold at most 8 envs)
  const bool stg = G != 32 && !WARP && !tc && A.stage.on && use_mlp;
  StagePipe sp;
  sp.stages = reinterpret_cast<float*>(tsm + A.stage.off);
  sp.full = reinterpret_cast<uint64_t*>(tsm + A.stage.bar_off);
  sp.flag = reinterpret_cast<volatile int*>(tsm + A.stage.bar_off + 8u * (uint32_t)A.stage.S);
  sp.cc = 0u;
  sp.total = (uint32_t)A.H * (uint32_t)A.stage.n;
  if (stg && threadIdx.x == 0) stage_start(A.mlp, A.stage, sp);

  for (int t = 0; t < A.H; ++t) {
    // phase 1: observation (Sec. 4.1) into column `slot` of X0
    if (live) {
      if (ROUTE) observe_route<G>(c, g, s, L, ocol, Bs);
      else observe_single<G>(c, g, s, L, ringb, ocol, Bs);
      write_obs<G>(g, ocol, Bs, D, A.obs ? A.obs + (int64_t)t * D * A.ld : nullptr, A.ld, env);
    }
    __syncwarp();
    // phase 2: action from the policy (Sec. 4.2, block-wide MLP) or a baseline
    float logp = 0.0f, value = 0.0f;
    int a = 0;
    if (use_mlp) {
      // WARP: each warp runs the policy for its own 1-2 envs (narrow policies); else
      // block-wide, whose warps share each weight row instead of each loading it.  A
      // template parameter: both forwards in one kernel slowed the narrow case by 16 %.
      const float* Z;
      if (tc) {
        Z = tcf::forward(A, tsm, tc_tmem, X0, X1, B, Bs, tc_phase, tc_timeout);
        if (tc_timeout) s.status |= SIMX_DEV_TC_TIMEOUT;
      } else if (stg) {
        Z = mlp_forward_staged<GRID>(A.mlp, A.stage, sp, X0, X1, B, Bs);
        if (*sp.flag) s.status |= SIMX_DEV_COPY_TIMEOUT;
      } else {
        Z = WARP ? mlp_forward_warp<GRID>(A.mlp, X0, X1, 32 / G, Bs, (int)(threadIdx.x / 32) * (32 / G))
                 : mlp_forward_block<GRID>(A.mlp, X0, X1, B, Bs);
      }
      if (live)
        a = sample_action<G>(A.mlp, Z + slot, Bs, scratch, A.policy_mode, A.key0, A.key1, s.tg,
                             env, logp, value, g);
    } else if (live) {
      a = baseline_action<G, ROUTE>(A, g, env, s, L, ringb);
    }
    __syncwarp();
    uint32_t k, b;
    decode_action(c, (uint32_t)a, k, b);
    const bool frozen = s.status != 0;
    const uint32_t now = ROUTE ? s.pt : s.now;
    uint32_t n_step = 0, qafter = 0;
    uint64_t w_step = 0;
    float reward = 0.0f;
    // phase 3: apply the action; phase 4: advance to the next decision point
    if (!ROUTE) {
      uint32_t n = 0;
      if (live) {
        uint64_t W = 0, csum = 0;
        if (!frozen) {
          n = b < L.qc[k] ? b : L.qc[k];
          uint64_t wp = 0, cp = 0;
          for (uint32_t i = g.gl; i < n; i += G) {
            const uint32_t sl = (L.qh[k] + i) & (cap - 1u);
            wp += (uint64_t)(now - ringb[k * cap + sl]);
            if ((int32_t)k == c.cost_type) cp += costb[sl];
          }
          W = g.sum64(wp);
          csum = g.sum64(cp);
          L.qh.set(k, (L.qh[k] + n) & (cap - 1u));
          L.qc.set(k, L.qc[k] - n);
          if (n > 0) {
            L.busy = add_time(now, service_us(c, 0u, k, n, csum), s.status);
            s.nlast = n;
            s.tlast = k;
            s.tld = now;
            s.lmw = __fdiv_rn(__ull2float_rn(W), __uint2float_rn(n));
            s.nbat += 1u;
          }
          s.ndisp += n;
          s.swait += W;
        }
        reward = __fsub_rn(__uint2float_rn(n), __fmul_rn(c.w_wait[k], __ull2float_rn(W)));
        n_step = n;
        w_step = W;
        qafter = L.qc[0] + (T > 1 ? L.qc[1] : 0u);
        s.prev = now;
        s.na = Pair{0u, 0u};
        s.nd = Pair{0u, 0u};
        s.tg += 1u;
      }
      __syncwarp();
      if (live && !frozen) {
        s.events = 0;
        if (n > 0) {
          const uint32_t next = L.busy;
          advance_single<G, TR>(A, g, env, s, L, ringb, costb, next);
          s.now = next;
          if (L.qc[0] + (T > 1 ? L.qc[1] : 0u) == 0u) jump_single<G, TR>(A, g, env, s, L, ringb, costb);
        } else {
          jump_single<G, TR>(A, g, env, s, L, ringb, costb);
        }
      }
      __syncwarp();
    } else {
      const uint32_t mt = s.pty;
      uint32_t stn = 0, nbat = 0, lstat = 0;
      uint64_t w0 = 0, w1 = 0;
      if (live) {
        if (!frozen) {
          s.events = 0;
          uint32_t dropped = 0;
          if (g.gl == k) {
            if (L.qc[mt] < cap) {
              const uint32_t sl = (L.qh[mt] + L.qc[mt]) & (cap - 1u);
              ringS[mt * cap + sl] = now;
              if ((int32_t)mt == c.cost_type) costS[sl] = s.pc;
              L.qc.add(mt, 1u);
            } else {
              dropped = 1u;
            }
            L.bsize = b;
            if (L.busy <= now) try_start(c, g.gl, ringS, costS, L, now, stn, w0, w1, nbat, lstat);
          }
          dropped = g.shfl(dropped, (int)k);
          s.ndrop += dropped;
          s.nd.add(mt, dropped);
        }
        qafter = g.sum(g.gl < K ? L.qc[0] + L.qc[1] : 0u);
      }
      __syncwarp();
      if (live && !frozen) {
        next_arrival<G, TR>(A, g, env, s);
        uint32_t gap = s.pt - now;
        if (gap < 1u) gap = 1u;
        const float inst = __fdiv_rn(1.0e6f, __uint2float_rn(gap));
        s.rate = __fadd_rn(s.rate, __fmul_rn(0.0625f, __fsub_rn(inst, s.rate)));
        if (g.gl < K)
          while (L.busy <= s.pt && (L.qc[0] + L.qc[1]) > 0u)
            try_start(c, g.gl, ringS, costS, L, L.busy, stn, w0, w1, nbat, lstat);
        s.now = s.pt;
      }
      __syncwarp();
      if (live) {
        stn = g.sum(stn);
        w0 = g.sum64(w0);
        w1 = g.sum64(w1);
        nbat = g.sum(nbat);
        s.status |= g.bor(lstat);
        s.ndisp += stn;
        s.swait += w0 + w1;
        s.nbat += nbat;
        reward = __fsub_rn(__uint2float_rn(stn),
                           __fadd_rn(__fmul_rn(c.w_wait[0], __ull2float_rn(w0)),
                                     __fmul_rn(c.w_wait[1], __ull2float_rn(w1))));
        n_step = stn;
        w_step = w0 + w1;
        s.prev = now;
        s.tg += 1u;
      }
    }
    // phase 5: records of step t
    if (live && g.gl == 0) {
      const int64_t o = (int64_t)t * A.ld + env;
      if (A.action) A.action[o] = (uint8_t)a;
      if (A.logp) A.logp[o] = logp;
      if (A.value) A.value[o] = value;
      if (A.reward) A.reward[o] = reward;
      if (A.done) A.done[o] = (uint8_t)(((s.tg) % c.episode_len) == 0u);
      if (A.trace) {
        int64_t* tr = A.trace + (int64_t)t * SIMX_TRACE_WIDTH * A.ld + env;
        tr[0] = now;
        tr[A.ld] = n_step;
        tr[2 * A.ld] = (int64_t)w_step;
        tr[3 * A.ld] = qafter;
      }
    }
    __syncwarp();
  }
  if (tc) tcf::teardown(A, tc_tmem);
  if (stg && threadIdx.x == 0 && *sp.flag) stage_drain(A.stage, sp);
  if (!live) return;
  if (A.next_obs) {
    if (ROUTE) observe_route<G>(c, g, s, L, ocol, Bs);
    else observe_single<G>(c, g, s, L, ringb, ocol, Bs);
    write_obs<G>(g, ocol, Bs, D, A.next_obs, A.next_ld, env);
  }
  if (g.gl == 0) store_scal(st, env, s);
  if (ROUTE) {
    if (g.gl < K) store_srv(st, env, g.gl, L);
  } else if (g.gl == 0) {
    store_srv(st, env, 0, L);
  }
}

// Reset: empty queues, idle servers, chain state from the INIT stream, then advance
// to the first decision point.
template <bool ROUTE, int G, bool TR>
__global__ void __launch_bounds__(kMaxThreads) k_reset(const __grid_constant__ RolloutArgs A) {
  const Grp<G> g;
  const uint32_t slot = threadIdx.x / G;
  const uint32_t env = blockIdx.x * (blockDim.x / G) + slot;
  if (env >= A.st.E) return;
  const simx_config& c = A.cfg;
  const DevState& st = A.st;
  const uint32_t K = c.n_servers, T = c.n_types, cap = c.queue_cap;
  uint32_t* ringb = st.ring + (size_t)env * K * T * cap;
  uint32_t* costb = st.cost ? st.cost + (size_t)env * K * cap : nullptr;
  for (uint32_t i = g.gl; i < K * T * cap; i += G) ringb[i] = 0u;
  if (costb)
    for (uint32_t i = g.gl; i < K * cap; i += G) costb[i] = 0u;
  Scal s;
  s.now = s.tg = s.cj = s.cT = 0u;
  s.ep = s.epo = s.pt = s.pty = s.pc = 0u;
  s.narr = s.ndrop = s.ndisp = s.nbat = 0u;
  s.swait = 0u;
  s.tld = s.prev = s.nlast = 0u;
  s.tlast = kNone;
  s.lmw = 0.0f;
  s.rate = c.rate_ref;
  s.na = Pair{0u, 0u};
  s.nd = Pair{0u, 0u};
  s.status = 0u;
  s.events = 0u;
  s.ep_cached = kNone;
  s.ep_factor = 0.0f;
  const U4 w = philox(0u, env, kStreamInit, 0u, A.key0, A.key1);
  if (c.n_mod_states == 2) {
    s.mst = w.x >> 31;
    s.swi = 1u;
    s.swT = switch_time(A, env, 1u, 0u, s.status);
  } else {
    s.mst = 0u;
    s.swi = 0u;
    s.swT = kNone;
  }
  if (c.arrival_kind == SIMX_ARR_DIURNAL)
    s.epo = (uint32_t)(((uint64_t)(w.y >> 8) * c.diurnal_len) >> 24);
  if (TR)  // this env's starting entry of the trace
    s.cj = (uint32_t)(((uint64_t)w.z * A.tr_n) >> 32);
  Srv L{0u, static_bsize(c), Pair{0u, 0u}, Pair{0u, 0u}};
  __syncwarp(g.mask);
  if (ROUTE) {
    next_arrival<G, TR>(A, g, env, s);
    s.now = s.pt;
  } else {
    jump_single<G, TR>(A, g, env, s, L, ringb, costb);
  }
  if (g.gl == 0) store_scal(st, env, s);
  if (ROUTE) {
    if (g.gl < K) store_srv(st, env, g.gl, L);
  } else if (g.gl == 0) {
    store_srv(st, env, 0, L);
  }
}

// Current observation of every env (no state change).
template <bool ROUTE, int G>
__global__ void __launch_bounds__(kMaxThreads) k_observe(const __grid_constant__ RolloutArgs A) {
  extern __shared__ float smem[];
  const Grp<G> g;
  const int B = (int)blockDim.x / G;
  const uint32_t slot = threadIdx.x / G;
  const uint32_t env = blockIdx.x * (uint32_t)B + slot;
  if (env >= A.st.E) return;
  float* ocol = smem + slot;
  const simx_config& c = A.cfg;
  const uint32_t K = c.n_servers, T = c.n_types, cap = c.queue_cap;
  const uint32_t* ringb = A.st.ring + (size_t)env * K * T * cap;
  Scal s;
  load_scal(A.st, env, s);
  Srv L{0u, 0u, Pair{0u, 0u}, Pair{0u, 0u}};
  if (ROUTE) {
    if (g.gl < K) load_srv(A.st, env, g.gl, L);
    observe_route<G>(c, g, s, L, ocol, B + A.bs_pad);
  } else {
    load_srv(A.st, env, 0, L);
    observe_single<G>(c, g, s, L, ringb, ocol, B + A.bs_pad);
  }
  write_obs<G>(g, ocol, B + A.bs_pad, A.obs_dim, A.next_obs, A.next_ld, env);
}

// Canonical state image of each env (header, servers, queue lengths, FIFO contents
// from index 0, costs), one thread per env.
__global__ void k_save(DevState st, int32_t cost_type, uint64_t words, uint32_t* out) {
  const uint32_t e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= st.E) return;
  uint32_t* w = out + (uint64_t)e * words;
  const uint32_t E = st.E, K = st.K, T = st.T, cap = st.cap;
  for (int f = 0; f < SIMX_STATE_HEADER_WORDS; ++f) w[f] = f < F_COUNT ? st.hdr[(uint64_t)f * E + e] : 0u;
  uint32_t* p = w + SIMX_STATE_HEADER_WORDS;
  for (uint32_t k = 0; k < K; ++k) {
    *p++ = st.srv[(0 * K + k) * E + e];
    *p++ = st.srv[(1 * K + k) * E + e];
  }
  for (uint32_t k = 0; k < K; ++k)
    for (uint32_t t = 0; t < T; ++t) *p++ = st.qc[(k * T + t) * E + e];
  const uint32_t* ringb = st.ring + (size_t)e * K * T * cap;
  for (uint32_t k = 0; k < K; ++k)
    for (uint32_t t = 0; t < T; ++t) {
      const uint32_t h = st.qh[(k * T + t) * E + e], n = st.qc[(k * T + t) * E + e];
      for (uint32_t i = 0; i < cap; ++i) p[i] = i < n ? ringb[(k * T + t) * cap + ((h + i) & (cap - 1u))] : 0u;
      p += cap;
    }
  if (cost_type >= 0) {
    const uint32_t* costb = st.cost + (size_t)e * K * cap;
    for (uint32_t k = 0; k < K; ++k) {
      const uint32_t h = st.qh[(k * T + cost_type) * E + e], n = st.qc[(k * T + cost_type) * E + e];
      for (uint32_t i = 0; i < cap; ++i) p[i] = i < n ? costb[k * cap + ((h + i) & (cap - 1u))] : 0u;
      p += cap;
    }
  }
}

__global__ void k_load(DevState st, int32_t cost_type, uint64_t words, const uint32_t* in) {
  const uint32_t e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= st.E) return;
  const uint32_t* w = in + (uint64_t)e * words;
  const uint32_t E = st.E, K = st.K, T = st.T, cap = st.cap;
  for (int f = 0; f < F_COUNT; ++f) st.hdr[(uint64_t)f * E + e] = w[f];
  const uint32_t* p = w + SIMX_STATE_HEADER_WORDS;
  for (uint32_t k = 0; k < K; ++k) {
    st.srv[(0 * K + k) * E + e] = *p++;
    st.srv[(1 * K + k) * E + e] = *p++;
  }
  for (uint32_t k = 0; k < K; ++k)
    for (uint32_t t = 0; t < T; ++t) {
      st.qc[(k * T + t) * E + e] = *p++;
      st.qh[(k * T + t) * E + e] = 0u;
    }
  uint32_t* ringb = st.ring + (size_t)e * K * T * cap;
  for (uint32_t i = 0; i < K * T * cap; ++i) ringb[i] = p[i];
  p += K * T * cap;
  if (cost_type >= 0) {
    uint32_t* costb = st.cost + (size_t)e * K * cap;
    for (uint32_t i = 0; i < K * cap; ++i) costb[i] = p[i];
  }
}

// Aggregate counters: out[0..7] (u64) arrived, dropped, dispatched, batches, queued,
// sum_wait, decisions, flagged; out[8] = OR of status words.
__global__ void k_stats(DevState st, unsigned long long* out) {
  const uint32_t e = blockIdx.x * blockDim.x + threadIdx.x;
  unsigned long long v[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  uint32_t sor = 0;
  if (e < st.E) {
    const uint32_t E = st.E;
    v[0] = st.hdr[F_NARR * E + e];
    v[1] = st.hdr[F_NDROP * E + e];
    v[2] = st.hdr[F_NDISP * E + e];
    v[3] = st.hdr[F_NBAT * E + e];
    for (uint32_t i = 0; i < st.K * st.T; ++i) v[4] += st.qc[i * E + e];
    v[5] = (unsigned long long)st.hdr[F_SWLO * E + e] | ((unsigned long long)st.hdr[F_SWHI * E + e] << 32);
    v[6] = st.hdr[F_TG * E + e];
    sor = st.hdr[F_STATUS * E + e];
    v[7] = sor ? 1ull : 0ull;
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    unsigned long long x = v[i];
    for (int d = 16; d > 0; d >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, d);
    if ((threadIdx.x & 31u) == 0 && x) atomicAdd(out + i, x);
  }
  for (int d = 16; d > 0; d >>= 1) sor |= __shfl_xor_sync(0xFFFFFFFFu, sor, d);
  if ((threadIdx.x & 31u) == 0 && sor) atomicOr(reinterpret_cast<unsigned int*>(out + 8), sor);
}

// W [N][K] row-major -> Wt [K][Npad] (zero-padded columns), b [N] -> bias [Npad].
__global__ void k_repack(const float* __restrict__ W, const float* __restrict__ b, int N, int K,
                         int Npad, float* __restrict__ Wt, float* __restrict__ bias) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < K * Npad) {
    const int k = i / Npad, j = i % Npad;
    Wt[i] = j < N ? W[(size_t)j * K + k] : 0.0f;
  }
  if (i < Npad) bias[i] = i < N ? b[i] : 0.0f;
}

// Batched policy forward (Sec. 4.2) over observation columns [D][ld]: a block of
// B = blockDim.x / G columns runs the block-wide MLP, then each column's G lanes
// sample.  Every lane stays alive for the block barriers.
template <int G>
__global__ void __launch_bounds__(kMaxThreads)
k_policy_forward(const __grid_constant__ PolicyArgs P) {
  extern __shared__ float smem[];
  const Grp<G> g;
  const int B = (int)blockDim.x / G;
  const int Bs = B + 4;
  const uint32_t slot = threadIdx.x / G;
  const int64_t i = (int64_t)blockIdx.x * B + slot;
  const bool live = i < P.n;
  float* X0 = smem;
  float* X1 = smem + (size_t)P.maxd4 * Bs;
  float* scratch = smem + (size_t)2 * P.maxd4 * Bs + (size_t)slot * P.apad;
  const int D = P.mlp.dims[0];
  for (int d = (int)g.gl; d < D; d += G) X0[d * Bs + slot] = live ? P.obs[(int64_t)d * P.ld + i] : 0.0f;
  const float* Z = P.mlp.grid ? mlp_forward_block<true>(P.mlp, X0, X1, B, Bs)
                              : mlp_forward_block<false>(P.mlp, X0, X1, B, Bs);
  if (!live) return;
  float logp, value;
  const uint32_t env = P.env_base + (uint32_t)i;
  const int a = sample_action<G>(P.mlp, Z + slot, Bs, scratch, P.mode, P.key0, P.key1, P.step, env,
                                 logp, value, g);
  if (P.logits)
    for (int j = (int)g.gl; j < P.mlp.n_actions; j += G) P.logits[(int64_t)j * P.ld + i] = Z[j * Bs + slot];
  if (g.gl == 0) {
    if (P.value) P.value[i] = value;
    if (P.action) P.action[i] = (uint8_t)a;
    if (P.logp) P.logp[i] = logp;
  }
}

// ---------------------------------------------------------------------------
// Host launchers
// ---------------------------------------------------------------------------
static unsigned grid_for(int64_t n, int envs_per_block) {
  return (unsigned)((n + envs_per_block - 1) / envs_per_block);
}

int act_stride_pad(const DevMlp& m, int B, int threads) {
  for (int l = 0; l < m.n_layers; ++l)
    if ((B / 4) * ((m.dims[l + 1] + 3) / 4) >= threads) return 4;  // the forward's TE test
  return 1;
}

static size_t env_smem(const RolloutArgs& a, int B) {
  return ((size_t)2 * a.maxd4 * (B + a.bs_pad) + (size_t)a.apad * B) * sizeof(float);
}

// The tensor-core grid forward applies to block-wide forwards of grid policies in blocks
// of at least 128 threads (4 warps cover the 128 lanes of a tile) with layers up to 256
// wide; SIMX_TC_FORWARD=0 turns it off (the FP32 tiles then give the same bits).
size_t plan_tc_forward(RolloutArgs& a, int B) {
  std::memset(&a.tc, 0, sizeof(a.tc));
  const DevMlp& m = a.mlp;
  const bool net = a.policy_mode == SIMX_POLICY_SAMPLE || a.policy_mode == SIMX_POLICY_ARGMAX;
  bool ok = net && m.grid && !a.mlp_warp && a.threads >= 128 && B >= 1 && B <= 32;
  if (const char* f = getenv("SIMX_TC_FORWARD"))
    if (f[0] == '0') ok = false;
  for (int l = 0; ok && l < m.n_layers; ++l)
    if (m.dims[l] > 256 || m.dims[l + 1] > 256) ok = false;
  if (!ok) return env_smem(a, B);
  RolloutArgs t = a;
  const int L = m.n_layers;
  int rows = m.dims[0] > m.dims[L] ? m.dims[0] : m.dims[L];
  t.maxd4 = (rows + 3) / 4 * 4;   // X0 holds the observation, X1 the last layer
  TcPlan& P = t.tc;
  P.Bn = (B + 15) / 16 * 16;
  size_t off = (env_smem(t, B) + 127) / 128 * 128;
  int Kx = 16, cols = 0;
  for (int l = 0; l < L; ++l) {
    P.Kp[l] = (m.dims[l] + 15) / 16 * 16;
    P.nmt[l] = (m.dims[l + 1] + 127) / 128;
    P.w_off[l] = (uint32_t)off;
    off += (size_t)P.nmt[l] * 128 * P.Kp[l] * 2;
    Kx = Kx > P.Kp[l] ? Kx : P.Kp[l];
    cols = cols > P.nmt[l] * P.Bn ? cols : P.nmt[l] * P.Bn;
  }
  for (int b = 0; b < 2; ++b) {
    P.x_off[b] = (uint32_t)off;
    off += (size_t)P.Bn * Kx * 2;
  }
  P.bar_off = (uint32_t)off;
  off += 16;
  P.tcols = cols <= 32 ? 32 : (cols <= 64 ? 64 : 128);
  if (off > 227 * 1024) return env_smem(a, B);
  P.on = 1;
  a = t;
  return off;
}

// Weights of at least this many fp32 bytes are staged in shared memory by default
// (SIMX_STAGE=0 / 1 turns staging off / on for any size); L1 holds smaller ones.
constexpr size_t kStageMinBytes = 64 * 1024;

// Register tiles of the staged forward, layer by layer: the first of 4x8, 2x8, 4x4, 2x4,
// 1x8, 1x4 (envs x outputs) whose tiles keep at least 3/4 of the threads busy, else the
// one that keeps the most busy; false when a layer's tiles outnumber the threads.
static bool stage_tiles(const DevMlp& m, int B, int threads, StagePlan& P) {
  static const int shapes[6][2] = {{4, 8}, {2, 8}, {4, 4}, {2, 4}, {1, 8}, {1, 4}};
  for (int l = 0; l < m.n_layers; ++l) {
    const int N = m.dims[l + 1], Np = m.npad[l + 1];
    int best = -1, best_nt = 0;
    for (int q = 0; q < 6; ++q) {
      const int te = shapes[q][0], to = shapes[q][1];
      if (B % te != 0 || Np % to != 0) continue;
      const int nt = (B / te) * ((N + to - 1) / to);
      if (nt > threads) continue;
      if (4 * nt >= 3 * threads) {
        best = q;
        break;
      }
      if (nt > best_nt) {
        best_nt = nt;
        best = q;
      }
    }
    if (best < 0) return false;
    P.te[l] = shapes[best][0];
    P.to[l] = shapes[best][1];
  }
  return true;
}

// The staged forward's plan (fp32 block-wide forwards of 8 or 16 lanes per env whose
// weights are large): two
// stages of the largest chunk size in 16, 12, 8, 4 KB that keeps the blocks per SM of the
// unstaged launch of `kfn`.  Sets a.stage (and a.bs_pad = 4, so the activation rows stay
// 16-byte aligned) and returns the dynamic shared memory; otherwise leaves a.stage off.
static size_t plan_stage_forward(RolloutArgs& a, int B, const void* kfn) {
  std::memset(&a.stage, 0, sizeof(a.stage));
  const DevMlp& m = a.mlp;
  const size_t plain = env_smem(a, B);
  const bool net = a.policy_mode == SIMX_POLICY_SAMPLE || a.policy_mode == SIMX_POLICY_ARGMAX;
  if (!net || a.mlp_warp || a.tc.on || a.G == 32) return plain;
  int force = -1;
  if (const char* f = getenv("SIMX_STAGE"))
    if (f[0]) force = f[0] == '0' ? 0 : 1;
  if (force == 0) return plain;
  size_t wbytes = 0;
  for (int l = 0; l < m.n_layers; ++l) wbytes += (size_t)m.dims[l] * m.npad[l + 1] * sizeof(float);
  if (force < 0 && wbytes < kStageMinBytes) return plain;
  RolloutArgs t = a;
  t.bs_pad = 4;
  StagePlan& P = t.stage;
  P.S = 2;
  if (!stage_tiles(m, B, a.threads, P)) return plain;
  int r0 = 0;
  cudaFuncSetAttribute(kfn, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&r0, kfn, a.threads, plain) != cudaSuccess) {
    cudaGetLastError();
    return plain;
  }
  const size_t off = (env_smem(t, B) + 127) / 128 * 128;
  for (const uint32_t cb : {16384u, 12288u, 8192u, 4096u}) {
    const size_t total = off + (size_t)P.S * cb + 32;
    int r = 0;
    if (total > 227 * 1024) continue;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&r, kfn, a.threads, total) != cudaSuccess) {
      cudaGetLastError();
      return plain;
    }
    if (r < r0) continue;
    P.cb = cb;
    P.off = (uint32_t)off;
    P.bar_off = (uint32_t)(off + (size_t)P.S * cb);
    P.n = 0;
    for (int l = 0; l < m.n_layers; ++l) {
      const int K = m.dims[l];
      int rpc = (int)(cb / (uint32_t)(m.npad[l + 1] * 4));
      rpc = rpc < K ? rpc : K;
      P.rpc[l] = rpc;
      P.cnt[l] = (K + rpc - 1) / rpc;
      P.n += P.cnt[l];
    }
    P.on = 1;
    a = t;
    return total;
  }
  return plain;
}

// The k_rollout instantiation a launch takes.
template <bool ROUTE, int G>
static auto pick_rollout(const RolloutArgs& a) {
  const bool tr = a.cfg.arrival_kind == SIMX_ARR_TRACE;
  // GRID: the grid policy's instantiations (a.mlp.grid is 0 without a policy)
  const bool gr = a.mlp.grid != 0;
  auto k = tr ? (gr ? k_rollout<ROUTE, G, true, false, true> : k_rollout<ROUTE, G, true, false, false>)
              : (gr ? k_rollout<ROUTE, G, false, false, true> : k_rollout<ROUTE, G, false, false, false>);
  if constexpr (!ROUTE && G >= 16)  // the warp-local forward is instantiated where it applies
    if (a.mlp_warp)
      k = tr ? (gr ? k_rollout<ROUTE, G, true, true, true> : k_rollout<ROUTE, G, true, true, false>)
             : (gr ? k_rollout<ROUTE, G, false, true, true> : k_rollout<ROUTE, G, false, true, false>);
  return k;
}

// The launch's forward plans (tensor-core grid forward, else staged weights); returns the
// dynamic shared memory.
template <bool ROUTE, int G>
static size_t plan_rollout_t(RolloutArgs& a) {
  const int B = a.threads / G;
  const size_t sh = plan_tc_forward(a, B);
  if (a.tc.on) {
    std::memset(&a.stage, 0, sizeof(a.stage));
    return sh;
  }
  return plan_stage_forward(a, B, (const void*)pick_rollout<ROUTE, G>(a));
}

size_t plan_rollout(RolloutArgs& a) {
  const bool route = a.cfg.mode == SIMX_MODE_ROUTE;
  switch (a.G) {
    case 8: return route ? plan_rollout_t<true, 8>(a) : plan_rollout_t<false, 8>(a);
    case 16: return route ? plan_rollout_t<true, 16>(a) : plan_rollout_t<false, 16>(a);
    case 32: return route ? plan_rollout_t<true, 32>(a) : plan_rollout_t<false, 32>(a);
    default: return 0;
  }
}

template <bool ROUTE, int G>
static cudaError_t rollout_t(const RolloutArgs& a0, cudaStream_t s) {
  RolloutArgs a = a0;
  const size_t sh = plan_rollout_t<ROUTE, G>(a);
  auto k = pick_rollout<ROUTE, G>(a);
  cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sh);
  k<<<grid_for(a.st.E, a.threads / G), a.threads, sh, s>>>(a);
  count_launches(1);
  return cudaGetLastError();
}

template <bool ROUTE, int G>
static cudaError_t reset_t(const RolloutArgs& a, cudaStream_t s) {
  auto k = a.cfg.arrival_kind == SIMX_ARR_TRACE ? k_reset<ROUTE, G, true> : k_reset<ROUTE, G, false>;
  k<<<grid_for(a.st.E, a.threads / G), a.threads, 0, s>>>(a);
  count_launches(1);
  return cudaGetLastError();
}

template <bool ROUTE, int G>
static cudaError_t observe_t(const RolloutArgs& a, cudaStream_t s) {
  const int B = a.threads / G;
  const size_t sh = env_smem(a, B);
  cudaFuncSetAttribute(k_observe<ROUTE, G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sh);
  k_observe<ROUTE, G><<<grid_for(a.st.E, B), a.threads, sh, s>>>(a);
  count_launches(1);
  return cudaGetLastError();
}

#define SIMX_DISPATCH(fn, a, s)                                                        \
  do {                                                                                 \
    const bool route = (a).cfg.mode == SIMX_MODE_ROUTE;                                \
    switch ((a).G) {                                                                   \
      case 8: return route ? fn<true, 8>(a, s) : fn<false, 8>(a, s);                  \
      case 16: return route ? fn<true, 16>(a, s) : fn<false, 16>(a, s);               \
      case 32: return route ? fn<true, 32>(a, s) : fn<false, 32>(a, s);               \
      default: return cudaErrorInvalidValue;                                           \
    }                                                                                  \
  } while (0)

cudaError_t launch_rollout(const RolloutArgs& a, cudaStream_t s) { SIMX_DISPATCH(rollout_t, a, s); }
cudaError_t launch_reset(const RolloutArgs& a, cudaStream_t s) { SIMX_DISPATCH(reset_t, a, s); }
cudaError_t launch_observe(const RolloutArgs& a, cudaStream_t s) { SIMX_DISPATCH(observe_t, a, s); }

cudaError_t launch_save(const DevState& st, int32_t cost_type, uint64_t words, uint32_t* out,
                        cudaStream_t s) {
  k_save<<<(st.E + 127) / 128, 128, 0, s>>>(st, cost_type, words, out);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_load(const DevState& st, int32_t cost_type, uint64_t words, const uint32_t* in,
                        cudaStream_t s) {
  k_load<<<(st.E + 127) / 128, 128, 0, s>>>(st, cost_type, words, in);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_stats(const DevState& st, unsigned long long* out, cudaStream_t s) {
  k_stats<<<(st.E + 255) / 256, 256, 0, s>>>(st, out);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_repack(const float* W, const float* b, int N, int K, int Npad, float* Wt,
                          float* bias, cudaStream_t s) {
  const int n = K * Npad > Npad ? K * Npad : Npad;
  k_repack<<<(n + 255) / 256, 256, 0, s>>>(W, b, N, K, Npad, Wt, bias);
  count_launches(1);
  return cudaGetLastError();
}

template <int G>
static cudaError_t policy_forward_t(const PolicyArgs& p, cudaStream_t s) {
  const int B = p.threads / G;
  const size_t sh = ((size_t)2 * p.maxd4 * (B + 4) + (size_t)p.apad * B) * sizeof(float);
  cudaFuncSetAttribute(k_policy_forward<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sh);
  k_policy_forward<G><<<grid_for(p.n, B), p.threads, sh, s>>>(p);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_policy_forward(const PolicyArgs& p, cudaStream_t s) {
  switch (p.G) {
    case 8: return policy_forward_t<8>(p, s);
    case 16: return policy_forward_t<16>(p, s);
    case 32: return policy_forward_t<32>(p, s);
    default: return cudaErrorInvalidValue;
  }
}

// Lanes per env: enough warps to cover every SM at the occupancy the registers
// allow (about 16 warps per SM), but never fewer than 8 lanes per env.
// The environment variable SIMX_LANES (8, 16 or 32) overrides the choice.
int choose_lanes(int64_t envs) {
  if (const char* f = getenv("SIMX_LANES")) {
    const int v = atoi(f);
    if (v == 8 || v == 16 || v == 32) return v;
  }
  const int64_t target_warps = (int64_t)sm_count() * 16;
  if (envs <= target_warps) return 32;
  if (envs * 16 / 32 <= target_warps) return 16;
  return 8;
}

// Threads per block: the largest of 256, 128, 64 that still gives at least four
// blocks per SM (two for 64), so small env counts spread over every SM.
// The environment variable SIMX_THREADS (64, 128 or 256) overrides the choice.
int choose_threads(int64_t envs, int G) {
  if (const char* f = getenv("SIMX_THREADS")) {
    const int v = atoi(f);
    if ((v == 64 || v == 128 || v == 256) && v >= G) return v;
  }
  const int64_t sms = sm_count();
  for (int t = 256; t >= 64; t /= 2) {
    const int64_t blocks = (envs + t / G - 1) / (t / G);
    if (blocks >= (t == 64 ? 2 : 4) * sms || t == 64) return t;
  }
  return 64;
}

}  // namespace simx
