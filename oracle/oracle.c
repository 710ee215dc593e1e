/*
 * oracle.c — TEST INFRASTRUCTURE ONLY.  Plain single-threaded reference of the
 * rollout engine.  Only tests/, the smoke check and bench.py's cpu_baseline leg
 * may build, load or run it; the product library never does.
 *
 * What it follows (paper: "Adaptive Inference Batching using Policy Gradients"):
 *   Sec. 3.1  discrete-event simulator: request arrivals, batch completions and
 *             decision steps on one timeline; requests (arrival time, type);
 *             batch latency L(b) = alpha + beta * b; FIFO queues that drop arrivals
 *             when full; K servers behind a dispatcher that routes or waits.
 *   Sec. 3.2  workloads: Poisson, bursty (two-state MMPP), trace-shaped (diurnal
 *             x lognormal), heterogeneous short/long mix.
 *   Sec. 4.1  MDP: state (queue lengths, time since last batch, head request type,
 *             server status), action (batch size; (server, batch size)), reward
 *             throughput minus weighted queueing latency.
 *   Sec. 4.2  stochastic policy pi(a|s): a tanh MLP with categorical output
 *             (value row appended when present).
 *   Sec. 5.1  baselines: Static, Random, Round-Robin, Shortest-Queue.
 * Every point the paper leaves open (integer microsecond time, tie order, what a
 * decision point is, the observation vector, the random-number mapping) follows
 * the resolved readings listed in the repository's design notes; each function
 * below states the reading it implements.
 *
 * Floating point: every value that decides an integer (event times, acceptance,
 * actions) is computed in fp32 with an explicit operation order, because the GPU
 * takes the same decisions in fp32.  Build with -ffp-contract=off and no fast-math.
 */
#include "oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

#define NONE 0xFFFFFFFFu
#define TIME_LIMIT 0x7FFFFFFFu        /* times are clamped here and flagged */
#define EVENT_CAP (1u << 20)          /* candidates consumed in one decision */
#define ST_TIME 1u
#define ST_EVENT 2u
#define ST_ACTION 4u

/* ------------------------------------------------------------------------- */
/* Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy
 * as 1, 2, 3", SC'11): ten rounds of two 32x32->64 multiplies with the Weyl key
 * schedule.                                                                  */
/* ------------------------------------------------------------------------- */
void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    uint64_t p0 = (uint64_t)0xD2511F53u * (uint64_t)c0;
    uint64_t p1 = (uint64_t)0xCD9E8D57u * (uint64_t)c2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t n0 = hi1 ^ c1 ^ k0;
    uint32_t n2 = hi0 ^ c3 ^ k1;
    c0 = n0;
    c1 = lo1;
    c2 = n2;
    c3 = lo0;
  }
  out[0] = c0;
  out[1] = c1;
  out[2] = c2;
  out[3] = c3;
}

/* ------------------------------------------------------------------------- */
/* Deterministic fp32 elementary functions.  Only IEEE-exact operations (+ - *
 * / sqrt, fused multiply-add, integer bit manipulation) in a fixed order, so any
 * IEEE-754 machine returns the same bits.                                    */
/* ------------------------------------------------------------------------- */
static float f_of(uint32_t u) { float f; memcpy(&f, &u, 4); return f; }
static uint32_t u_of(float f) { uint32_t u; memcpy(&u, &f, 4); return u; }

/* ln 2 split after Cody & Waite: the high part keeps 12 significant bits, so
   k * LN2_HI is exact for |k| < 2^12. */
static const float LN2_HI = 2839.0f / 4096.0f;
static const float LN2_LO = (float)(0.69314718055994530942 - 2839.0 / 4096.0);
static const float LOG2E_F = (float)1.44269504088896340736;
static const float SQRT2_F = (float)1.41421356237309504880;
static const float HALF_PI_F = (float)1.57079632679489661923;
static const float TWO_M24 = 1.0f / 16777216.0f;

/* ln x for positive normal x.  x = 2^e m with m in [sqrt(1/2), sqrt(2)];
   ln m = 2 atanh(s), s = (m-1)/(m+1), through s^11 (|s| <= 0.1716). */
float orc_detlog(float x) {
  uint32_t u = u_of(x);
  int e = (int)((u >> 23) & 0xFFu) - 127;
  float m = f_of((u & 0x7FFFFFu) | 0x3F800000u);
  if (m > SQRT2_F) {
    m = m * 0.5f;
    e += 1;
  }
  float f = m - 1.0f;
  float s = f / (m + 1.0f);
  float z = s * s;
  float p = (float)(1.0 / 11.0);
  p = fmaf(p, z, (float)(1.0 / 9.0));
  p = fmaf(p, z, (float)(1.0 / 7.0));
  p = fmaf(p, z, (float)(1.0 / 5.0));
  p = fmaf(p, z, (float)(1.0 / 3.0));
  float t = s + s;
  float lnm = fmaf(t * z, p, t);
  float fe = (float)e;
  return fmaf(fe, LN2_HI, fmaf(fe, LN2_LO, lnm));
}

/* e^x: k = rint(x log2 e), r = x - k ln 2 (two-part), Taylor to r^7, scale 2^k.
   x < -87 returns 0 and x > 88 returns +inf. */
float orc_detexp(float x) {
  if (x < -87.0f) return 0.0f;
  if (x > 88.0f) return f_of(0x7F800000u);
  float k = rintf(x * LOG2E_F);
  float r = fmaf(-k, LN2_HI, x);
  r = fmaf(-k, LN2_LO, r);
  float p = (float)(1.0 / 5040.0);
  p = fmaf(p, r, (float)(1.0 / 720.0));
  p = fmaf(p, r, (float)(1.0 / 120.0));
  p = fmaf(p, r, (float)(1.0 / 24.0));
  p = fmaf(p, r, (float)(1.0 / 6.0));
  p = fmaf(p, r, 0.5f);
  p = fmaf(p, r, 1.0f);
  p = fmaf(p, r, 1.0f);
  int ki = (int)k;
  return p * f_of((uint32_t)(ki + 127) << 23);
}

/* e^y - 1 for 0 <= y < 0.35: y * (1 + y/2! + ... + y^8/9!). */
static float expm1_small(float y) {
  float q = (float)(1.0 / 362880.0);
  q = fmaf(q, y, (float)(1.0 / 40320.0));
  q = fmaf(q, y, (float)(1.0 / 5040.0));
  q = fmaf(q, y, (float)(1.0 / 720.0));
  q = fmaf(q, y, (float)(1.0 / 120.0));
  q = fmaf(q, y, (float)(1.0 / 24.0));
  q = fmaf(q, y, (float)(1.0 / 6.0));
  q = fmaf(q, y, 0.5f);
  q = fmaf(q, y, 1.0f);
  return q * y;
}

/* tanh z = (e^{2|z|} - 1) / (e^{2|z|} + 1) with the sign of z; |z| >= 10 gives 1. */
float orc_dettanh(float z) {
  float a = fabsf(z);
  float t;
  if (a >= 10.0f) {
    t = 1.0f;
  } else {
    float y = a + a;
    float em1 = (y < 0.35f) ? expm1_small(y) : orc_detexp(y) - 1.0f;
    t = em1 / (em1 + 2.0f);
  }
  return copysignf(t, z);
}

/* GELU in its tanh form (Sec. 4.2 policy head): 0.5 x (1 + tanh(c (x + a x^3))),
   c = sqrt(2/pi), a = 0.044715, in this order: u = fma(a, (x*x)*x, x), t = tanh(c*u),
   (0.5*x) * (1 + t). */
float orc_detgelu(float x) {
  float x3 = (x * x) * x;
  float u = fmaf(0.044715f, x3, x);
  float t = orc_dettanh(0.7978845608028654f * u);
  return (0.5f * x) * (1.0f + t);
}

/* cos(2 pi u) for u in [0, 1): quadrant from 4u, reflection to [0, pi/4],
   Taylor series of sin to theta^11 and of cos to theta^12. */
float orc_detcos2pi(float u) {
  float v = u * 4.0f;
  int q = (int)v;
  float g = v - (float)q;
  int want_sin = q & 1;
  float sign = (q == 1 || q == 2) ? -1.0f : 1.0f;
  if (g > 0.5f) {
    g = 1.0f - g;
    want_sin = !want_sin;
  }
  float th = g * HALF_PI_F;
  float w = th * th;
  float r;
  if (want_sin) {
    float p = (float)(-1.0 / 39916800.0);
    p = fmaf(p, w, (float)(1.0 / 362880.0));
    p = fmaf(p, w, (float)(-1.0 / 5040.0));
    p = fmaf(p, w, (float)(1.0 / 120.0));
    p = fmaf(p, w, (float)(-1.0 / 6.0));
    r = fmaf(th * w, p, th);
  } else {
    float p = (float)(1.0 / 479001600.0);
    p = fmaf(p, w, (float)(-1.0 / 3628800.0));
    p = fmaf(p, w, (float)(1.0 / 40320.0));
    p = fmaf(p, w, (float)(-1.0 / 720.0));
    p = fmaf(p, w, (float)(1.0 / 24.0));
    p = fmaf(p, w, -0.5f);
    r = fmaf(w, p, 1.0f);
  }
  return sign * r;
}

static float u_open0(uint32_t w) { return (float)((w >> 8) + 1u) * TWO_M24; } /* (0, 1] */
static float u_open1(uint32_t w) { return (float)(w >> 8) * TWO_M24; }        /* [0, 1) */
static float expo1(uint32_t w) { return -orc_detlog(u_open0(w)); }            /* Exp(1) */

/* Standard normal by Box-Muller (Box & Muller 1958) from two Philox words. */
float orc_normal(uint32_t w0, uint32_t w1) {
  float r = sqrtf(-2.0f * orc_detlog(u_open0(w0)));
  return r * orc_detcos2pi(u_open1(w1));
}

/* A sampled duration in integer microseconds: round half up, saturated at 2^26. */
uint32_t orc_duration(float x) {
  float y = x + 0.5f;
  if (!(y < 67108864.0f)) return 67108864u;
  return (uint32_t)floorf(y);
}

/* ------------------------------------------------------------------------- */
/* Environment                                                                */
/* ------------------------------------------------------------------------- */
struct orc_env {
  orc_config c;
  uint32_t id, key[2];
  uint32_t K, T, cap, A;
  uint32_t now, t_global, cand_j, cand_T, sw_i, sw_T, mstate, epoch, epoch_off;
  uint32_t pend_time, pend_type, pend_cost;
  uint32_t n_arrived, n_dropped, n_dispatched, n_batches;
  uint64_t sum_wait;
  uint32_t t_last_dispatch, prev_now, n_last, type_last;
  float last_mean_wait, rate_est;
  uint32_t narr_since[2], ndrop_since[2];
  uint32_t status;
  uint32_t busy_until[ORC_MAX_SERVERS], bsize[ORC_MAX_SERVERS];
  uint32_t qhead[ORC_MAX_SERVERS][2], qcnt[ORC_MAX_SERVERS][2];
  uint32_t* qarr;  /* [K][2][cap] arrival times */
  uint32_t* qcost; /* [K][cap] per-request cost of the Pareto type */
  uint32_t events;
  uint64_t q_area[ORC_MAX_SERVERS][2]; /* integral of queue length, event by event */
  uint32_t q_last[ORC_MAX_SERVERS][2]; /* time of that queue's last change */
  uint32_t step_n;
  uint64_t step_w[2];
  uint32_t* swlog;   /* optional log of the modulating chain: (time, state) pairs */
  uint32_t swlog_cap, swlog_n;
};

uint32_t orc_obs_dim(const orc_config* c) {
  if (c->mode == ORC_SINGLE) return 2u * c->n_types + 6u + (c->obs_extra ? 6u : 0u);
  return 3u * c->n_servers + 1u + (c->obs_extra ? 3u : 0u);
}

uint64_t orc_state_words(const orc_config* c) {
  uint64_t K = c->n_servers, T = c->n_types, cap = c->queue_cap;
  uint64_t w = ORC_HEADER_WORDS + 2 * K + K * T + K * T * cap;
  if (c->cost_type >= 0) w += K * cap;
  return w;
}

static void draw(const orc_env* e, uint32_t idx, uint32_t stream, uint32_t w[4]) {
  uint32_t ctr[4] = {idx, e->id, stream, 0u};
  orc_philox4x32_10(ctr, e->key, w);
}

static uint32_t add_time(orc_env* e, uint32_t a, uint64_t b) {
  uint64_t s = (uint64_t)a + b;
  if (s >= TIME_LIMIT) {
    e->status |= ST_TIME;
    return TIME_LIMIT;
  }
  return (uint32_t)s;
}

static int count_event(orc_env* e) {
  if (++e->events > EVENT_CAP) {
    e->status |= ST_EVENT;
    return 1;
  }
  return 0;
}

static uint32_t* ring(orc_env* e, uint32_t k, uint32_t t) {
  return e->qarr + ((size_t)k * 2 + t) * e->cap;
}

/* Queue-length integral: add length x elapsed time before every change at time at. */
static void area_to(orc_env* e, uint32_t k, uint32_t t, uint32_t at) {
  e->q_area[k][t] += (uint64_t)e->qcnt[k][t] * (uint64_t)(at - e->q_last[k][t]);
  e->q_last[k][t] = at;
}

static void push(orc_env* e, uint32_t k, uint32_t t, uint32_t arr, uint32_t cost) {
  area_to(e, k, t, arr);
  uint32_t slot = (e->qhead[k][t] + e->qcnt[k][t]) & (e->cap - 1);
  ring(e, k, t)[slot] = arr;
  if ((int32_t)t == e->c.cost_type) e->qcost[(size_t)k * e->cap + slot] = cost;
  e->qcnt[k][t] += 1;
}

/* Remove the head of queue (k, t) when its batch starts at time s. */
static void pop(orc_env* e, uint32_t k, uint32_t t, uint32_t s, uint32_t* arr, uint32_t* cost) {
  area_to(e, k, t, s);
  uint32_t slot = e->qhead[k][t];
  *arr = ring(e, k, t)[slot];
  *cost = ((int32_t)t == e->c.cost_type) ? e->qcost[(size_t)k * e->cap + slot] : 0u;
  e->qhead[k][t] = (slot + 1) & (e->cap - 1);
  e->qcnt[k][t] -= 1;
}

static uint32_t queued(const orc_env* e) {
  uint32_t s = 0;
  for (uint32_t k = 0; k < e->K; ++k)
    for (uint32_t t = 0; t < e->T; ++t) s += e->qcnt[k][t];
  return s;
}

/* The type whose head request arrived first at server k (tie: lower type). */
static uint32_t head_type(orc_env* e, uint32_t k) {
  uint32_t best = NONE, bt = 0;
  for (uint32_t t = 0; t < e->T; ++t) {
    if (e->qcnt[k][t] == 0) continue;
    uint32_t h = ring(e, k, t)[e->qhead[k][t]];
    if (best == NONE || h < bt) {
      best = t;
      bt = h;
    }
  }
  return best;
}

/* Request type from word w1 and, for the cost type, its per-request cost from
   word w3 with E ~ Exp(1): Pareto by inversion, cost = round(x_m exp(E / alpha));
   exponential, cost = round(mean E).  Under trace replay, candidate j takes the type
   (clamped to the last type) and the cost of trace entry j mod n where the trace has
   them. */
static void request_attrs(const orc_env* e, uint32_t j, const uint32_t w[4], uint32_t* type,
                          uint32_t* cost) {
  uint32_t t = (e->T > 1 && (w[1] >> 8) >= e->c.type0_thr) ? 1u : 0u;
  if (e->c.trace_type) {
    t = e->c.trace_type[j % e->c.trace_len];
    if (t >= e->T) t = e->T - 1u;
  }
  uint32_t cst = 0;
  if ((int32_t)t == e->c.cost_type && e->c.trace_cost) {
    cst = e->c.trace_cost[j % e->c.trace_len];
  } else if ((int32_t)t == e->c.cost_type) {
    float E = expo1(w[3]);
    if (e->c.cost_kind == 0) {
      float y = e->c.pareto_inv_alpha * E;
      cst = orc_duration(e->c.cost_scale_us * orc_detexp(y));
    } else {
      cst = orc_duration(e->c.cost_scale_us * E);
    }
  }
  *type = t;
  *cost = cst;
}

/* Dwell of the modulating chain before switch i: round(dwell * E_i) with E_i the
   exponential of the switch's draw, or exactly round(dwell) for a fixed dwell (the
   square wave of the paper's Extreme Burst workload, Sec. 3.2). */
static uint32_t dwell_us(orc_env* e, uint32_t i) {
  if (e->c.dwell_kind == 1) return orc_duration(e->c.dwell_mean_us);
  uint32_t w[4];
  draw(e, i, ORC_STREAM_SWITCH, w);
  return orc_duration(e->c.dwell_mean_us * expo1(w[0]));
}

/* Test hook: record (time, state) of the modulating chain, at reset and at every switch
   processed, when the caller attached a log (orc_env_switch_log).  Records nothing
   that the simulation reads. */
static void swlog_push(orc_env* e, uint32_t t, uint32_t state) {
  if (!e->swlog || e->swlog_n >= e->swlog_cap) return;
  e->swlog[2 * e->swlog_n] = t;
  e->swlog[2 * e->swlog_n + 1] = state;
  e->swlog_n += 1u;
}

/* Modulating chain: switch i >= 1 at S_i = S_{i-1} + dwell_i, S_0 = 0.
   All switches at times <= limit take effect. */
static void process_switches(orc_env* e, uint32_t limit) {
  if (e->c.n_mod_states < 2) return;
  while (e->sw_T <= limit) {
    if (count_event(e)) return;
    e->mstate ^= 1u;
    swlog_push(e, e->sw_T, e->mstate);
    e->sw_i += 1u;
    e->sw_T = add_time(e, e->sw_T, dwell_us(e, e->sw_i));
  }
}

/* Time of candidate j given the previous candidate's time: a drawn exponential gap,
   or under trace replay the gap of trace entry j mod n. */
static uint32_t cand_time(orc_env* e, uint32_t j, uint32_t base, uint32_t w[4]) {
  draw(e, j, ORC_STREAM_ARRIVAL, w);
  if (e->c.arrival_kind == ORC_ARR_TRACE) return add_time(e, base, e->c.trace_gap[j % e->c.trace_len]);
  return add_time(e, base, orc_duration(e->c.cand_mean_gap_us * expo1(w[0])));
}

/* Thinning (Lewis & Shedler 1979): candidate accepted with probability
   accept_thr[state] / 2^24 where state is the chain's state at its time. */
static int accepted(const orc_env* e, const uint32_t w[4]) {
  return (w[2] >> 8) < e->c.accept_thr[e->mstate];
}

/* SINGLE mode: a consumed candidate joins its type's FIFO or is dropped. */
static int consume_single(orc_env* e, const uint32_t w[4], uint32_t T) {
  if (!accepted(e, w)) return 0;
  uint32_t type, cost;
  request_attrs(e, e->cand_j, w, &type, &cost);
  e->n_arrived += 1;
  e->narr_since[type] += 1;
  if (e->qcnt[0][type] < e->cap) {
    push(e, 0, type, T, cost);
  } else {
    e->n_dropped += 1;
    e->ndrop_since[type] += 1;
  }
  return 1;
}

/* SINGLE mode: consume every candidate with time <= target. */
static void advance_single(orc_env* e, uint32_t target) {
  for (;;) {
    uint32_t w[4];
    uint32_t T = cand_time(e, e->cand_j, e->cand_T, w);
    if (T > target) break;
    if (count_event(e)) return;
    process_switches(e, T);
    consume_single(e, w, T);
    e->cand_j += 1;
    e->cand_T = T;
  }
  process_switches(e, target);
}

/* SINGLE mode: move to the next accepted arrival (the next decision point when
   no request is waiting) and take in everything up to that time. */
static void jump_single(orc_env* e) {
  for (;;) {
    uint32_t w[4];
    uint32_t T = cand_time(e, e->cand_j, e->cand_T, w);
    if (count_event(e)) return;
    process_switches(e, T);
    int acc = consume_single(e, w, T);
    e->cand_j += 1;
    e->cand_T = T;
    if (acc) {
      e->now = T;
      advance_single(e, T);
      return;
    }
  }
}

/* ROUTE mode: draw the next request arrival into the pending slot. */
static void next_arrival(orc_env* e) {
  for (;;) {
    if (count_event(e)) return;
    uint32_t w[4];
    if (e->c.arrival_kind != ORC_ARR_DIURNAL) { /* THINNED or TRACE */
      uint32_t j = e->cand_j;
      uint32_t T = cand_time(e, j, e->cand_T, w);
      process_switches(e, T);
      int acc = accepted(e, w);
      e->cand_j += 1;
      e->cand_T = T;
      if (!acc) continue;
      request_attrs(e, j, w, &e->pend_type, &e->pend_cost);
      e->pend_time = T;
      e->n_arrived += 1;
      return;
    }
    /* DIURNAL: constant rate inside an epoch; a gap that crosses the epoch end is
       discarded and redrawn from the epoch end at the next epoch's rate (exact for a
       piecewise-constant Poisson rate by memorylessness). */
    uint32_t we[4];
    draw(e, e->epoch, ORC_STREAM_EPOCH, we);
    float factor = orc_detexp(e->c.burst_sigma * orc_normal(we[0], we[1]));
    float rate = e->c.diurnal_rate[(e->epoch + e->epoch_off) % e->c.diurnal_len] * factor;
    float mean = 1.0e6f / rate;
    draw(e, e->cand_j, ORC_STREAM_ARRIVAL, w);
    uint32_t g = orc_duration(mean * expo1(w[0]));
    e->cand_j += 1;
    uint64_t end = (uint64_t)(e->epoch + 1u) * (uint64_t)e->c.epoch_us;
    if ((uint64_t)e->cand_T + g < end) {
      e->cand_T = add_time(e, e->cand_T, g);
      request_attrs(e, 0, w, &e->pend_type, &e->pend_cost);
      e->pend_time = e->cand_T;
      e->n_arrived += 1;
      return;
    }
    if (end >= TIME_LIMIT) {
      e->status |= ST_TIME;
      e->cand_T = TIME_LIMIT;
    } else {
      e->cand_T = (uint32_t)end;
    }
    e->epoch += 1u;
  }
}

/* Batch latency on server k (Sec. 3.1 execution model; K heterogeneous GPUs): L =
   alpha + beta n, or alpha + the sum of the batch's per-request costs for the cost type,
   scaled by the server's speed factor s/16 and rounded to the nearest microsecond
   (halves up): (L s + 8) / 16 in integers, which is L itself for s = 16. */
static uint64_t service_time(const orc_env* e, uint32_t k, uint32_t type, uint32_t n, uint64_t csum) {
  uint64_t L;
  if ((int32_t)type == e->c.cost_type) L = (uint64_t)e->c.alpha_us[type] + csum;
  else L = (uint64_t)e->c.alpha_us[type] + (uint64_t)e->c.beta_us[type] * n;
  const uint64_t s = e->c.srv_speed16[k] ? e->c.srv_speed16[k] : 16u;
  return (L * s + 8u) / 16u;
}

/* ROUTE mode: server k starts a batch at time s from the queue whose head is
   oldest: n = min(b_k, queue length); L = alpha + beta n, or alpha + sum of the
   requests' Pareto costs for the Pareto type. */
static void try_start(orc_env* e, uint32_t k, uint32_t s) {
  uint32_t h = head_type(e, k);
  if (h == NONE) return;
  uint32_t n = e->bsize[k] < e->qcnt[k][h] ? e->bsize[k] : e->qcnt[k][h];
  uint64_t W = 0, csum = 0;
  for (uint32_t i = 0; i < n; ++i) {
    uint32_t arr, cost;
    pop(e, k, h, s, &arr, &cost);
    W += (uint64_t)(s - arr);
    csum += cost;
  }
  uint64_t L = service_time(e, k, h, n, csum);
  e->busy_until[k] = add_time(e, s, L);
  e->step_n += n;
  e->step_w[h] += W;
  e->n_dispatched += n;
  e->sum_wait += W;
  e->n_batches += 1;
}

/* ROUTE mode: every completion at or before t starts the next batch of its server. */
static void advance_servers(orc_env* e, uint32_t t) {
  for (uint32_t k = 0; k < e->K; ++k)
    while (e->busy_until[k] <= t && (e->qcnt[k][0] + e->qcnt[k][1]) > 0)
      try_start(e, k, e->busy_until[k]);
}

orc_env* orc_env_new(const orc_config* c, uint32_t env_id, uint64_t seed) {
  orc_env* e = (orc_env*)calloc(1, sizeof(orc_env));
  if (!e) return NULL;
  e->c = *c;
  e->id = env_id;
  e->key[0] = (uint32_t)seed;
  e->key[1] = (uint32_t)(seed >> 32);
  e->K = c->n_servers;
  e->T = c->n_types;
  e->cap = c->queue_cap;
  e->A = (c->mode == ORC_SINGLE ? c->n_types : c->n_servers) * c->n_bsizes +
         (c->action_layout == 1 ? 1u : 0u);
  e->qarr = (uint32_t*)calloc((size_t)e->K * 2 * e->cap, sizeof(uint32_t));
  e->qcost = (uint32_t*)calloc((size_t)e->K * e->cap, sizeof(uint32_t));
  if (!e->qarr || !e->qcost) {
    orc_env_free(e);
    return NULL;
  }
  return e;
}

void orc_env_free(orc_env* e) {
  if (!e) return;
  free(e->qarr);
  free(e->qcost);
  free(e);
}

uint32_t orc_env_status(const orc_env* e) { return e->status; }

void orc_env_switch_log(orc_env* e, uint32_t* pairs, uint32_t cap) {
  e->swlog = pairs;
  e->swlog_cap = pairs ? cap : 0u;
  e->swlog_n = 0;
}

uint32_t orc_env_switch_log_count(const orc_env* e) { return e->swlog_n; }

void orc_env_little(const orc_env* ec, uint32_t t_end, uint64_t* area, uint64_t* waits) {
  orc_env* e = (orc_env*)ec;
  uint64_t a = 0, w = e->sum_wait;
  for (uint32_t k = 0; k < e->K; ++k)
    for (uint32_t t = 0; t < e->T; ++t) {
      a += e->q_area[k][t] + (uint64_t)e->qcnt[k][t] * (uint64_t)(t_end - e->q_last[k][t]);
      for (uint32_t i = 0; i < e->qcnt[k][t]; ++i)
        w += (uint64_t)(t_end - ring(e, k, t)[(e->qhead[k][t] + i) & (e->cap - 1)]);
    }
  *area = a;
  *waits = w;
}

void orc_env_reset(orc_env* e) {
  uint32_t id = e->id, key0 = e->key[0], key1 = e->key[1];
  orc_config c = e->c;
  uint32_t* qa = e->qarr;
  uint32_t* qc = e->qcost;
  uint32_t K = e->K, T = e->T, cap = e->cap, A = e->A;
  uint32_t* swlog = e->swlog;
  const uint32_t swlog_cap = e->swlog_cap;
  memset(e, 0, sizeof(*e));
  e->swlog = swlog;
  e->swlog_cap = swlog_cap;
  e->c = c;
  e->id = id;
  e->key[0] = key0;
  e->key[1] = key1;
  e->qarr = qa;
  e->qcost = qc;
  e->K = K;
  e->T = T;
  e->cap = cap;
  e->A = A;
  memset(qa, 0, (size_t)K * 2 * cap * sizeof(uint32_t));
  memset(qc, 0, (size_t)K * cap * sizeof(uint32_t));
  e->type_last = NONE;
  e->rate_est = c.rate_ref;
  for (uint32_t k = 0; k < K; ++k)
    e->bsize[k] = c.action_layout == 1 ? c.static_bi + 1u : c.bsizes[c.static_bi];
  uint32_t w[4];
  draw(e, 0, ORC_STREAM_INIT, w);
  if (c.n_mod_states == 2) {
    e->mstate = w[0] >> 31;
    swlog_push(e, 0, e->mstate);
    e->sw_i = 1;
    e->sw_T = add_time(e, 0, dwell_us(e, 1));
  } else {
    e->mstate = 0;
    e->sw_i = 0;
    e->sw_T = NONE;
  }
  if (c.arrival_kind == ORC_ARR_DIURNAL)
    e->epoch_off = (uint32_t)(((uint64_t)(w[1] >> 8) * c.diurnal_len) >> 24);
  if (c.arrival_kind == ORC_ARR_TRACE) /* this env's first trace entry: floor(u n / 2^32) */
    e->cand_j = (uint32_t)(((uint64_t)w[2] * c.trace_len) >> 32);
  if (c.mode == ORC_SINGLE) {
    jump_single(e);
  } else {
    next_arrival(e);
    e->now = e->pend_time;
  }
  e->events = 0;
}

void orc_env_observe(const orc_env* ec, float* obs) {
  orc_env* e = (orc_env*)ec;
  const orc_config* c = &e->c;
  uint32_t i = 0;
  if (c->mode == ORC_SINGLE) {
    float fcap = (float)e->cap;
    for (uint32_t t = 0; t < e->T; ++t) obs[i++] = (float)e->qcnt[0][t] / fcap;
    obs[i++] = (float)(e->now - e->t_last_dispatch) / c->t_window_us;
    uint32_t h = head_type(e, 0);
    obs[i++] = (h == 0) ? 1.0f : 0.0f;
    obs[i++] = (h == 1) ? 1.0f : 0.0f;
    obs[i++] = 0.0f; /* server status: always free at a SINGLE-mode decision */
    uint32_t dt = e->now - e->prev_now;
    if (dt < 1) dt = 1;
    float fdt = (float)dt;
    obs[i++] = ((float)(e->narr_since[0] + e->narr_since[1]) * c->rate_scale) / fdt;
    obs[i++] = (float)e->n_last / 32.0f;
    for (uint32_t t = 0; t < e->T; ++t)
      obs[i++] = e->qcnt[0][t] > 0
                     ? (float)(e->now - ring(e, 0, t)[e->qhead[0][t]]) / c->t_window_us
                     : 0.0f;
    if (c->obs_extra) {
      obs[i++] = ((float)e->narr_since[0] * c->rate_scale) / fdt;
      obs[i++] = ((float)e->narr_since[1] * c->rate_scale) / fdt;
      obs[i++] = (e->type_last == 0) ? 1.0f : 0.0f;
      obs[i++] = (e->type_last == 1) ? 1.0f : 0.0f;
      obs[i++] = (float)(e->ndrop_since[0] + e->ndrop_since[1]) / 32.0f;
      obs[i++] = e->last_mean_wait / c->t_window_us;
    }
  } else {
    float fcap = (float)e->cap;
    for (uint32_t k = 0; k < e->K; ++k) {
      obs[i++] = (float)e->qcnt[k][0] / fcap;
      obs[i++] = (float)(e->T > 1 ? e->qcnt[k][1] : 0u) / fcap;
      uint32_t rem = e->busy_until[k] > e->now ? e->busy_until[k] - e->now : 0u;
      obs[i++] = (float)rem / c->busy_norm_us;
    }
    obs[i++] = e->rate_est / c->rate_ref;
    if (c->obs_extra) {
      obs[i++] = (e->pend_type == 0) ? 1.0f : 0.0f;
      obs[i++] = (e->pend_type == 1) ? 1.0f : 0.0f;
      uint32_t ph = (e->now + e->epoch_off * c->epoch_us) % c->phase_period_us;
      obs[i++] = (float)ph / (float)c->phase_period_us;
    }
  }
}

/* Policy (Sec. 4.2): tanh MLP; categorical sampling by inversion of the cumulative
   softmax with a POLICY-stream uniform, or argmax.  All fp32, sums in index order. */
/* Grid rounding of the grid policy: v 2^e is an exact power-of-two scaling in fp64,
   nearbyint rounds to nearest with ties to even (the default mode), and the clamped
   integer times 2^-e is exact in fp32. */
float orc_gridq(float v, int32_t e) {
  double r = nearbyint(ldexp((double)v, e));
  if (r > 255.0) r = 255.0;
  if (r < -255.0) r = -255.0;
  return (float)ldexp(r, -e);
}

void orc_gridq_n(const float* v, int64_t n, int32_t e, float* out) {
  for (int64_t i = 0; i < n; ++i) out[i] = orc_gridq(v[i], e);
}

void orc_policy(const orc_mlp* m, const float* obs, int mode, uint64_t seed, uint32_t step,
                uint32_t env_id, float* logits, float* value, int32_t* action, float* logp) {
  float bufa[512], bufb[512], bufq[512];
  const float* x = obs;
  float* y = bufa;
  if (m->grid) {
    for (int k = 0; k < m->dims[0]; ++k) bufq[k] = orc_gridq(obs[k], m->gx[0]);
    x = bufq;
  }
  for (int l = 0; l < m->n_layers; ++l) {
    int K = m->dims[l], N = m->dims[l + 1];
    const float* W = m->W[l];
    for (int j = 0; j < N; ++j) {
      float z;
      if (m->grid) {
        /* the exact dot product: each fp64 product of two floats is exact, and so is the
           fp64 sum of grid products; one rounding to fp32 at the end */
        double acc = 0.0;
        for (int k = 0; k < K; ++k) acc += (double)W[(size_t)j * K + k] * (double)x[k];
        z = (float)(acc + (double)m->b[l][j]);
      } else {
        float acc = 0.0f;
        for (int k = 0; k < K; ++k) acc = fmaf(W[(size_t)j * K + k], x[k], acc);
        z = acc + m->b[l][j];
      }
      if (l + 1 < m->n_layers) {
        if (m->act[l] == 1) y[j] = z;
        else if (m->act[l] == 2) y[j] = orc_detgelu(z);
        else y[j] = orc_dettanh(z);
        if (m->grid) y[j] = orc_gridq(y[j], m->gx[l + 1]);
      } else {
        y[j] = z;
      }
    }
    x = y;
    y = (y == bufa) ? bufb : bufa;
  }
  int N = m->dims[m->n_layers];
  int A = N - (m->has_value ? 1 : 0);
  if (value) *value = m->has_value ? x[A] : 0.0f;
  if (logits)
    for (int i = 0; i < A; ++i) logits[i] = x[i];
  float mx = x[0];
  int amax = 0;
  for (int i = 1; i < A; ++i)
    if (x[i] > mx) {
      mx = x[i];
      amax = i;
    }
  float p[512];
  float S = 0.0f;
  for (int i = 0; i < A; ++i) {
    p[i] = orc_detexp(x[i] - mx);
    S = S + p[i];
  }
  int a;
  if (mode == ORC_ARGMAX) {
    a = amax;
  } else {
    uint32_t ctr[4] = {step, env_id, ORC_STREAM_POLICY, 0u};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t w[4];
    orc_philox4x32_10(ctr, key, w);
    float thr = u_open1(w[0]) * S;
    float cum = 0.0f;
    a = A - 1;
    for (int i = 0; i < A; ++i) {
      cum = cum + p[i];
      if (cum > thr) {
        a = i;
        break;
      }
    }
  }
  *action = a;
  if (logp) *logp = (x[a] - mx) - orc_detlog(S);
}

static int32_t choose_action(orc_env* e, const orc_mlp* m, int mode, int32_t ext,
                             const float* obs, orc_step_out* o) {
  const orc_config* c = &e->c;
  o->logp = 0.0f;
  o->value = 0.0f;
  if (mode == ORC_SAMPLE || mode == ORC_ARGMAX) {
    uint64_t seed = (uint64_t)e->key[0] | ((uint64_t)e->key[1] << 32);
    int32_t a;
    orc_policy(m, obs, mode, seed, e->t_global, e->id, o->logits, &o->value, &a, &o->logp);
    return a;
  }
  if (mode == ORC_EXTERNAL) {
    if (ext < 0 || (uint32_t)ext >= e->A) {
      e->status |= ST_ACTION;
      return 0;
    }
    return ext;
  }
  if (mode == ORC_RANDOM) {
    uint32_t w[4];
    draw(e, e->t_global, ORC_STREAM_POLICY, w);
    return (int32_t)(((uint64_t)(w[1] >> 8) * e->A) >> 24);
  }
  if (mode == ORC_STATIC) {
    uint32_t h = head_type(e, 0);
    if (h == NONE) h = 0;
    return (int32_t)((c->action_layout == 1 ? 1u : 0u) + h * c->n_bsizes + c->static_bi);
  }
  if (mode == ORC_RR) return (int32_t)((e->t_global % e->K) * c->n_bsizes + c->static_bi);
  /* ORC_SQ: fewest queued requests, first such server */
  uint32_t best = 0, bq = NONE;
  for (uint32_t k = 0; k < e->K; ++k) {
    uint32_t q = e->qcnt[k][0] + e->qcnt[k][1];
    if (q < bq) {
      bq = q;
      best = k;
    }
  }
  return (int32_t)(best * c->n_bsizes + c->static_bi);
}

/* Action a -> (major, batch size) (Sec. 4.1).  Layout 0: major a / n_bsizes, batch
   bsizes[a % n_bsizes].  Layout 1: a = 0 is "Wait" (batch 0: nothing is dispatched and the
   next decision is at the next arrival), a >= 1 is major (a - 1) / n_bsizes with batch
   ((a - 1) % n_bsizes) + 1. */
static void decode_action(const orc_config* c, int32_t a, uint32_t* major, uint32_t* b) {
  if (c->action_layout == 1) {
    if (a == 0) {
      *major = 0;
      *b = 0;
    } else {
      *major = (uint32_t)(a - 1) / c->n_bsizes;
      *b = (uint32_t)(a - 1) % c->n_bsizes + 1u;
    }
    return;
  }
  *major = (uint32_t)a / c->n_bsizes;
  *b = c->bsizes[(uint32_t)a % c->n_bsizes];
}

static void step_single(orc_env* e, const orc_mlp* m, int mode, int32_t ext, orc_step_out* o) {
  const orc_config* c = &e->c;
  int frozen = e->status != 0;
  orc_env_observe(e, o->obs);
  int32_t a = choose_action(e, m, mode, ext, o->obs, o);
  uint32_t k, b;
  decode_action(c, a, &k, &b);
  uint32_t now = e->now;
  uint32_t n = 0;
  uint64_t W = 0, csum = 0;
  if (!frozen) {
    n = b < e->qcnt[0][k] ? b : e->qcnt[0][k];
    for (uint32_t i = 0; i < n; ++i) {
      uint32_t arr, cost;
      pop(e, 0, k, now, &arr, &cost);
      W += (uint64_t)(now - arr);
      csum += cost;
    }
    if (n > 0) {
      e->busy_until[0] = add_time(e, now, service_time(e, 0, k, n, csum));
      e->n_last = n;
      e->type_last = k;
      e->t_last_dispatch = now;
      e->last_mean_wait = (float)W / (float)n;
      e->n_batches += 1;
    }
    e->n_dispatched += n;
    e->sum_wait += W;
  }
  o->action = a;
  o->reward = (float)n - c->w_wait[k] * (float)W;
  o->done = ((e->t_global + 1u) % c->episode_len) == 0u;
  o->trace[0] = now;
  o->trace[1] = n;
  o->trace[2] = (int64_t)W;
  o->trace[3] = queued(e);
  e->prev_now = now;
  e->narr_since[0] = e->narr_since[1] = 0;
  e->ndrop_since[0] = e->ndrop_since[1] = 0;
  e->t_global += 1;
  if (frozen) return;
  e->events = 0;
  if (n > 0) {
    uint32_t next = e->busy_until[0];
    advance_single(e, next);
    e->now = next;
    if (queued(e) == 0) jump_single(e);
  } else {
    jump_single(e);
  }
}

static void step_route(orc_env* e, const orc_mlp* m, int mode, int32_t ext, orc_step_out* o) {
  const orc_config* c = &e->c;
  int frozen = e->status != 0;
  orc_env_observe(e, o->obs);
  int32_t a = choose_action(e, m, mode, ext, o->obs, o);
  uint32_t k, b;
  decode_action(c, a, &k, &b);
  uint32_t A = e->pend_time;
  e->step_n = 0;
  e->step_w[0] = e->step_w[1] = 0;
  uint32_t qafter = queued(e);
  if (!frozen) {
    e->events = 0;
    uint32_t mt = e->pend_type;
    if (e->qcnt[k][mt] < e->cap) {
      push(e, k, mt, A, e->pend_cost);
    } else {
      e->n_dropped += 1;
      e->ndrop_since[mt] += 1;
    }
    e->bsize[k] = b;
    if (e->busy_until[k] <= A) try_start(e, k, A);
    qafter = queued(e);
    next_arrival(e);
    uint32_t gap = e->pend_time - A;
    if (gap < 1) gap = 1;
    float inst = 1.0e6f / (float)gap;
    e->rate_est = e->rate_est + 0.0625f * (inst - e->rate_est);
    advance_servers(e, e->pend_time);
    e->now = e->pend_time;
  }
  o->action = a;
  o->reward = (float)e->step_n -
              (c->w_wait[0] * (float)e->step_w[0] + c->w_wait[1] * (float)e->step_w[1]);
  o->done = ((e->t_global + 1u) % c->episode_len) == 0u;
  o->trace[0] = A;
  o->trace[1] = e->step_n;
  o->trace[2] = (int64_t)(e->step_w[0] + e->step_w[1]);
  o->trace[3] = qafter;
  e->prev_now = A;
  e->t_global += 1;
}

void orc_env_step(orc_env* e, const orc_mlp* m, int mode, int32_t ext, orc_step_out* o) {
  if (e->c.mode == ORC_SINGLE)
    step_single(e, m, mode, ext, o);
  else
    step_route(e, m, mode, ext, o);
}

void orc_env_export(const orc_env* ec, uint32_t* w) {
  orc_env* e = (orc_env*)ec;
  memset(w, 0, orc_state_words(&e->c) * sizeof(uint32_t));
  w[0] = e->now;
  w[1] = e->t_global;
  w[2] = e->cand_j;
  w[3] = e->cand_T;
  w[4] = e->sw_i;
  w[5] = e->sw_T;
  w[6] = e->mstate;
  w[7] = e->epoch;
  w[8] = e->epoch_off;
  w[9] = e->pend_time;
  w[10] = e->pend_type;
  w[11] = e->pend_cost;
  w[12] = e->n_arrived;
  w[13] = e->n_dropped;
  w[14] = e->n_dispatched;
  w[15] = e->n_batches;
  w[16] = (uint32_t)e->sum_wait;
  w[17] = (uint32_t)(e->sum_wait >> 32);
  w[18] = e->t_last_dispatch;
  w[19] = e->prev_now;
  w[20] = e->n_last;
  w[21] = e->type_last;
  w[22] = u_of(e->last_mean_wait);
  w[23] = u_of(e->rate_est);
  w[24] = e->narr_since[0];
  w[25] = e->narr_since[1];
  w[26] = e->ndrop_since[0];
  w[27] = e->ndrop_since[1];
  w[28] = e->status;
  uint32_t* p = w + ORC_HEADER_WORDS;
  for (uint32_t k = 0; k < e->K; ++k) {
    *p++ = e->busy_until[k];
    *p++ = e->bsize[k];
  }
  for (uint32_t k = 0; k < e->K; ++k)
    for (uint32_t t = 0; t < e->T; ++t) *p++ = e->qcnt[k][t];
  for (uint32_t k = 0; k < e->K; ++k)
    for (uint32_t t = 0; t < e->T; ++t) {
      for (uint32_t i = 0; i < e->qcnt[k][t]; ++i)
        p[i] = ring(e, k, t)[(e->qhead[k][t] + i) & (e->cap - 1)];
      p += e->cap;
    }
  if (e->c.cost_type >= 0) {
    uint32_t t = (uint32_t)e->c.cost_type;
    for (uint32_t k = 0; k < e->K; ++k) {
      for (uint32_t i = 0; i < e->qcnt[k][t]; ++i)
        p[i] = e->qcost[(size_t)k * e->cap + ((e->qhead[k][t] + i) & (e->cap - 1))];
      p += e->cap;
    }
  }
}

void orc_env_import(orc_env* e, const uint32_t* w) {
  e->now = w[0];
  e->t_global = w[1];
  e->cand_j = w[2];
  e->cand_T = w[3];
  e->sw_i = w[4];
  e->sw_T = w[5];
  e->mstate = w[6];
  e->epoch = w[7];
  e->epoch_off = w[8];
  e->pend_time = w[9];
  e->pend_type = w[10];
  e->pend_cost = w[11];
  e->n_arrived = w[12];
  e->n_dropped = w[13];
  e->n_dispatched = w[14];
  e->n_batches = w[15];
  e->sum_wait = (uint64_t)w[16] | ((uint64_t)w[17] << 32);
  e->t_last_dispatch = w[18];
  e->prev_now = w[19];
  e->n_last = w[20];
  e->type_last = w[21];
  e->last_mean_wait = f_of(w[22]);
  e->rate_est = f_of(w[23]);
  e->narr_since[0] = w[24];
  e->narr_since[1] = w[25];
  e->ndrop_since[0] = w[26];
  e->ndrop_since[1] = w[27];
  e->status = w[28];
  const uint32_t* p = w + ORC_HEADER_WORDS;
  for (uint32_t k = 0; k < e->K; ++k) {
    e->busy_until[k] = *p++;
    e->bsize[k] = *p++;
  }
  for (uint32_t k = 0; k < e->K; ++k)
    for (uint32_t t = 0; t < e->T; ++t) {
      e->qcnt[k][t] = *p++;
      e->qhead[k][t] = 0;
    }
  for (uint32_t k = 0; k < e->K; ++k)
    for (uint32_t t = 0; t < e->T; ++t) {
      memcpy(ring(e, k, t), p, e->cap * sizeof(uint32_t));
      p += e->cap;
    }
  if (e->c.cost_type >= 0) {
    for (uint32_t k = 0; k < e->K; ++k) {
      memcpy(e->qcost + (size_t)k * e->cap, p, e->cap * sizeof(uint32_t));
      p += e->cap;
    }
  }
}

int orc_rollout(const orc_config* c, const orc_mlp* m, uint64_t seed, int mode,
                const uint32_t* env_ids, int64_t n, int32_t H, float* obs, int32_t* action,
                float* logp, float* value, float* reward, uint8_t* done, int64_t* trace,
                uint32_t* final_state) {
  uint32_t D = orc_obs_dim(c);
  uint64_t SW = orc_state_words(c);
  float ob[256];
  float lg[512];
  for (int64_t i = 0; i < n; ++i) {
    orc_env* e = orc_env_new(c, env_ids[i], seed);
    if (!e) return 1;
    orc_env_reset(e);
    for (int32_t t = 0; t < H; ++t) {
      orc_step_out o;
      memset(&o, 0, sizeof(o));
      o.obs = ob;
      o.logits = lg;
      orc_env_step(e, m, mode, 0, &o);
      if (obs)
        for (uint32_t d = 0; d < D; ++d) obs[((int64_t)t * D + d) * n + i] = ob[d];
      if (action) action[(int64_t)t * n + i] = o.action;
      if (logp) logp[(int64_t)t * n + i] = o.logp;
      if (value) value[(int64_t)t * n + i] = o.value;
      if (reward) reward[(int64_t)t * n + i] = o.reward;
      if (done) done[(int64_t)t * n + i] = o.done;
      if (trace)
        for (int q = 0; q < 4; ++q) trace[((int64_t)t * 4 + q) * n + i] = o.trace[q];
    }
    if (final_state) orc_env_export(e, final_state + (uint64_t)i * SW);
    orc_env_free(e);
  }
  return 0;
}

/* ------------------------------------------------------------------------- */
/* Vectorised helpers for the pin tests (same code paths as the simulator).   */
/* ------------------------------------------------------------------------- */
void orc_map(int fn, const float* x, float* y, int64_t n) {
  for (int64_t i = 0; i < n; ++i) {
    switch (fn) {
      case 0: y[i] = orc_detlog(x[i]); break;
      case 1: y[i] = orc_detexp(x[i]); break;
      case 2: y[i] = orc_dettanh(x[i]); break;
      case 4: y[i] = orc_detgelu(x[i]); break;
      default: y[i] = orc_detcos2pi(x[i]); break;
    }
  }
}

/* Philox blocks for counters (idx0 + i, env, stream, 0), key = seed. */
void orc_philox_n(uint32_t idx0, uint32_t env, uint32_t stream, uint64_t seed, int64_t n,
                  uint32_t* out) {
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  for (int64_t i = 0; i < n; ++i) {
    uint32_t ctr[4] = {idx0 + (uint32_t)i, env, stream, 0u};
    orc_philox4x32_10(ctr, key, out + 4 * i);
  }
}

/* The samplers the simulator uses, applied to Philox blocks w [n][4]:
   kind 0: Exp(1) from word 0; kind 1: duration(scale * Exp(1)) from word 0;
   kind 2: standard normal from words 0, 1; kind 3: request type from word 1;
   kind 4: per-request cost of the cost type (config's cost model) from word 3. */
void orc_samplers(const orc_config* c, int kind, float scale, const uint32_t* w, int64_t n,
                  float* out) {
  orc_env e;
  memset(&e, 0, sizeof(e));
  e.c = *c;
  e.c.trace_type = NULL;
  e.c.trace_cost = NULL;
  e.T = c->n_types;
  for (int64_t i = 0; i < n; ++i) {
    const uint32_t* q = w + 4 * i;
    uint32_t t, cost;
    switch (kind) {
      case 0: out[i] = expo1(q[0]); break;
      case 1: out[i] = (float)orc_duration(scale * expo1(q[0])); break;
      case 2: out[i] = orc_normal(q[0], q[1]); break;
      case 3: request_attrs(&e, 0, q, &t, &cost); out[i] = (float)t; break;
      default: {
        uint32_t qq[4] = {q[0], (uint32_t)c->cost_type == 1u ? 0xFFFFFFFFu : 0u, q[2], q[3]};
        request_attrs(&e, 0, qq, &t, &cost);
        out[i] = (float)cost;
      }
    }
  }
}
