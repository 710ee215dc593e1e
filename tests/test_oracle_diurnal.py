"""Pins of the oracle's diurnal x lognormal arrival process as a whole (Sec. 3.2: load
shaped like a production trace, with a daily cycle and bursts).

The process: within 500 ms epoch k of env e the arrivals are Poisson at rate
table[(k + o_e) mod n] x exp(sigma Z_k), o_e the env's slot offset from its INIT draw
and Z_k a standard normal per (env, epoch).  In ROUTE mode every decision is one arriving
request, so the routed requests' times give each env's arrival counts per epoch, and:

* sigma = 0: the count of (env, epoch) with slot s is Poisson with mean table[s] x 0.5 s,
  so the summed counts per slot are within 4 sd of M_s table[s] / 2 and the per-slot
  dispersion (variance / mean) is 1.  A wrong offset sign or slot index, a lost or doubled
  arrival at an epoch boundary, or a wrong time unit fails this on the steep table below.
* sigma > 0: the mean count is table[s] / 2 x exp(sigma^2 / 2) (the lognormal mean) and
  the variance is lam m + lam^2 (e^{sigma^2} - 1) e^{sigma^2}, lam = table[s] / 2, m the
  lognormal mean: a missing or doubled burst factor, or a factor per env instead of per
  epoch, moves one of the two.
* The offsets o_e are spread over all n slots (the envs sample the whole cycle).
"""
import math

import numpy as np

import oracle
from paper_2607_05272_gb300 import workloads as W

STATIC, INIT = 2, 4
TABLE = [20.0, 200.0, 60.0, 400.0]       # req/s per slot: a steep, asymmetric cycle
EPOCH = 500_000


def _cfg(sigma, E):
    c = W.c3(E)
    c.update(arrival_kind=W.ARR_DIURNAL, cand_mean_gap_us=0.0, epoch_us=EPOCH,
             diurnal_len=len(TABLE), diurnal_rate=TABLE + [0.0] * (128 - len(TABLE)),
             burst_sigma=sigma, queue_cap=4096, episode_len=1 << 20)
    return c


def _offset(env, seed, n):
    w = oracle.philox_n(0, env, INIT, seed, 1)[0]
    return ((int(w[1]) >> 8) * n) >> 24


def _counts(sigma, E=256, H=1200, seed=0xD1A1):
    """Per slot: the arrival counts of every fully observed (env, epoch)."""
    out = oracle.rollout(_cfg(sigma, E), None, seed, STATIC, list(range(E)), H)
    t = out["trace"][:, 0, :]                       # arrival time of each decision
    assert np.all(np.diff(t, axis=0) >= 0)
    per_slot = [[] for _ in TABLE]
    offs = []
    for e in range(E):
        o = _offset(e, seed, len(TABLE))
        offs.append(o)
        k = t[:, e] // EPOCH
        full = int(k[-1])                            # epochs 0 .. full-1 are complete
        c = np.bincount(k[k < full], minlength=full)
        for j in range(full):
            per_slot[(j + o) % len(TABLE)].append(c[j])
    return [np.asarray(p, np.float64) for p in per_slot], offs


def test_constant_rate_per_slot_is_poisson():
    per_slot, offs = _counts(0.0)
    for s, c in enumerate(per_slot):
        lam = TABLE[s] * EPOCH * 1e-6
        M = len(c)
        assert M > 200
        assert abs(c.sum() - M * lam) <= 4.0 * math.sqrt(M * lam), (s, c.mean(), lam)
        # dispersion of a Poisson count: var / mean = 1 (sd of the sample variance ratio
        # about sqrt(2 / M) for large lam)
        d = c.var(ddof=1) / c.mean()
        assert abs(d - 1.0) <= 4.0 * math.sqrt(2.0 / M + 1.0 / (M * lam)), (s, d)
    assert set(offs) == set(range(len(TABLE)))


def test_lognormal_burst_factor_mean_and_variance():
    sigma = 0.5
    m = math.exp(0.5 * sigma * sigma)
    v = (math.exp(sigma * sigma) - 1.0) * math.exp(sigma * sigma)
    per_slot, _ = _counts(sigma, E=384, seed=0xB0257)
    for s, c in enumerate(per_slot):
        lam = TABLE[s] * EPOCH * 1e-6
        M = len(c)
        mean, var = lam * m, lam * m + lam * lam * v
        assert abs(c.mean() - mean) <= 4.0 * math.sqrt(var / M), (s, c.mean(), mean)
        if lam >= 100:                               # the lam^2 term dominates: a factor
            got = c.var(ddof=1)                      # per env, or none, would move it
            assert 0.6 * var <= got <= 1.5 * var, (s, got, var)
