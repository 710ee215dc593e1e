"""The two-state MMPP of c2 (Sec. 3.2 bursty arrivals; c2's 300 / 3000 req/s with mean
dwell 200 ms in each state), pinned through the modulating chain itself.

The oracle logs its chain (the state at time 0, then the time and new state of every
switch it processes) while a c2 env is stepped under the Static policy, so every
sojourn is seen, none selected by when decisions happen:

* the state alternates at every switch (two states);
* the sojourn times S_i - S_{i-1} are exponential with mean 200,000 us: their mean
  within 4 standard errors (sd = mean for an exponential) and a Kolmogorov-Smirnov
  test against Exp(200,000 us);
* the arrivals each env admitted up to its current time match the rate integrated
  over the logged chain, rate(s) = candidate rate x accept_thr[s] / 2^24 (N(t) minus
  that integral is a martingale, so at the decision times its sum over envs has mean 0
  and variance equal to the summed integral): within 4 sd.

A wrong dwell scale, a fixed or uniform dwell, states that do not alternate, or the
two rates attached to the wrong states each fail one of these.
"""
import math

import numpy as np
import pytest

import oracle
from paper_2607_05272_gb300 import workloads as W

STATIC = 2
scipy_stats = pytest.importorskip("scipy.stats")


def _chain_run(env_id, n_switches, seed=0x5EED0002):
    cfg = W.c2(1)
    cfg["static_bi"] = 5   # batches of 32: fewer decisions per simulated second
    e = oracle.OracleEnv(cfg, env_id, seed)
    e.attach_switch_log(n_switches + 64)
    e.reset()
    while len(e.switch_log()) < n_switches + 1:
        for _ in range(200):
            e.step(STATIC, None)
    s = e.export()
    assert e.status() == 0
    return cfg, e.switch_log(), s


@pytest.fixture(scope="module")
def runs():
    return [_chain_run(env_id, 2000) for env_id in range(4)]


def test_chain_alternates(runs):
    for _, log, _ in runs:
        assert log[0, 0] == 0
        k = np.arange(len(log))
        assert np.array_equal(log[:, 1], log[0, 1] ^ (k & 1))
        assert np.all(np.diff(log[:, 0].astype(np.int64)) >= 0)


def test_sojourns_exponential_200ms(runs):
    gaps = np.concatenate([np.diff(log[:, 0].astype(np.float64)) for _, log, _ in runs])
    mean = 200000.0
    assert gaps.size >= 8000
    se = mean / math.sqrt(gaps.size)
    assert abs(gaps.mean() - mean) < 4.0 * se, (gaps.mean(), se)
    assert scipy_stats.kstest(gaps, "expon", args=(0.0, mean)).pvalue > 1e-3
    # exponential: sd equal to the mean (a uniform or fixed dwell of the same mean fails)
    assert abs(gaps.std() / mean - 1.0) < 0.05


def test_admitted_arrivals_follow_the_chain(runs):
    resid, var = 0.0, 0.0
    for cfg, log, s in runs:
        now = int(s[0])
        cand_rate = 1e6 / float(np.float32(cfg["cand_mean_gap_us"]))
        rate = [cand_rate * cfg["accept_thr"][k] / float(1 << 24) for k in (0, 1)]
        t = np.append(log[:, 0].astype(np.float64), np.inf)
        lam = 0.0
        for i in range(len(log)):
            lo, hi = t[i], min(t[i + 1], now)
            if hi > lo:
                lam += rate[int(log[i, 1])] * (hi - lo) * 1e-6
        resid += float(s[12]) - lam      # s[12]: requests arrived (admitted + dropped)
        var += lam
    assert abs(resid) < 4.0 * math.sqrt(var), (resid, math.sqrt(var))
