"""Pins of the oracle's event simulator (Sec. 3.1 dynamics, Sec. 3.2 workloads).

* M/D/1 and M/M/1 mean waiting time against the Pollaczek-Khinchine closed forms
  at fixed batch size 1 (the paper calls its Poisson workload M/M/1 traffic).
* The exact finite-horizon Little identity: the integral of the queue length equals
  the summed time requests spent queued, in integer microseconds.
* Request conservation after every step: arrived = dropped + dispatched + queued.
* The latency model L(b) = alpha + beta b and the reward on hand-built states.
* The two-state MMPP's long-run arrival rate.
* The Extreme Burst square wave: switch times exactly periodic, arrivals only in the
  high-rate phases, and their count against 100 req/s over those phases.
* Heterogeneous server speeds: batch times scaled by s/16 on hand-built states and in
  traces.
"""
import math

import numpy as np
import pytest

import oracle
from paper_2607_05272_gb300 import workloads as W

STATIC, RR, SQ, RANDOM, SAMPLE, EXTERNAL = 2, 3, 4, 5, 0, 6


def _mean_wait_per_env(cfg, H, warm, seed, n_envs):
    out = oracle.rollout(cfg, None, seed, STATIC, list(range(n_envs)), H)
    n = out["trace"][warm:, 1, :].astype(np.float64)   # dispatched (0 or 1)
    w = out["trace"][warm:, 2, :].astype(np.float64)   # their queueing microseconds
    return w.sum(0) / n.sum(0)


@pytest.mark.parametrize("lam", [200.0, 400.0])
def test_md1_mean_wait(lam):
    D = 2100.0
    rho = lam * D * 1e-6
    Wq = (lam * 1e-6) * D * D / (2.0 * (1.0 - rho))   # Pollaczek-Khinchine, deterministic service
    per_env = _mean_wait_per_env(W.md1(lam), 40000 if lam > 300 else 12000, 2000, 11, 96)
    est, se = per_env.mean(), per_env.std(ddof=1) / math.sqrt(per_env.size)
    assert abs(est - Wq) < 4.0 * se
    assert abs(est - Wq) < 0.03 * Wq


def test_mm1_mean_wait():
    lam, ms = 300.0, 2100.0
    mu = 1.0 / ms
    rho = lam * 1e-6 * ms
    Wq = rho / (mu - lam * 1e-6)                     # M/M/1 waiting time in queue
    per_env = _mean_wait_per_env(W.mm1(lam, ms), 30000, 2000, 13, 96)
    est, se = per_env.mean(), per_env.std(ddof=1) / math.sqrt(per_env.size)
    assert abs(est - Wq) < 4.0 * se
    assert abs(est - Wq) < 0.03 * Wq


def _policy_for(name):
    dims, hv = W.mlp_dims(name)
    Ws, bs = W.mlp_weights(dims, 7)
    return (Ws, bs, hv)


CASES = [("c1", W.c1(4), SAMPLE), ("c2", W.c2(4), SAMPLE), ("c3", W.c3(4), SAMPLE),
         ("c4", W.c4(4), SAMPLE), ("c3", W.c3(4), SQ), ("c2", W.c2(4), STATIC),
         ("c4", W.c4(4), RANDOM), ("c2t", W.c2t(4), SAMPLE), ("c2t", W.c2t(4), STATIC),
         ("c3t", W.c3t(4), SAMPLE), ("c3t", W.c3t(4), SQ)]


def _conserved(cfg, s):
    K, T, route = cfg["n_servers"], cfg["n_types"], cfg["mode"] == 1
    queued = int(s[32 + 2 * K: 32 + 2 * K + K * T].sum())
    arrived, dropped, dispatched = int(s[12]), int(s[13]), int(s[14])
    pending = 1 if route else 0
    return arrived == dropped + dispatched + queued + pending


@pytest.mark.parametrize("name,cfg,mode", CASES)
def test_conservation_and_little(name, cfg, mode):
    mlp = _policy_for(name) if mode == SAMPLE else None
    for env_id in (0, 3):
        e = oracle.OracleEnv(cfg, env_id, W.SEED[name])
        e.reset()
        H = 300
        for t in range(H):
            e.step(mode, mlp)
            s = e.export()
            assert _conserved(cfg, s)
            assert s[28] == 0  # no status flag
        s = e.export()
        area, waits = e.little(int(s[0]))
        assert area == waits
        assert area > 0


def test_latency_model_from_traces():
    """After a dispatch of n requests of type k with work still queued, the next decision
    comes exactly alpha_k + beta_k n later (single server)."""
    for name, cfg in (("c1", W.c1(8)), ("c2", W.c2(8))):
        out = oracle.rollout(cfg, _policy_for(name), W.SEED[name], SAMPLE, list(range(8)), 400)
        tr, act = out["trace"], out["action"]
        nb = cfg["n_bsizes"]
        checked = 0
        for t in range(399):
            for e in range(8):
                n, qafter = tr[t, 1, e], tr[t, 3, e]
                if n == 0:
                    continue
                k = act[t, e] // nb
                L = cfg["alpha_us"][k] + cfg["beta_us"][k] * n
                if qafter > 0:
                    assert tr[t + 1, 0, e] == tr[t, 0, e] + L
                    checked += 1
                else:
                    assert tr[t + 1, 0, e] >= tr[t, 0, e] + L
        assert checked > 100


def test_single_hand_scenario():
    """c1: queue [1000, 3000, 9000, 9500] at t = 10,000 us; action b = 2."""
    cfg = W.c1(1)
    e = oracle.OracleEnv(cfg, 0, 5)
    e.reset()
    s = np.zeros(e.SW, np.uint32)
    s[0] = 10000          # now
    s[2], s[3] = 5, 10000  # next candidate index, time of the last candidate
    s[5] = 0xFFFFFFFF
    s[21] = 0xFFFFFFFF     # no previous batch type
    s[23] = np.float32(800.0).view(np.uint32)
    s[19] = 8000           # previous decision
    base = 32 + 2 * 1
    s[33] = 8              # b of the server
    s[base] = 4            # queue length
    s[base + 1: base + 5] = [1000, 3000, 9000, 9500]
    s[12], s[14] = 4, 0    # arrived, dispatched
    e.load(s)
    o = e.step(EXTERNAL, None, action=1)   # batch size 2
    assert o["trace"][:3] == [10000, 2, 9000 + 7000]
    assert o["reward"] == np.float32(2.0) - np.float32(0.001) * np.float32(16000.0)
    assert o["obs"][0] == np.float32(4 / 128)
    assert o["obs"][7] == np.float32(9000 / 10000)   # head-of-line wait
    s2 = e.export()
    assert s2[32] == 10000 + 2000 + 100 * 2          # busy until: alpha + beta n
    assert s2[0] == 12200                             # next decision at completion
    assert list(s2[base + 1: base + 3]) == [9000, 9500]
    assert s2[20] == 2 and s2[18] == 10000            # n_last, time of last dispatch


def test_route_hand_scenario():
    """c3: a long request at t = 50,000 routed to idle server 0 with b = 16 starts at once;
    one routed to busy server 1 waits in its long queue."""
    cfg = W.c3(1)
    e = oracle.OracleEnv(cfg, 0, 5)
    e.reset()
    K, T, cap = 4, 2, 256
    s = np.zeros(e.SW, np.uint32)
    s[0] = 50000
    s[2], s[3] = 10, 50000
    s[5] = 0xFFFFFFFF
    s[9], s[10] = 50000, 1       # pending arrival: time, type long
    s[21] = 0xFFFFFFFF
    s[23] = np.float32(4000.0).view(np.uint32)
    srv = 32
    for k in range(K):
        s[srv + 2 * k + 1] = 4   # b_k
    s[srv + 2 * 1] = 60000       # server 1 busy until 60,000
    s[12] = 1
    e.load(s)
    o = e.step(EXTERNAL, None, action=0 * 4 + 2)   # server 0, b = 16
    s2 = e.export()
    busy0 = s2[srv + 0]
    assert busy0 == 50000 + 20000 + 2000 * 1       # alpha_long + beta_long * 1
    assert s2[srv + 1] == 16
    cnt = 32 + 2 * K
    assert s2[cnt + 0] == 0 and s2[cnt + 1] == 0   # server 0 queues empty
    assert o["trace"][1] >= 1                     # the batch was dispatched in this step
    assert o["obs"][0:3].tolist() == [0.0, 0.0, 0.0]
    assert o["obs"][5] == np.float32(10000 / 100000)  # server 1 busy remaining


def test_mmpp_long_run_rate():
    cfg = W.c2(32)
    out = oracle.rollout(cfg, None, 99, STATIC, list(range(32)), 6000)
    s = out["state"]
    rate = s[:, 12].astype(np.float64) / (s[:, 0].astype(np.float64) * 1e-6)
    per_env_mean = rate.mean()
    se = rate.std(ddof=1) / math.sqrt(rate.size)
    assert abs(per_env_mean - 1650.0) < 4.0 * se + 0.02 * 1650.0


def _burst_state_at(t, init, D):
    """Modulating state at time t of a square wave that starts in `init` and switches at
    every multiple of D (a candidate at a switch time sees the new state)."""
    return init ^ ((t // D) & 1)


def test_square_wave_switches_and_arrival_phases():
    """Extreme Burst: switch i is at exactly i D; every queued request arrived in a
    high-rate phase; the arrival count matches 100 req/s over the high phases only."""
    cfg = W.burst(6)
    D = int(cfg["dwell_mean_us"])
    expected = observed = 0.0
    for env_id in range(6):
        e = oracle.OracleEnv(cfg, env_id, 31)
        e.reset()
        s = e.export()
        init = int(s[6]) ^ ((int(s[4]) - 1) & 1)   # each processed switch toggled the state
        for _ in range(1500):
            assert s[5] == s[4] * D                            # S_i = i D exactly
            assert int(s[6]) == _burst_state_at(int(s[5]) - 1, init, D)
            q = int(s[34])
            for t in s[35:35 + q]:
                assert _burst_state_at(int(t), init, D) == 1   # only the 100 req/s state
            e.step(STATIC, None)
            s = e.export()
        now = int(s[0])
        high = sum(min(now, (p + 1) * D) - p * D
                   for p in range(now // D + 1) if p * D < now and _burst_state_at(p * D, init, D))
        expected += 100.0 * high * 1e-6
        observed += float(s[12])
    assert expected > 1000.0
    assert abs(observed - expected) < 4.0 * math.sqrt(expected) + 2.0


def test_server_speed_single_hand_scenario():
    """c1 with the server at speed 24/16: a batch of 2 takes (2200 x 24 + 8) / 16 = 3300 us."""
    cfg = W.c1(1)
    cfg["srv_speed16"] = [24, 0, 0, 0, 0, 0, 0, 0]
    e = oracle.OracleEnv(cfg, 0, 5)
    e.reset()
    s = np.zeros(e.SW, np.uint32)
    s[0] = 10000
    s[2], s[3] = 5, 10000
    s[5] = 0xFFFFFFFF
    s[21] = 0xFFFFFFFF
    s[23] = np.float32(800.0).view(np.uint32)
    s[19] = 8000
    base = 32 + 2 * 1
    s[33] = 8
    s[base] = 4
    s[base + 1: base + 5] = [1000, 3000, 9000, 9500]
    s[12], s[14] = 4, 0
    e.load(s)
    e.step(EXTERNAL, None, action=1)
    s2 = e.export()
    assert s2[32] == 10000 + 3300
    assert s2[0] == 13300


def test_server_speed_route_hand_scenario():
    """c3h-style speeds: a long request routed to idle server 0 at speed 40/16 runs
    (22000 x 40 + 8) / 16 = 55000 us; server 1 (busy) keeps its completion time."""
    cfg = W.c3(1)
    cfg["srv_speed16"] = [40, 32, 16, 16, 0, 0, 0, 0]
    e = oracle.OracleEnv(cfg, 0, 5)
    e.reset()
    K = 4
    s = np.zeros(e.SW, np.uint32)
    s[0] = 50000
    s[2], s[3] = 10, 50000
    s[5] = 0xFFFFFFFF
    s[9], s[10] = 50000, 1
    s[21] = 0xFFFFFFFF
    s[23] = np.float32(4000.0).view(np.uint32)
    srv = 32
    for k in range(K):
        s[srv + 2 * k + 1] = 4
    s[srv + 2 * 1] = 60000
    s[12] = 1
    e.load(s)
    e.step(EXTERNAL, None, action=0 * 4 + 2)
    s2 = e.export()
    assert s2[srv + 0] == 50000 + 55000
    assert s2[srv + 2] == 60000


def test_server_speed_latency_from_traces():
    """With speed s/16 the next decision after a dispatch with work still queued comes
    exactly (L s + 8) / 16 later, L = alpha_k + beta_k n."""
    cfg = W.c2(8)
    cfg["srv_speed16"] = [21, 0, 0, 0, 0, 0, 0, 0]
    out = oracle.rollout(cfg, _policy_for("c2"), W.SEED["c2"], SAMPLE, list(range(8)), 300)
    tr, act = out["trace"], out["action"]
    nb = cfg["n_bsizes"]
    checked = 0
    for t in range(299):
        for e in range(8):
            n, qafter = int(tr[t, 1, e]), int(tr[t, 3, e])
            if n == 0 or qafter == 0:
                continue
            k = act[t, e] // nb
            L = cfg["alpha_us"][k] + cfg["beta_us"][k] * n
            assert tr[t + 1, 0, e] == tr[t, 0, e] + (L * 21 + 8) // 16
            checked += 1
    assert checked > 100


def test_wait_action_layout_hand_scenario():
    """c1w (Sec. 4.1 action space): from queue [1000, 3000, 9000, 9500] at t = 10,000 us,
    action 0 waits (nothing dispatched, reward 0, queue kept, next decision later), and
    action 3 dispatches a batch of 3 (waits 9000 + 7000 + 1000 us)."""
    cfg = W.c1w(1)
    def state():
        s = np.zeros(oracle.OracleEnv(cfg, 0, 5).SW, np.uint32)
        s[0] = 10000
        s[2], s[3] = 5, 10000
        s[5] = 0xFFFFFFFF
        s[21] = 0xFFFFFFFF
        s[23] = np.float32(800.0).view(np.uint32)
        s[19] = 8000
        s[33] = 8
        s[34] = 4
        s[35:39] = [1000, 3000, 9000, 9500]
        s[12], s[14] = 4, 0
        return s
    e = oracle.OracleEnv(cfg, 0, 5)
    e.reset()
    e.load(state())
    o = e.step(EXTERNAL, None, action=0)
    assert o["trace"][1] == 0 and o["reward"] == 0.0
    s2 = e.export()
    assert s2[14] == 0                                   # nothing dispatched
    assert s2[0] > 10000                                 # the next decision is at an arrival
    assert list(s2[35:39]) == [1000, 3000, 9000, 9500]   # the queue is kept, in order
    e2 = oracle.OracleEnv(cfg, 0, 5)
    e2.reset()
    e2.load(state())
    o2 = e2.step(EXTERNAL, None, action=3)
    assert o2["trace"][:3] == [10000, 3, 9000 + 7000 + 1000]
    s3 = e2.export()
    assert s3[32] == 10000 + 2000 + 100 * 3
    assert list(s3[35:36]) == [9500]
