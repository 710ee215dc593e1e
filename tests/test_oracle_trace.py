"""Pins of the oracle's trace replay input (Sec. 3.2 replays real-world request traces).

* Exact replay: in ROUTE mode every decision is one arriving request, so the pending
  request's time, type and cost walk the trace's cumulative gaps from the env's starting
  entry floor(u n / 2^32) (u the third word of its INIT draw), through several wraps.
* Thinning on a trace keeps exactly the candidates whose ARRIVAL draw passes the
  threshold; the kept requests are that subsequence of the trace.
* D/D/1 closed forms on a one-entry trace (deterministic arrivals every g us, batch 1):
  with g above the 2100 us service every request is served on arrival (no wait, reward
  1 per decision); with g = 1000 us request k starts at 1000 + 2100 (k - 1) and waits
  1100 (k - 1) us.
(Conservation and the Little identity on the trace workloads are with the other
workloads' in the queueing pins.)
"""
import numpy as np
import pytest

import oracle
from paper_2607_05272_gb300 import workloads as W

STATIC, EXTERNAL = 2, 6
INIT, ARRIVAL = 4, 1


def _start(env, seed, n):
    w = oracle.philox_n(0, env, INIT, seed, 1)[0]
    return (int(w[2]) * n) >> 32


def _route_cfg(trace, **kw):
    c = W.c3(1)
    c.update(arrival_kind=W.ARR_TRACE, n_mod_states=1, accept_thr=[W.TWO24, W.TWO24],
             cost_type=1, cost_kind=1, cost_scale_us=8000.0, trace=trace, queue_cap=4096)
    c.update(kw)
    return c


def test_route_replays_the_trace_exactly():
    gap = np.array([5, 0, 12, 3, 100, 7, 1], np.uint32)
    typ = np.array([0, 1, 1, 0, 5, 0, 1], np.uint8)     # 5 counts as the last type (1)
    cost = np.array([11, 22, 33, 44, 55, 66, 77], np.uint32)
    n = len(gap)
    for env, seed in ((0, 3), (1, 3), (17, 99), (4, 0xABCDEF)):
        e = oracle.OracleEnv(_route_cfg((gap, typ, cost)), env, seed)
        e.reset()
        o = _start(env, seed, n)
        t = 0
        for k in range(3 * n + 2):
            i = (o + k) % n
            t += int(gap[i])
            ty = min(int(typ[i]), 1)
            s = e.export()
            assert s[9] == t and s[10] == ty             # pending request time and type
            assert s[11] == (cost[i] if ty == 1 else 0)  # its cost (cost type 1 only)
            assert s[2] == o + k + 1                     # candidate counter
            e.step(EXTERNAL, None, action=k % 4 * 4)     # route to a server, batch 1
        assert e.status() == 0


def test_route_trace_without_types_or_costs_draws_them():
    """A trace of gaps only: types and costs are drawn as for generated arrivals."""
    gap = np.full(5, 40, np.uint32)
    cfg = _route_cfg((gap, None, None), type0_thr=W._thr(0.7))
    env, seed = 2, 7
    e = oracle.OracleEnv(cfg, env, seed)
    e.reset()
    o = _start(env, seed, 5)
    words = oracle.philox_n(o, env, ARRIVAL, seed, 40)
    for k in range(40):
        s = e.export()
        assert s[9] == 40 * (k + 1)
        assert s[10] == (1 if (int(words[k][1]) >> 8) >= cfg["type0_thr"] else 0)
        e.step(EXTERNAL, None, action=0)


def test_thinned_trace_keeps_the_passing_candidates():
    rng = np.random.default_rng(4)
    n = 257
    gap = rng.integers(0, 50, n).astype(np.uint32)
    typ = rng.integers(0, 2, n).astype(np.uint8)
    thr = 1 << 23
    cfg = _route_cfg((gap, typ, None), accept_thr=[thr, thr])
    env, seed = 5, 21
    e = oracle.OracleEnv(cfg, env, seed)
    e.reset()
    o = _start(env, seed, n)
    words = oracle.philox_n(o, env, ARRIVAL, seed, 3 * n)
    t = 0
    kept = []
    for j in range(3 * n):
        t += int(gap[(o + j) % n])
        if (int(words[j][2]) >> 8) < thr:
            kept.append((t, int(typ[(o + j) % n])))
    for k in range(len(kept) - 1):
        s = e.export()
        assert (int(s[9]), int(s[10])) == kept[k]
        e.step(EXTERNAL, None, action=0)
    assert 0.4 < len(kept) / (3 * n) < 0.6


def _dd1_cfg(g):
    return W._base(n_envs=1, arrival_kind=W.ARR_TRACE, static_bi=0, queue_cap=4096,
                   episode_len=1 << 30, trace=(np.array([g], np.uint32), None, None))


def test_dd1_underloaded_serves_every_request_on_arrival():
    H = 200
    out = oracle.rollout(_dd1_cfg(5000), None, 9, STATIC, [0], H)
    tr = out["trace"][:, :, 0]
    assert np.array_equal(tr[:, 0], 5000 * np.arange(1, H + 1))   # decision times
    assert np.all(tr[:, 1] == 1) and np.all(tr[:, 2] == 0)       # one request, no wait
    assert np.all(out["reward"][:, 0] == np.float32(1.0))


def test_dd1_overloaded_waits_grow_linearly():
    H = 100
    out = oracle.rollout(_dd1_cfg(1000), None, 9, STATIC, [0], H)
    tr = out["trace"][:, :, 0]
    k = np.arange(1, H + 1)
    assert np.array_equal(tr[:, 0], 1000 + 2100 * (k - 1))
    assert np.all(tr[:, 1] == 1)
    assert np.array_equal(tr[:, 2], 1100 * (k - 1))
    assert out["state"][0][13] == 0   # nothing dropped


def test_trace_from_timestamps_round_trip():
    t = np.array([1000.0, 1000.0, 1250.4, 1300.0, 9000.0])
    gap, typ, cost = W.trace_from_timestamps(t, [0, 1, 3, 1, 0], [5.0, 6.4, 7.5, 0.0, 1e3])
    assert list(gap[1:]) == [0, 250, 50, 7700]            # t rounded to us, then differenced
    assert gap[0] == 2000                                   # wrap gap: the mean gap (8000 / 4)
    assert np.array_equal(np.cumsum(gap[1:]), np.rint(t[1:] - t[0]))
    assert list(typ) == [0, 1, 3, 1, 0] and list(cost) == [5, 6, 8, 0, 1000]
    g2, _, _ = W.trace_from_timestamps(t, wrap_gap_us=123)
    assert g2[0] == 123
    with pytest.raises(ValueError):
        W.trace_from_timestamps([3.0, 1.0])


def test_trace_from_csv(tmp_path):
    p = tmp_path / "log.csv"
    p.write_text("ts,model,out_tokens\n0.5,big,10\n0.1,small,3\n0.25,small,4\n")
    gap, typ, cost = W.trace_from_csv(p, "ts", 1e6, "model", {"small": 0, "big": 1},
                                      "out_tokens", 20000.0)
    assert list(gap[1:]) == [150000, 250000] and gap[0] == 200000
    assert list(typ) == [0, 0, 1] and list(cost) == [60000, 80000, 200000]
    # the oracle replays it: the first pending request is entry o's gap away
    cfg = _route_cfg((gap, typ, cost))
    e = oracle.OracleEnv(cfg, 0, 3)
    e.reset()
    o = _start(0, 3, 3)
    assert e.export()[9] == gap[o]
