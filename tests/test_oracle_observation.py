"""Pins of the oracle's observation vector (Sec. 4.1's decision state), every feature of the
SINGLE and ROUTE layouts computed by hand on constructed states.

Each feature is (num x mul) / den in fp32 with the numerators, multipliers and denominators
of the layout (queue counts over the ring capacity, times over the 10 ms window, the arrival
rate as count x rate_scale / elapsed us, the last batch over 32, busy time over 100 ms, the
rate estimate over its reference, the diurnal phase over its period).  The expected values
below are that arithmetic on the hand-built state, so a swapped feature, a wrong index or
denominator, or the wrong head of line fails here.
"""
import numpy as np

import oracle
from paper_2607_05272_gb300 import workloads as W

f32 = np.float32
HDR = 32


def _env(cfg):
    e = oracle.OracleEnv(cfg, 0, 3)
    e.reset()
    s = np.zeros(e.SW, np.uint32)
    s[5] = 0xFFFFFFFF                     # no modulating switch pending
    s[21] = 0xFFFFFFFF                    # no previous batch type
    return e, s


def _rings(cfg, s, queues):
    """Servers (busy_until, b), counts K x T, then K x T rings of cap arrival times."""
    K, T, cap = cfg["n_servers"], cfg["n_types"], cfg["queue_cap"]
    cnt = HDR + 2 * K
    ring = cnt + K * T
    for (k, t), times in queues.items():
        s[cnt + k * T + t] = len(times)
        base = ring + (k * T + t) * cap
        s[base: base + len(times)] = times


def test_single_observation_c2_every_feature():
    cfg = W.c2(1)
    e, s = _env(cfg)
    now = 100_000
    s[0], s[19], s[18] = now, 96_000, 95_000          # now, previous decision, last dispatch
    s[2], s[3] = 9, now
    s[20], s[21] = 8, 1                                # n_last, type of the last batch
    s[22] = f32(2500.0).view(np.uint32)               # last batch's mean wait (us)
    s[24], s[25], s[26], s[27] = 3, 1, 1, 1            # arrivals / drops since, per type
    s[HDR + 1] = 8                                     # b of the server
    _rings(cfg, s, {(0, 0): [90_000, 99_000], (0, 1): [85_000]})
    s[12], s[13] = 5, 2
    e.load(s)
    o = e.observe()
    rs, tw, dt = f32(cfg["rate_scale"]), f32(10_000.0), f32(4000.0)
    want = [
        f32(2) / f32(256), f32(1) / f32(256),          # queue counts / capacity
        f32(5000) / tw,                                # time since the last dispatch
        0.0, 1.0,                                      # head of line: the type-1 request (85 ms)
        0.0,                                           # server free at a decision
        (f32(4) * rs) / dt,                            # arrival rate since the last decision
        f32(8) / f32(32),                              # last batch size / 32
        f32(10_000) / tw, f32(15_000) / tw,            # head-of-line waits per type
        (f32(3) * rs) / dt, (f32(1) * rs) / dt,        # per-type rates
        0.0, 1.0,                                      # last batch's type
        f32(2) / f32(32),                              # drops since / 32
        f32(2500.0) / tw,                              # last mean wait / window
    ]
    assert o.dtype == np.float32 and len(o) == 16
    assert np.array_equal(o.view(np.uint32), np.array(want, np.float32).view(np.uint32))


def test_single_observation_c1_empty_queue():
    cfg = W.c1(1)
    e, s = _env(cfg)
    s[0], s[19], s[18] = 7000, 7000, 1000              # dt = 0 counts as 1 us
    s[2], s[3] = 1, 7000
    s[24] = 2
    s[HDR + 1] = 8
    e.load(s)
    o = e.observe()
    want = [0.0, f32(6000) / f32(10_000), 0.0, 0.0, 0.0,
            (f32(2) * f32(cfg["rate_scale"])) / f32(1), 0.0, 0.0]
    assert np.array_equal(o.view(np.uint32), np.array(want, np.float32).view(np.uint32))


def test_route_observation_c4_every_feature():
    cfg = W.c4(1)
    e, s = _env(cfg)
    K, now = 8, 2_000_000
    s[0], s[9], s[10] = now, now, 1                    # the pending request is long
    s[2], s[3] = 40, now
    s[8] = 7                                           # the env's diurnal slot offset
    s[23] = f32(3000.0).view(np.uint32)               # EWMA arrival rate (req/s)
    busy = [0, now + 50_000, now - 5, now + 250_000, 0, 0, now + 1, 0]
    for k in range(K):
        s[HDR + 2 * k], s[HDR + 2 * k + 1] = busy[k], 4
    _rings(cfg, s, {(1, 0): [1_990_000, 1_995_000, 1_999_000], (3, 1): [1_900_000],
                    (6, 0): [1_999_999]})
    s[12] = 5
    e.load(s)
    o = e.observe()
    cap, bn = f32(256), f32(100_000.0)
    q = {(1, 0): 3, (3, 1): 1, (6, 0): 1}
    want = []
    for k in range(K):
        rem = max(busy[k] - now, 0)
        want += [f32(q.get((k, 0), 0)) / cap, f32(q.get((k, 1), 0)) / cap, f32(rem) / bn]
    want.append(f32(3000.0) / f32(8000.0))             # rate estimate / reference
    want += [0.0, 1.0]                                 # arriving type: long
    ph = (now + 7 * 500_000) % 60_000_000
    want.append(f32(ph) / f32(60_000_000))             # diurnal phase of the env's cycle
    assert len(o) == 28 == len(want)
    assert np.array_equal(o.view(np.uint32), np.array(want, np.float32).view(np.uint32))


def test_route_observation_c3_layout():
    cfg = W.c3(1)
    e, s = _env(cfg)
    now = 10_000
    s[0], s[9], s[10] = now, now, 0
    s[2], s[3] = 2, now
    s[23] = f32(4000.0).view(np.uint32)
    for k in range(4):
        s[HDR + 2 * k + 1] = 4
    s[HDR + 2 * 2] = now + 12_345
    _rings(cfg, s, {(0, 1): [9000, 9500], (2, 0): [1000]})
    s[12] = 4
    e.load(s)
    o = e.observe()
    cap = f32(256)
    want = [0.0, f32(2) / cap, 0.0, 0.0, 0.0, 0.0,
            f32(1) / cap, 0.0, f32(12_345) / f32(100_000.0), 0.0, 0.0, 0.0, 1.0]
    assert np.array_equal(o.view(np.uint32), np.array(want, np.float32).view(np.uint32))


def test_single_long_batch_reward_weight():
    """c2, Sec. 4.1 reward: a batch of the long type is charged the long type's 0.0001 per
    us of queueing (the paper's 10:1 ratio), and served in alpha_1 + beta_1 n."""
    cfg = W.c2(1)
    e, s = _env(cfg)
    now = 100_000
    s[0], s[19], s[18] = now, 96_000, 95_000
    s[2], s[3] = 9, now
    s[HDR + 1] = 8
    _rings(cfg, s, {(0, 0): [90_000], (0, 1): [85_000, 95_000]})
    s[12] = 3
    e.load(s)
    o = e.step(6, None, action=1 * 6 + 2)             # type 1, b = bsizes[2] = 4: takes both
    assert o["trace"][:3] == [now, 2, 15_000 + 5_000]
    assert o["reward"] == f32(2.0) - f32(0.0001) * f32(20_000.0)
    s2 = e.export()
    assert s2[HDR] == now + 20_000 + 2_000 * 2        # long: alpha 20 ms + 2 ms per request
    assert s2[21] == 1 and s2[20] == 2
    assert s2[22] == f32(10_000.0).view(np.uint32)    # last mean wait 20,000 / 2


def test_route_reward_counts_every_batch_until_the_next_arrival():
    """c3 router, Sec. 4.1 reward r = n - sum_type w_type W_type over the batches started
    between this decision and the next: a one-entry trace (gap 30 ms) fixes the next
    arrival at 80 ms.  The long request routed to idle server 1 (b = 1) starts at once
    (wait 0); server 0 frees at 60 ms and starts its two queued short requests (waits 20
    and 15 ms).  r = 3 - 0.001 * 35,000 - 0.0001 * 0."""
    cfg = W.c3(1)
    cfg.update(arrival_kind=W.ARR_TRACE, n_mod_states=1, accept_thr=[W.TWO24, W.TWO24],
               trace=(np.array([30_000], np.uint32), None, None), queue_cap=256)
    e, s = _env(cfg)
    K = 4
    now = 50_000
    s[0], s[9], s[10] = now, now, 1                    # pending: a long request at 50 ms
    s[2], s[3] = 5, now                                # next candidate: 50 ms + 30 ms
    s[23] = f32(4000.0).view(np.uint32)
    for k in range(K):
        s[HDR + 2 * k + 1] = 4
    s[HDR + 0] = 60_000                                # server 0 busy until 60 ms
    _rings(cfg, s, {(0, 0): [40_000, 45_000]})
    s[12] = 3
    e.load(s)
    o = e.step(6, None, action=1 * 4 + 0)              # server 1, b = bsizes[0] = 1
    assert o["trace"] == [now, 3, 35_000, 2]           # qafter: server 0's two, before 60 ms
    want = f32(3.0) - (f32(0.001) * f32(35_000.0) + f32(0.0001) * f32(0.0))
    assert o["reward"] == want
    s2 = e.export()
    assert s2[0] == 80_000 and s2[9] == 80_000         # the next decision: the next arrival
    assert s2[HDR + 0] == 60_000 + 1_000 + 50 * 2      # short batch of 2: alpha_0 + 2 beta_0
    assert s2[HDR + 2] == now + 20_000 + 2_000 * 1     # long batch of 1: alpha_1 + beta_1
    cnt = HDR + 2 * K
    assert list(s2[cnt: cnt + 2 * K]) == [0] * (2 * K)  # every queue empty
    assert s2[14] == 3                                 # dispatched
