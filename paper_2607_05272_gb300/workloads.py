"""Seeded synthetic inputs shared by the CUDA path, the oracle and the benchmark.

This module holds only workload *inputs*: the five environment configurations the
engine is measured on, policy weights, the diurnal rate table and minibatch
permutations.  It contains none of the method's arithmetic (no simulation, policy,
return or loss code), so both sides can take their inputs from here.

The configurations restate the paper's workloads (Sec. 3.2: Poisson, bursty,
trace-shaped, heterogeneous multi-server) and latency model (Sec. 3.1,
L = alpha + beta * b) at the sizes of the engine's five benchmark configurations:

* ``c1``  64 envs x 10,000 steps, one server, one type, Poisson 800 req/s,
  2000 + 100 n us, queue 128, batch sizes {1,2,4,8,16,32}, MLP 8-32-6, REINFORCE.
* ``c2``  4096 envs x 512, one server, two-state MMPP 300 / 3000 req/s (dwell
  200 ms), 80/20 short (1000 + 50 n) / long (20,000 + 2000 n), queues 256,
  action (type, batch), MLP 16-64-64-12, REINFORCE with a mean baseline.
* ``c3``  16,384 envs x 256, four servers, Poisson 4000 req/s, 70/30 mix,
  action (server, batch in {1,4,16,32}), MLP 13-128-128-16 + value, PPO/GAE.
* ``c4``  65,536 envs x 512, eight servers, diurnal 1000-8000 req/s over 60 s x
  lognormal(0, 1) per 500 ms, long requests with Pareto(1.5, 10 ms) per-request
  cost, 85/15 mix, MLP 28-256-256-48 + value, PPO/GAE.
* ``c5``  c3's environment at 1024 ... 1,048,576 envs x 1024, argmax policy.

The public Azure Functions / BurstGPT traces the paper replays are not available
here; ``c4``'s diurnal x lognormal x Pareto load stands in for them.
"""
from __future__ import annotations

import math

import numpy as np

ABI_VERSION = 5
MODE_SINGLE, MODE_ROUTE = 0, 1
ARR_THINNED, ARR_DIURNAL, ARR_TRACE = 0, 1, 2
POLICY = {"sample": 0, "argmax": 1, "static": 2, "rr": 3, "sq": 4, "random": 5, "external": 6}
TWO24 = 1 << 24

# Field order of the configuration record (same order as the C struct).
CONFIG_FIELDS = [
    ("abi_version", "u32"), ("mode", "u32"), ("n_envs", "u32"), ("n_servers", "u32"),
    ("n_types", "u32"), ("queue_cap", "u32"), ("episode_len", "u32"), ("arrival_kind", "u32"),
    ("cand_mean_gap_us", "f32"), ("n_mod_states", "u32"), ("accept_thr", "u32[2]"),
    ("dwell_mean_us", "f32"), ("epoch_us", "u32"), ("diurnal_len", "u32"),
    ("diurnal_rate", "f32[128]"), ("burst_sigma", "f32"), ("type0_thr", "u32"),
    ("alpha_us", "u32[2]"), ("beta_us", "u32[2]"), ("cost_type", "i32"), ("cost_kind", "u32"),
    ("cost_scale_us", "f32"), ("pareto_inv_alpha", "f32"), ("w_wait", "f32[2]"),
    ("n_bsizes", "u32"), ("bsizes", "u32[8]"), ("static_bi", "u32"), ("obs_extra", "u32"),
    ("obs_dim", "u32"), ("t_window_us", "f32"), ("rate_scale", "f32"), ("rate_ref", "f32"),
    ("busy_norm_us", "f32"), ("phase_period_us", "u32"), ("dwell_kind", "u32"),
    ("srv_speed16", "u32[8]"), ("action_layout", "u32"),
]


def _thr(p: float) -> int:
    """Probability as an integer threshold out of 2^24 (rounded to nearest)."""
    return int(round(p * TWO24))


def diurnal_table(n: int = 120, lo: float = 1000.0, hi: float = 8000.0) -> list:
    """Base arrival rate per 500 ms slot of a 60 s period: a sinusoid from lo to hi.

    This is workload input, like a trace file: computed once in fp64 and stored as fp32.
    """
    mid, amp = 0.5 * (lo + hi), 0.5 * (hi - lo)
    return [float(np.float32(mid + amp * math.sin(2.0 * math.pi * i / n))) for i in range(n)]


def _base(**kw) -> dict:
    c = dict(
        abi_version=ABI_VERSION, mode=MODE_SINGLE, n_envs=64, n_servers=1, n_types=1,
        queue_cap=128, episode_len=1000, arrival_kind=ARR_THINNED,
        cand_mean_gap_us=1250.0, n_mod_states=1, accept_thr=[TWO24, TWO24],
        dwell_mean_us=0.0, epoch_us=0, diurnal_len=1, diurnal_rate=[0.0] * 128,
        burst_sigma=0.0, type0_thr=TWO24, alpha_us=[2000, 0], beta_us=[100, 0],
        cost_type=-1, cost_kind=0, cost_scale_us=0.0, pareto_inv_alpha=0.0,
        w_wait=[0.001, 0.0], n_bsizes=6, bsizes=[1, 2, 4, 8, 16, 32, 0, 0], static_bi=3,
        obs_extra=0, obs_dim=8, t_window_us=10000.0, rate_scale=1250.0, rate_ref=800.0,
        busy_norm_us=100000.0, phase_period_us=0, dwell_kind=0, srv_speed16=[0] * 8,
        action_layout=0,
    )
    c.update(kw)
    return c


def c1(n_envs: int = 64) -> dict:
    """Tiny single-server env: Poisson 800 req/s, 2000 + 100 n us, queue 128."""
    return _base(n_envs=n_envs)


def c2(n_envs: int = 4096) -> dict:
    """Single-server bursty heterogeneous env: MMPP 300/3000 req/s, 80/20 short/long."""
    return _base(
        n_envs=n_envs, n_types=2, queue_cap=256, episode_len=512,
        cand_mean_gap_us=float(np.float32(1e6 / 3000.0)), n_mod_states=2,
        accept_thr=[_thr(300.0 / 3000.0), TWO24], dwell_mean_us=200000.0,
        type0_thr=_thr(0.8), alpha_us=[1000, 20000], beta_us=[50, 2000],
        w_wait=[0.001, 0.0001], obs_extra=1, obs_dim=16,
        rate_scale=float(np.float32(1e6 / 1650.0)), rate_ref=1650.0,
    )


def c3(n_envs: int = 16384, episode_len: int = 256) -> dict:
    """Multi-server routing env: 4 servers, Poisson 4000 req/s, 70/30 short/long."""
    return _base(
        mode=MODE_ROUTE, n_envs=n_envs, n_servers=4, n_types=2, queue_cap=256,
        episode_len=episode_len, cand_mean_gap_us=250.0, type0_thr=_thr(0.7),
        alpha_us=[1000, 20000], beta_us=[50, 2000], w_wait=[0.001, 0.0001],
        n_bsizes=4, bsizes=[1, 4, 16, 32, 0, 0, 0, 0], static_bi=2, obs_dim=13,
        rate_scale=0.0, rate_ref=4000.0,
    )


def c4(n_envs: int = 65536) -> dict:
    """Trace-shaped env: 8 servers, diurnal x lognormal arrivals, Pareto long costs."""
    tab = diurnal_table()
    return _base(
        mode=MODE_ROUTE, n_envs=n_envs, n_servers=8, n_types=2, queue_cap=256,
        episode_len=512, arrival_kind=ARR_DIURNAL, cand_mean_gap_us=0.0,
        epoch_us=500000, diurnal_len=len(tab), diurnal_rate=tab + [0.0] * (128 - len(tab)),
        burst_sigma=1.0, type0_thr=_thr(0.85), alpha_us=[1000, 20000], beta_us=[50, 0],
        cost_type=1, cost_kind=0, cost_scale_us=10000.0,
        pareto_inv_alpha=float(np.float32(1.0 / 1.5)), w_wait=[0.001, 0.0001],
        obs_extra=1, obs_dim=28, rate_scale=0.0, rate_ref=8000.0, phase_period_us=60_000_000,
    )


def c5(n_envs: int = 65536) -> dict:
    """Scale sweep of c3's env: horizon 1024, one segment per rollout."""
    return c3(n_envs=n_envs, episode_len=1024)


def md1(lam: float, n_envs: int = 64) -> dict:
    """c1 with fixed batch 1 (M/D/1, D = 2100 us) at arrival rate lam req/s."""
    return _base(n_envs=n_envs, cand_mean_gap_us=float(np.float32(1e6 / lam)), static_bi=0,
                 queue_cap=4096, episode_len=1 << 30)


def mm1(lam: float, mean_service_us: float = 2100.0, n_envs: int = 64) -> dict:
    """Single server, batch 1, exponential per-request cost (M/M/1)."""
    return _base(n_envs=n_envs, cand_mean_gap_us=float(np.float32(1e6 / lam)), static_bi=0,
                 queue_cap=4096, episode_len=1 << 30, alpha_us=[0, 0], beta_us=[0, 0],
                 cost_type=0, cost_kind=1, cost_scale_us=float(mean_service_us))


def burst(n_envs: int = 64) -> dict:
    """Extreme Burst (Sec. 3.2): c1's server under a square wave between 0 and 100 req/s.

    The paper switches "every 200 steps"; here the rate switches every 2 s of simulated
    time (200 steps at the high rate's 10 ms mean gap) through the modulating chain with a
    fixed dwell: candidates at 100/s, all kept in the high state and none in the low one.
    """
    return _base(n_envs=n_envs, cand_mean_gap_us=10000.0, n_mod_states=2,
                 accept_thr=[0, TWO24], dwell_mean_us=2_000_000.0, dwell_kind=1,
                 rate_scale=10000.0, rate_ref=100.0)


def c3h(n_envs: int = 16384) -> dict:
    """Heterogeneous multi-GPU routing (Sec. 3.1 K heterogeneous GPUs, Sec. 3.2 Multi-GPU
    Routing): c3's router with a 50/50 fast/slow request mix over two full-speed servers
    and two at half speed (batch times x 2)."""
    c = c3(n_envs)
    c.update(type0_thr=_thr(0.5), srv_speed16=[16, 16, 32, 32, 0, 0, 0, 0])
    return c


def c1w(n_envs: int = 64) -> dict:
    """c1 with the paper's action space (Sec. 4.1): action 0 waits, actions 1..32 dispatch
    a batch of that size (33 actions)."""
    return _base(n_envs=n_envs, action_layout=1, n_bsizes=32, static_bi=7)


def c2w(n_envs: int = 4096) -> dict:
    """c2 with Wait plus (type, batch size 1..32): 65 actions (Sec. 4.1)."""
    c = c2(n_envs)
    c.update(action_layout=1, n_bsizes=32, static_bi=7)
    return c


def synthetic_trace(n: int, seed: int, mean_gap_us: float = 300.0, cv: float = 2.0,
                    p_long: float = 0.2, stay: float = 0.9, cost_median_us: float = 8000.0,
                    cost_sigma: float = 1.0):
    """A seeded request trace of n entries in the trace replay format (gap_us u32,
    type u8, cost_us u32), shaped like an LLM serving log of the BurstGPT kind: Gamma
    inter-arrival gaps with coefficient of variation `cv` (bursty when cv > 1), request
    types from a two-state chain that stays on its type with probability `stay` (runs of
    one model; a fraction `p_long` of long requests overall), and lognormal per-request
    costs (response-length shaped).  Synthetic: no real trace is reproduced."""
    rng = np.random.default_rng(seed)
    k = 1.0 / (cv * cv)
    gap = np.rint(rng.gamma(k, mean_gap_us / k, n)).astype(np.uint32)
    # chain with stationary P(long) = p_long: P(short -> long) = (1 - stay) p_long / (1 - p_long)
    # scaled so that both switch rates stay in [0, 1]
    a = (1.0 - stay) * min(1.0, p_long / (1.0 - p_long))
    b = a * (1.0 - p_long) / p_long
    u = rng.random(n)
    typ = np.zeros(n, np.uint8)
    t = 1 if rng.random() < p_long else 0
    for i in range(n):
        typ[i] = t
        if u[i] < (b if t else a):
            t ^= 1
    cost = np.rint(cost_median_us * np.exp(cost_sigma * rng.standard_normal(n)))
    cost = np.minimum(cost, 2.0 ** 26).astype(np.uint32)
    return gap, typ, cost


def trace_from_timestamps(t_us, types=None, costs_us=None, wrap_gap_us=None):
    """The trace format of sim_set_trace from absolute request timestamps (sorted, in us):
    gap_i = t_i - t_{i-1} for i >= 1 and gap_0 = the gap taken when the replay wraps from
    the last entry to the first (default: the mean gap).  Types (values >= n_types count as
    the last type) and per-request costs in us pass through; rounding to whole us and
    clamping to u32 / u8 are the only changes."""
    t = np.asarray(t_us, dtype=np.float64)
    if t.ndim != 1 or len(t) < 1:
        raise ValueError("need a non-empty 1-D array of timestamps")
    if np.any(np.diff(t) < 0):
        raise ValueError("timestamps must be sorted")
    t = np.rint(t - t[0])
    gap = np.empty(len(t), np.float64)
    gap[1:] = np.diff(t)
    if wrap_gap_us is None:
        wrap_gap_us = t[-1] / (len(t) - 1) if len(t) > 1 else 1.0
    gap[0] = np.rint(wrap_gap_us)
    gap = np.clip(gap, 0, 2 ** 32 - 1).astype(np.uint32)
    typ = None if types is None else np.clip(np.asarray(types), 0, 255).astype(np.uint8)
    cost = None if costs_us is None else np.clip(np.rint(np.asarray(costs_us, np.float64)), 0,
                                                 2 ** 32 - 1).astype(np.uint32)
    for a in (typ, cost):
        if a is not None and len(a) != len(gap):
            raise ValueError("types and costs need one entry per timestamp")
    return gap, typ, cost


def trace_from_csv(path, time_col, time_unit_us=1.0, type_col=None, type_map=None,
                   cost_col=None, cost_unit_us=1.0, wrap_gap_us=None, delimiter=","):
    """A trace from a CSV request log with a header row (for instance a user's copy of a
    serving log): the timestamp column (seconds -> time_unit_us = 1e6), an optional type
    column mapped through `type_map` (a dict from the column's strings to type numbers, or
    numeric types when None) and an optional cost column (scaled by cost_unit_us, e.g. a
    token count times the us per token).  Rows are sorted by time."""
    import csv
    with open(path, newline="") as f:
        rows = list(csv.DictReader(f, delimiter=delimiter))
    if not rows:
        raise ValueError("no rows in %s" % path)
    t = np.array([float(r[time_col]) * time_unit_us for r in rows])
    order = np.argsort(t, kind="stable")
    typ = None
    if type_col is not None:
        raw = [rows[i][type_col] for i in order]
        typ = [type_map[v] if type_map is not None else int(float(v)) for v in raw]
    cost = None
    if cost_col is not None:
        cost = [float(rows[i][cost_col]) * cost_unit_us for i in order]
    return trace_from_timestamps(t[order], typ, cost, wrap_gap_us)


def c2t(n_envs: int = 4096) -> dict:
    """Trace replay (Sec. 3.2 real-world traces) on c2's server: every arrival, its gap
    and its type come from a 100,000-entry synthetic BurstGPT-shaped trace (mean gap
    600 us, CV 2, 20 % long requests in runs); each env starts at its own entry."""
    c = c2(n_envs)
    c.update(arrival_kind=ARR_TRACE, n_mod_states=1, accept_thr=[TWO24, TWO24],
             trace=synthetic_trace(100_000, 0x7ACE0002, mean_gap_us=600.0))
    return c


def c3t(n_envs: int = 16384) -> dict:
    """Trace replay on c3's 4-server router: gaps, types and the long requests' costs
    (batch time alpha + the sum of its requests' costs) from a synthetic trace (mean gap
    250 us, CV 2, 30 % long, lognormal costs with median 8 ms)."""
    c = c3(n_envs)
    c.update(arrival_kind=ARR_TRACE, n_mod_states=1, accept_thr=[TWO24, TWO24],
             cost_type=1, cost_kind=1, cost_scale_us=8000.0, beta_us=[50, 0],
             trace=synthetic_trace(100_000, 0x7ACE0003, mean_gap_us=250.0, p_long=0.3))
    return c


def c3s(n_envs: int = 4096) -> dict:
    """Multi-GPU Routing (Heterogeneous) of Sec. 3.2, the setting of the segregation
    result of Sec. 5: two servers, Poisson 60 req/s, a 50/50 mix of fast and slow
    requests with the paper's V100 batch times (alpha 2 ms; beta 5 ms fast, 20 ms slow),
    batch sizes {1, 2, 4, 8} per server, and an observation that includes the arriving
    request's type (obs_extra), which segregation needs."""
    return _base(mode=MODE_ROUTE, n_envs=n_envs, n_servers=2, n_types=2, queue_cap=256,
                 episode_len=256, cand_mean_gap_us=float(np.float32(1e6 / 60.0)),
                 type0_thr=_thr(0.5), alpha_us=[2000, 2000], beta_us=[5000, 20000],
                 w_wait=[0.001, 0.0001], n_bsizes=4, bsizes=[1, 2, 4, 8, 0, 0, 0, 0],
                 static_bi=0, obs_extra=1, obs_dim=10, rate_scale=0.0, rate_ref=60.0,
                 phase_period_us=60_000_000)


def c1p(n_envs: int = 64) -> dict:
    """c1w's env and action space, served by the paper's policy network (Sec. 4.2; the
    network is described at ``PAPER_NET``)."""
    return c1w(n_envs)


CONFIGS = {"c1": c1, "c2": c2, "c3": c3, "c4": c4, "c5": c5, "burst": burst, "c3h": c3h,
           "c1w": c1w, "c2w": c2w, "c1p": c1p, "c2t": c2t, "c3t": c3t, "c3s": c3s}

# Policy network shapes (input, hidden..., actions) and whether a value row follows.
MLP_SHAPES = {
    "c1": ([8, 32, 6], False),
    "c2": ([16, 64, 64, 12], False),
    "c3": ([13, 128, 128, 16], True),
    "c4": ([28, 256, 256, 48], True),
    "c5": ([13, 128, 128, 16], True),
    "burst": ([8, 32, 6], False),
    "c3h": ([13, 128, 128, 16], True),
    "c1w": ([8, 32, 33], False),
    "c2w": ([16, 64, 64, 65], False),
    "c1p": ([8, 4, 4, 4, 128, 33], True),
    "c2t": ([16, 64, 64, 12], False),
    "c3t": ([13, 128, 128, 16], True),
    "c3s": ([10, 128, 128, 8], True),
}

# The paper's network (Sec. 4.2) as a plain MLP.  The 8-dim state is projected to a
# 4-dim embedding; self-attention (2 heads, embedding 4) then sees that single token, so
# its softmax weight is 1 and it returns the output projection of the value projection:
# two linear 4 -> 4 maps (query and key projections do not reach the output).  The
# policy head (4 -> 64 GELU -> 33 logits) and the value head (4 -> 64 GELU -> 1) become
# one 4 -> 128 GELU layer and a 128 -> 34 output layer whose logit rows read hidden
# units 0..63 and whose value row reads 64..127; the other entries start at zero
# (a trainer that keeps the heads separate leaves them there by masking their gradient).
PAPER_NET = ("c1p",)

# Policies whose value head is a separate network (Sec. 4.2), as one MLP: every layer
# after the first is block-diagonal between a policy tower (the first half of the hidden
# units) and a value tower (the second half), and the value row reads only the value
# tower.  A value row on a shared trunk let the value loss (returns of order -200 on c3s)
# drown the policy gradient; separate towers learn.
TWO_TOWER = ("c3s",)

# Activation after each hidden layer where it is not tanh (simx_act names).
MLP_ACTS = {"c1p": ["identity", "identity", "identity", "gelu"]}

HORIZON = {"c1": 10000, "c2": 512, "c3": 256, "c4": 512, "c5": 1024, "burst": 2000, "c3h": 256,
           "c1w": 2000, "c2w": 512, "c1p": 2000, "c2t": 512, "c3t": 256, "c3s": 256}
SEED = {name: 0x5EED0000 + i + 1
        for i, name in enumerate(["c1", "c2", "c3", "c4", "c5", "burst", "c3h", "c1w", "c2w", "c1p",
                                  "c2t", "c3t", "c3s"])}


def mlp_dims(name: str) -> tuple:
    dims, has_value = MLP_SHAPES[name]
    dims = list(dims)
    if has_value:
        dims[-1] += 1
    return dims, has_value


def mlp_weights(dims, seed: int, sigma: float = 0.1):
    """Gaussian(0, sigma) fp32 weights W_l [dims[l+1], dims[l]] and zero biases."""
    rng = np.random.default_rng(seed)
    Ws, bs = [], []
    for k, n in zip(dims[:-1], dims[1:]):
        Ws.append((rng.standard_normal((n, k)) * sigma).astype(np.float32))
        bs.append(np.zeros(n, dtype=np.float32))
    return Ws, bs


# Grid policy (the exact policy forward): layer l's input lives on the grid 2^-gx[l] with
# integer mantissas |m| <= GRID_M, its weights on 2^-ew[l] with |m| <= GRID_M, its biases
# on the product grid 2^-(gx[l] + ew[l]) with |m| <= GRID_MB, and dims[l] <= GRID_MAX_K,
# so that every pre-activation is an integer number of product units below 2^24.
GRID_M, GRID_MB, GRID_MAX_K = 255, 1 << 16, 256


def grid_weights(dims, seed: int, gx, ew, sigma: float = 1.0):
    """Weights and biases of a grid policy: integer mantissas drawn from a rounded
    Gaussian of sd sigma * 2^ew / sqrt(fan-in) (clipped to the mantissa range) times the
    layer's grid units; biases small multiples of the product unit."""
    rng = np.random.default_rng(seed)
    Ws, bs = [], []
    for l, (k, n) in enumerate(zip(dims[:-1], dims[1:])):
        sd = sigma * 2.0 ** ew[l] / math.sqrt(k)
        m = np.clip(np.rint(rng.standard_normal((n, k)) * sd), -GRID_M, GRID_M)
        Ws.append(np.ldexp(m, -int(ew[l])).astype(np.float32))
        mb = rng.integers(-GRID_M, GRID_M + 1, n)
        bs.append(np.ldexp(mb.astype(np.float64), -int(gx[l] + ew[l])).astype(np.float32))
    return Ws, bs


def grid_check(Ws, bs, gx, ew) -> None:
    """Raise ValueError unless the weights satisfy the grid policy's premise (each
    pre-activation an exact fp32 value in any summation order)."""
    for l, (w, b) in enumerate(zip(Ws, bs)):
        w = np.asarray(w, np.float64)
        b = np.asarray(b, np.float64)
        if w.shape[1] > GRID_MAX_K:
            raise ValueError("layer %d: fan-in %d above %d" % (l, w.shape[1], GRID_MAX_K))
        mw = np.ldexp(w, int(ew[l]))
        mb = np.ldexp(b, int(gx[l] + ew[l]))
        if np.any(mw != np.rint(mw)) or np.any(np.abs(mw) > GRID_M):
            raise ValueError("layer %d: weights off the grid 2^-%d or above %d units" % (l, ew[l], GRID_M))
        if np.any(mb != np.rint(mb)) or np.any(np.abs(mb) > GRID_MB):
            raise ValueError("layer %d: biases off the product grid or above 2^16 units" % l)


def mlp_acts(name: str) -> list:
    """The activation after each hidden layer of `name`'s policy."""
    n_hidden = len(MLP_SHAPES[name][0]) - 2
    return list(MLP_ACTS.get(name, ["tanh"] * n_hidden))


def _block_masks(name: str, dims):
    """Per-layer 0/1 masks of the weight entries that exist, or None for a dense MLP."""
    if name not in PAPER_NET and name not in TWO_TOWER:
        return None
    L = len(dims) - 1
    masks = []
    for l, (k, n) in enumerate(zip(dims[:-1], dims[1:])):
        m = np.ones((n, k), np.uint8)
        hk = k // 2
        if l == L - 1:                       # heads: logits <- first half, value <- second
            m[:-1, hk:] = 0
            m[-1, :hk] = 0
        elif name in TWO_TOWER and l > 0:    # towers: hidden layers block-diagonal
            hn = n // 2
            m[:hn, hk:] = 0
            m[hn:, :hk] = 0
        masks.append(m)
    return masks


def policy_weights(name: str, dims, seed: int):
    """Initial fp32 weights and biases of `name`'s policy with layer widths `dims`.

    Tanh policies: ``mlp_weights`` (two-tower ones with their off-diagonal blocks zeroed).
    The paper's network: N(0, 1 / (3 fan_in)) weights (the spread of a uniform
    +-1/sqrt(fan_in) draw), small random biases, and the last layer block-diagonal between
    the policy and value heads (the last hidden layer split in halves)."""
    masks = _block_masks(name, dims)
    if name not in PAPER_NET:
        Ws, bs = mlp_weights(dims, seed)
    else:
        rng = np.random.default_rng(seed)
        Ws, bs = [], []
        for k, n in zip(dims[:-1], dims[1:]):
            Ws.append((rng.standard_normal((n, k)) / np.sqrt(3.0 * k)).astype(np.float32))
            bs.append((rng.standard_normal(n) * 0.05).astype(np.float32))
    if masks is not None:
        Ws = [np.where(m != 0, w, np.float32(0.0)).astype(np.float32) for w, m in zip(Ws, masks)]
    return Ws, bs


def param_mask(name: str, dims):
    """Trainable-entry mask (uint8, the flat W0, b0, W1, b1, ... order) or None: the
    zero blocks of the paper's network and of two-tower policies stay frozen at zero,
    which keeps their policy and value heads separate."""
    masks = _block_masks(name, dims)
    if masks is None:
        return None
    return np.concatenate([np.concatenate([m.ravel(), np.ones(m.shape[0], np.uint8)])
                           for m in masks])


def minibatch_perm(n_rows: int, seed: int, epoch: int) -> np.ndarray:
    """The row permutation of one PPO epoch (int64)."""
    rng = np.random.default_rng([seed, epoch])
    return rng.permutation(n_rows).astype(np.int64)
