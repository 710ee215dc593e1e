"""Pins of the oracle's primitives against what mathematics and published sources fix.

Philox4x32-10: published known-answer vectors.  detlog / detexp / dettanh /
detcos2pi: accuracy against numpy's fp64 libm over whole input ranges, plus exact
identities.  Samplers (exponential, duration rounding, Box-Muller normal, Pareto,
type mix, categorical inversion): their distributions, by moments, tail
probabilities and Kolmogorov-Smirnov tests on 10^6 draws.
"""
import math
import os

import numpy as np
import pytest

import oracle
from paper_2607_05272_gb300 import workloads as W

HERE = os.path.dirname(os.path.abspath(__file__))


def _ulps(y32, ref64):
    ref32 = np.asarray(ref64, np.float64).astype(np.float32)
    sp = np.spacing(np.abs(ref32)).astype(np.float64)
    return np.abs(np.asarray(y32, np.float64) - np.asarray(ref64, np.float64)) / sp


def test_philox_known_answers():
    rows = [l.split() for l in open(os.path.join(HERE, "golden", "philox4x32_10_kat.txt"))
            if l.strip() and not l.startswith("#")]
    assert len(rows) == 3
    for r in rows:
        v = [int(x, 16) for x in r]
        out = oracle.philox(v[0:4], v[4:6])
        assert [int(x) for x in out] == v[6:10]


def test_philox_counter_words_uniform():
    w = oracle.philox_n(0, 7, 1, 0x1234, 1 << 16)
    top = (w >> 28).ravel()
    counts = np.bincount(top, minlength=16)
    exp = top.size / 16
    chi2 = ((counts - exp) ** 2 / exp).sum()
    assert chi2 < 60.0  # 15 d.o.f., p ~ 1e-7


def test_detlog_all_sampling_inputs():
    j = np.arange(1 << 24, dtype=np.float64)
    u = ((j + 1.0) * 2.0 ** -24).astype(np.float32)  # every uniform the simulator feeds
    y = oracle.map_fn("log", u)
    ref = np.log(u.astype(np.float64))
    nz = u != 1.0
    assert _ulps(y[nz], ref[nz]).max() <= 4.0
    assert oracle.detlog(1.0) == 0.0
    for k in range(-24, 11):
        x = 2.0 ** k
        assert abs(oracle.detlog(x) - k * math.log(2.0)) <= np.spacing(np.float32(abs(k) * math.log(2.0) or 1.0))


def test_detlog_general_range():
    x = np.exp(np.linspace(np.log(1e-30), np.log(1e30), 1 << 20)).astype(np.float32)
    x = x[np.abs(x - 1.0) > 1e-3]
    y = oracle.map_fn("log", x)
    assert _ulps(y, np.log(x.astype(np.float64))).max() <= 4.0


def test_detexp_range_and_identities():
    x = np.linspace(-86.9, 87.9, 1 << 22).astype(np.float32)
    y = oracle.map_fn("exp", x)
    ref = np.exp(x.astype(np.float64))
    assert _ulps(y, ref).max() <= 4.0
    assert oracle.detexp(0.0) == 1.0
    assert oracle.detexp(-100.0) == 0.0
    for k in range(-10, 11):
        assert oracle.detexp(k * math.log(2.0)) == pytest.approx(2.0 ** k, rel=3e-7)


def test_dettanh():
    x = np.linspace(-12.0, 12.0, 1 << 21).astype(np.float32)
    y = oracle.map_fn("tanh", x)
    ref = np.tanh(x.astype(np.float64))
    big = np.abs(x) > 1e-6
    assert _ulps(y[big], ref[big]).max() <= 4.0
    assert np.array_equal(oracle.map_fn("tanh", -x), -y)  # odd symmetry, bitwise
    assert oracle.dettanh(0.0) == 0.0
    tiny = np.float32(1e-7)
    assert oracle.dettanh(float(tiny)) == pytest.approx(float(tiny), rel=1e-6)


def test_detgelu():
    """GELU's tanh form against the same formula in fp64.  Bound: 8 eps relative, plus
    eps |x| absolute: tanh's error (<= 4 ulp of |t| <= 1) and the rounding of 1 + t,
    scaled by 0.5 |x|, which dominate where 1 + t cancels (x well below 0)."""
    x = np.linspace(-12.0, 12.0, 1 << 21).astype(np.float32)
    y = oracle.map_fn("gelu", x).astype(np.float64)
    xd = x.astype(np.float64)
    ref = 0.5 * xd * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (xd + 0.044715 * xd ** 3)))
    eps = 2.0 ** -23
    assert np.all(np.abs(y - ref) <= 8.0 * eps * np.abs(ref) + eps * np.abs(xd))
    assert oracle.map_fn("gelu", np.zeros(1, np.float32))[0] == 0.0
    big = x > 6.0
    assert np.array_equal(y[big], xd[big])     # tanh saturates at 1: gelu(x) = x exactly


def test_detcos2pi_all_inputs():
    j = np.arange(1 << 24, dtype=np.float64)
    u = (j * 2.0 ** -24).astype(np.float32)
    y = oracle.map_fn("cos2pi", u)
    ref = np.cos(2.0 * np.pi * u.astype(np.float64))
    assert np.abs(y - ref).max() <= 2.0 ** -22
    assert oracle.detcos2pi(0.0) == 1.0
    assert oracle.detcos2pi(0.5) == -1.0
    assert abs(oracle.detcos2pi(0.25)) <= 2.0 ** -23


def _ks(samples, cdf):
    x = np.sort(np.asarray(samples, np.float64))
    n = x.size
    F = cdf(x)
    d = max(np.max(np.arange(1, n + 1) / n - F), np.max(F - np.arange(n) / n))
    return d * math.sqrt(n)


def test_exponential_and_duration_samplers():
    cfg = W.c1()
    w = oracle.philox_n(0, 11, 1, 77, 1 << 20)
    E = oracle.samplers(cfg, 0, w).astype(np.float64)
    n = E.size
    assert abs(E.mean() - 1.0) < 4.0 / math.sqrt(n)
    assert abs(E.var() - 1.0) < 4.0 * math.sqrt(8.0 / n)
    assert _ks(E, lambda x: 1.0 - np.exp(-x)) < 1.95  # p ~ 0.001
    D = oracle.samplers(cfg, 1, w, scale=1250.0).astype(np.float64)
    assert np.all(D == np.floor(D))
    assert abs(D.mean() - 1250.0) < 4.0 * 1250.0 / math.sqrt(n)


def test_normal_sampler():
    w = oracle.philox_n(0, 3, 5, 99, 1 << 20)
    Z = oracle.samplers(W.c4(), 2, w).astype(np.float64)
    n = Z.size
    assert abs(Z.mean()) < 4.0 / math.sqrt(n)
    assert abs(Z.var() - 1.0) < 4.0 * math.sqrt(2.0 / n)
    from scipy.stats import norm
    assert _ks(Z, norm.cdf) < 1.95


def test_pareto_cost_tail():
    cfg = W.c4()
    w = oracle.philox_n(0, 5, 1, 123, 1 << 20)
    X = oracle.samplers(cfg, 4, w).astype(np.float64)
    xm, alpha = 10000.0, 1.5
    assert X.min() >= xm
    n = X.size
    for mult in (2.0, 5.0, 20.0, 100.0):
        p = (1.0 / mult) ** alpha
        phat = np.mean(X > mult * xm)
        assert abs(phat - p) < 4.0 * math.sqrt(p * (1 - p) / n) + 1.0 / n
    top = np.sort(X)[-n // 100:]
    hill = 1.0 / np.mean(np.log(top / top[0]))
    assert abs(hill - alpha) < 0.1


def test_exponential_cost_mean():
    cfg = W.mm1(300.0)
    w = oracle.philox_n(0, 5, 1, 321, 1 << 20)
    X = oracle.samplers(cfg, 4, w).astype(np.float64)
    assert abs(X.mean() - 2100.0) < 4.0 * 2100.0 / math.sqrt(X.size)


def test_type_mix():
    for cfg, p0 in ((W.c2(), 0.8), (W.c3(), 0.7), (W.c4(), 0.85)):
        w = oracle.philox_n(0, 1, 1, 5, 1 << 18)
        t = oracle.samplers(cfg, 3, w)
        p = np.mean(t == 0)
        assert abs(p - p0) < 4.0 * math.sqrt(p0 * (1 - p0) / t.size)


def test_categorical_sampler_frequencies():
    # one linear layer with zero weights: the logits are the biases, independent of obs
    logits = np.array([0.3, -1.0, 2.0, 0.0, 0.7, -0.4], np.float32)
    Ws = [np.zeros((6, 8), np.float32)]
    bs = [logits]
    obs = np.zeros(8, np.float32)
    n = 60000
    counts = np.zeros(6)
    for s in range(n):
        _, _, a, lp = oracle.policy((Ws, bs, False), obs, 0, 42, s, 0)
        counts[a] += 1
    p = np.exp(logits - logits.max())
    p /= p.sum()
    chi2 = ((counts - n * p) ** 2 / (n * p)).sum()
    assert chi2 < 30.0  # 5 d.o.f.
    lg, _, a, lp = oracle.policy((Ws, bs, False), obs, 1, 42, 0, 0)
    assert a == 2
    lse = np.log(np.exp(logits.astype(np.float64)).sum())
    assert lp == pytest.approx(float(logits[2]) - lse, abs=1e-6)


def test_policy_mlp_against_fp64():
    dims, hv = W.mlp_dims("c3")
    Ws, bs = W.mlp_weights(dims, 5)
    bs = [np.random.default_rng(1).standard_normal(b.shape).astype(np.float32) * 0.1 for b in bs]
    rng = np.random.default_rng(3)
    for i in range(50):
        obs = rng.standard_normal(dims[0]).astype(np.float32)
        lg, v, a, lp = oracle.policy((Ws, bs, hv), obs, 0, 1, i, 0)
        h = obs.astype(np.float64)
        mag = None
        for l in range(len(Ws)):
            Wd = Ws[l].astype(np.float64)
            z = Wd @ h + bs[l]
            mag = np.abs(Wd) @ np.abs(h) + np.abs(bs[l])
            h = np.tanh(z) if l + 1 < len(Ws) else z
        A = dims[-1] - 1
        tol = 1e-5 * (np.abs(h) + mag)
        assert np.all(np.abs(lg - h[:A]) <= tol[:A])
        assert abs(v - h[A]) <= tol[A]


@pytest.mark.parametrize("acts", [(1, 2, 1), (2, 0, 2)])
def test_policy_mlp_activations_against_fp64(acts):
    """The oracle's fp32 policy with identity (1) / GELU (2) / tanh (0) hidden layers
    against an fp64 evaluation of the same network (the paper's projection, attention
    over one token and GELU head are such layers)."""
    from oracle import rl
    dims = [8, 4, 4, 64, 7]
    rng = np.random.default_rng(8)
    Ws = [(rng.standard_normal((n, k)) * 0.4).astype(np.float32) for k, n in zip(dims[:-1], dims[1:])]
    bs = [(rng.standard_normal(n) * 0.1).astype(np.float32) for n in dims[1:]]
    for i in range(50):
        obs = (rng.standard_normal(dims[0]) * 2.0).astype(np.float32)
        lg, v, a, lp = oracle.policy((Ws, bs, True, list(acts)), obs, 0, 1, i, 0)
        h = obs.astype(np.float64)
        for l in range(len(Ws)):
            Wd = Ws[l].astype(np.float64)
            z = Wd @ h + bs[l]
            mag = np.abs(Wd) @ np.abs(h) + np.abs(bs[l])
            h = rl.act_fn(acts[l], z) if l + 1 < len(Ws) else z
        tol = 1e-4 * (np.abs(h) + mag)
        assert np.all(np.abs(lg - h[:6]) <= tol[:6])
        assert abs(v - h[6]) <= tol[6]
