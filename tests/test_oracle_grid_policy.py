"""Pins of the oracle's grid policy: the exact policy forward (the Sec. 4.2 network with its
inputs, hidden activations and weights on fixed-point grids, so that every logit is an exact
dot product that any summation order reproduces).

* Grid rounding Q(v, e) = clamp(rint(v 2^e), -255, 255) 2^-e: ties to even, the clamp, and
  random values against numpy's rint in fp64.
* A single layer at the premise's worst case (fan-in 256, every mantissa +-255, the
  largest bias): the logits equal the exact integer sum (Python integers) times the
  product unit, bit for bit.
* Two layers: Q(obs), the exact first layer, tanh, Q, the exact second layer, from
  integers and the oracle's tanh (pinned with the other deterministic functions), bit for
  bit: a missing or misplaced rounding step fails it.
* Order independence: a float32 sum of the same products in a shuffled order gives the
  same bits on the grid, and differs off the grid (the premise is what makes it exact).
* The premise check accepts grid weights and rejects off-grid, out-of-range and too-wide
  layers.
"""
import numpy as np
import pytest

import oracle
from paper_2607_05272_gb300 import workloads as W

ARGMAX = 1


def _policy(Ws, bs, gx, obs, hv=False, acts=None):
    return oracle.policy((Ws, bs, hv, acts, gx), obs, ARGMAX, 1, 0, 0)


def test_gridq_ties_clamp_and_random():
    v = np.array([0.5, 1.5, 2.5, -0.5, -2.5, 254.5, 255.5, 1e9, -1e9, 0.0], np.float32)
    assert oracle.gridq(v, 0).tolist() == [0, 2, 2, 0, -2, 254, 255, 255, -255, 0]
    assert oracle.gridq(np.float32([1.0 / 3.0]), 4)[0] == np.float32(5.0 / 16.0)
    rng = np.random.default_rng(5)
    for e in (0, 3, 7, 10):
        x = (rng.standard_normal(20000) * 300.0 / 2 ** e).astype(np.float32)
        want = np.ldexp(np.clip(np.rint(np.ldexp(x.astype(np.float64), e)), -255, 255), -e)
        assert np.array_equal(oracle.gridq(x, e), want.astype(np.float32))


def test_single_layer_worst_case_is_the_exact_sum():
    K, N, gx, ew = 256, 8, 6, 9
    rng = np.random.default_rng(11)
    mx = rng.choice([-255, 255], K)
    obs = np.ldexp(mx.astype(np.float64), -gx).astype(np.float32)   # already on the grid
    mw = rng.integers(-255, 256, (N, K)).astype(np.int64)
    mw[0] = np.sign(mx) * 255            # row 0: the largest sum, row 1: the smallest
    mw[1] = -mw[0]
    mb = np.array([1 << 16, -(1 << 16)] + list(rng.integers(-(1 << 16), (1 << 16) + 1, N - 2)))
    Wl = np.ldexp(mw.astype(np.float64), -ew).astype(np.float32)
    bl = np.ldexp(mb.astype(np.float64), -(gx + ew)).astype(np.float32)
    logits, _, _, _ = _policy([Wl], [bl], [gx], obs)
    for j in range(N):
        z = sum(int(a) * int(b) for a, b in zip(mw[j], mx)) + int(mb[j])
        assert abs(z) <= 1 << 24
        assert logits[j] == np.float32(np.ldexp(float(z), -(gx + ew))), j
    top = np.float32(np.ldexp(256.0 * 255 * 255 + (1 << 16), -(gx + ew)))
    assert logits[0] == top and logits[1] == -top


def test_two_layers_from_integers():
    dims, gx, ew = [13, 64, 17], [5, 7], [8, 8]
    Ws, bs = W.grid_weights(dims, 3, gx, ew)
    rng = np.random.default_rng(4)
    for _ in range(20):
        obs = (rng.standard_normal(13) * 2.0).astype(np.float32)
        logits, value, _, _ = _policy(Ws, bs, gx, obs, hv=True)
        # layer 0 from integers: Q(obs) on 2^-5, weights on 2^-8
        mx = np.clip(np.rint(np.ldexp(obs.astype(np.float64), gx[0])), -255, 255).astype(np.int64)
        mw0 = np.ldexp(Ws[0].astype(np.float64), ew[0]).astype(np.int64)
        mb0 = np.ldexp(bs[0].astype(np.float64), gx[0] + ew[0]).astype(np.int64)
        z0 = [np.float32(np.ldexp(float(int(mw0[j] @ mx) + int(mb0[j])), -(gx[0] + ew[0])))
              for j in range(64)]
        h = np.float32([oracle.dettanh(float(z)) for z in z0])
        mh = np.clip(np.rint(np.ldexp(h.astype(np.float64), gx[1])), -255, 255).astype(np.int64)
        mw1 = np.ldexp(Ws[1].astype(np.float64), ew[1]).astype(np.int64)
        mb1 = np.ldexp(bs[1].astype(np.float64), gx[1] + ew[1]).astype(np.int64)
        out = np.float32([np.ldexp(float(int(mw1[j] @ mh) + int(mb1[j])), -(gx[1] + ew[1]))
                          for j in range(17)])
        assert np.array_equal(logits.view(np.uint32), out[:16].view(np.uint32))
        assert np.float32(value) == out[16]


def _f32_sum(w, x, order):
    acc = np.float32(0.0)
    for k in order:
        acc = np.float32(acc + np.float32(w[k] * x[k]))
    return acc


def test_any_summation_order_gives_the_same_bits():
    dims, gx, ew = [200, 4], [6], [9]
    Ws, bs = W.grid_weights(dims, 9, gx, ew, sigma=3.0)
    rng = np.random.default_rng(2)
    obs = oracle.gridq((rng.standard_normal(200) * 3.0).astype(np.float32), gx[0])
    logits, _, _, _ = _policy(Ws, bs, gx, obs)
    for j in range(4):
        for _ in range(5):
            z = np.float32(_f32_sum(Ws[0][j], obs, rng.permutation(200)) + bs[0][j])
            assert z == logits[j]
    # off the grid the float32 sums depend on the order
    w = (rng.standard_normal(200) * 3.0).astype(np.float32)
    x = (rng.standard_normal(200) * 3.0).astype(np.float32)
    sums = {float(_f32_sum(w, x, rng.permutation(200))) for _ in range(20)}
    assert len(sums) > 1


def test_premise_check():
    dims, gx, ew = [13, 64, 17], [5, 7], [8, 8]
    Ws, bs = W.grid_weights(dims, 3, gx, ew)
    W.grid_check(Ws, bs, gx, ew)
    bad = [w.copy() for w in Ws]
    bad[1][0, 0] += np.float32(2.0 ** -10)
    with pytest.raises(ValueError):
        W.grid_check(bad, bs, gx, ew)
    big = [w.copy() for w in Ws]
    big[0][3, 2] = np.float32(256 * 2.0 ** -8)
    with pytest.raises(ValueError):
        W.grid_check(big, bs, gx, ew)
    wide, wb = W.grid_weights([300, 4], 1, [5], [8])
    with pytest.raises(ValueError):
        W.grid_check(wide, wb, [5], [8])
    bb = [b.copy() for b in bs]
    bb[0][0] = np.float32(np.ldexp(float((1 << 16) + 1), -(gx[0] + ew[0])))
    with pytest.raises(ValueError):
        W.grid_check(Ws, bb, gx, ew)


def _grid_problem(name, seed, n=24):
    dims, hv = W.mlp_dims(name)
    acts = W.mlp_acts(name)
    gx = [5] + [7] * (len(dims) - 2)
    ew = [8] * (len(dims) - 1)
    Ws, bs = W.grid_weights(dims, seed, gx, ew)
    rng = np.random.default_rng(seed)
    X = (rng.standard_normal((n, dims[0])) * 1.5).astype(np.float32)
    return Ws, bs, hv, acts, gx, X


@pytest.mark.parametrize("name", ["c3", "c1p"])
def test_loss_oracle_grid_forward_is_the_policy(name):
    """The loss oracle's grid forward (fp64 sums, fp32 activations and rounding) gives the
    simulator oracle's logits and value bit for bit (the rounding decisions agree)."""
    from oracle import rl
    Ws, bs, hv, acts, gx, X = _grid_problem(name, 5)
    _, Z = rl.forward(Ws, bs, X, acts, gx)
    for i in range(len(X)):
        lg, v, _, _ = oracle.policy((Ws, bs, hv, acts, gx), X[i], ARGMAX, 1, 0, 0)
        A = len(lg)
        assert np.array_equal(Z[i, :A].astype(np.float32).view(np.uint32), lg.view(np.uint32))
        assert np.all(Z[i, :A].astype(np.float32) == Z[i, :A])     # exact in fp32
        if hv:
            assert np.float32(Z[i, A]) == np.float32(v)


@pytest.mark.parametrize("name,algo", [("c3", 1), ("c1p", 0), ("c1p", 1)])
def test_grid_straight_through_gradient_matches_autograd(name, algo):
    """The grid policy's gradient passes the rounding straight through: PyTorch autograd of
    the same forward written as h = a + (q - a).detach() (q the rounded values) agrees."""
    torch = pytest.importorskip("torch")
    from oracle import rl
    Ws, bs, hv, acts, gx, X = _grid_problem(name, 9)
    n = len(X)
    rng = np.random.default_rng(3)
    inputs, Z = rl.forward(Ws, bs, X, acts, gx)
    A = Z.shape[1] - (1 if hv else 0)
    a = rng.integers(0, A, n)
    adv = rng.standard_normal(n)
    ret = rng.standard_normal(n)
    lpo = rng.standard_normal(n) * 0.3 - 1.4
    grads, stats = rl.loss_grad(Ws, bs, hv, X, a, lpo, adv, ret, algo, 0.2, 0.5, 0.01,
                                acts=acts, grid=gx)
    tW = [torch.tensor(w, dtype=torch.float64, requires_grad=True) for w in Ws]
    tb = [torch.tensor(b, dtype=torch.float64, requires_grad=True) for b in bs]
    fns = {rl.TANH: torch.tanh, rl.IDENTITY: lambda z: z,
           rl.GELU: lambda z: torch.nn.functional.gelu(z, approximate="tanh")}
    h = torch.tensor(inputs[0])
    for l in range(len(Ws)):
        z = h @ tW[l].T + tb[l]
        if l + 1 < len(Ws):
            act = fns[rl.ACT_NAMES.get(acts[l], acts[l])](z)
            h = act + (torch.tensor(inputs[l + 1]) - act).detach()
        else:
            h = z
    assert np.array_equal(h.detach().numpy(), Z)
    logpi = torch.log_softmax(h[:, :A], dim=1)
    lpa = logpi[torch.arange(n), torch.tensor(a)]
    advt = torch.tensor(adv)
    if algo == rl.REINFORCE:
        pg = -(advt * lpa).mean()
    else:
        rho = torch.exp(lpa - torch.tensor(lpo))
        pg = -torch.minimum(rho * advt, torch.clamp(rho, 0.8, 1.2) * advt).mean()
    loss = pg - 0.01 * (-(logpi.exp() * logpi).sum(1).mean())
    if hv:
        loss = loss + 0.5 * ((h[:, A] - torch.tensor(ret)) ** 2).mean()
    loss.backward()
    assert stats[0] == pytest.approx(loss.item(), rel=1e-12, abs=1e-12)
    for (gW, gb), w, b in zip(grads, tW, tb):
        assert np.allclose(gW, w.grad.numpy(), rtol=1e-10, atol=1e-12)
        assert np.allclose(gb, b.grad.numpy(), rtol=1e-10, atol=1e-12)


def test_gridq_over_all_finite_floats():
    """Q against its definition in fp64 (exact there) over every finite fp32 input and grid
    exponent 0 .. 24: huge values, subnormals and signed zeros included."""
    hyp = pytest.importorskip("hypothesis")
    st = pytest.importorskip("hypothesis.strategies")

    @hyp.settings(max_examples=3000, deadline=None)
    @hyp.given(st.floats(width=32, allow_nan=False, allow_infinity=False), st.integers(0, 24))
    def check(v, e):
        got = oracle.gridq(np.float32([v]), e)[0]
        want = np.float32(np.ldexp(min(max(np.rint(np.ldexp(np.float64(v), e)), -255.0), 255.0), -e))
        assert got.view(np.uint32) == want.view(np.uint32), (v, e, got, want)

    check()
