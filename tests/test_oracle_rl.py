"""Pins of the oracle's returns, GAE, baseline and loss gradients (Sec. 4.3).

* Returns and GAE against the O(T^2) direct sums, the constant-reward closed form,
  and the special cases lambda = 1 (A = G - V) and lambda = 0 (A = delta).
* The hand-written backward pass against PyTorch autograd (fp64, CPU) and against
  central finite differences of the loss.
* The PPO policy term at rho = 1 equals the REINFORCE form; loss values at uniform
  logits equal their closed forms.
* PPO's clipping by the sign of the advantage: one row at a tabulated ratio, the gradient 0
  exactly when the clipped branch is the minimum and rho times REINFORCE's otherwise (a max
  for the min, the branch test reversed or a clip that ignores the sign each fail a case).
* The entropy bonus alone is stationary at uniform logits (its maximum); the value term alone
  gives the value row's bias gradient 2 c_v mean(V - R) and zero on the action rows.
"""
import math

import numpy as np
import pytest

from oracle import rl


def _direct_returns(r, d, gamma, last):
    T = len(r)
    G = np.zeros(T)
    for t in range(T):
        acc, disc, alive = 0.0, 1.0, 1.0
        for j in range(t, T):
            acc += disc * alive * r[j]
            alive *= 1.0 - d[j]
            disc *= gamma
        acc += disc * alive * last
        G[t] = acc
    return G


def _direct_gae(r, v, d, gamma, lam, last):
    T = len(r)
    vn = np.append(v[1:], last)
    delta = r + gamma * (1.0 - d) * vn - v
    A = np.zeros(T)
    for t in range(T):
        acc, disc, alive = 0.0, 1.0, 1.0
        for j in range(t, T):
            acc += disc * alive * delta[j]
            alive *= 1.0 - d[j]
            disc *= gamma * lam
        A[t] = acc
    return A


def test_returns_brute_force():
    rng = np.random.default_rng(0)
    T, E = 48, 5
    r = rng.standard_normal((T, E))
    d = (rng.random((T, E)) < 0.1).astype(np.uint8)
    last = rng.standard_normal(E)
    G = rl.returns(r, d, 0.97, last)
    for e in range(E):
        assert np.allclose(G[:, e], _direct_returns(r[:, e], d[:, e], 0.97, last[e]), rtol=1e-12, atol=1e-12)


def test_returns_constant_reward_closed_form():
    T, g, c = 64, 0.99, 2.5
    G = rl.returns(np.full((T, 1), c), np.zeros((T, 1)), g)
    t = np.arange(T)
    assert np.allclose(G[:, 0], c * (1 - g ** (T - t)) / (1 - g), rtol=1e-12)


def test_gae_brute_force_and_special_cases():
    rng = np.random.default_rng(1)
    T, E = 40, 4
    r = rng.standard_normal((T, E))
    v = rng.standard_normal((T, E))
    d = (rng.random((T, E)) < 0.1).astype(np.uint8)
    last = rng.standard_normal(E)
    A, R = rl.gae(r, v, d, 0.99, 0.95, last)
    for e in range(E):
        assert np.allclose(A[:, e], _direct_gae(r[:, e], v[:, e], d[:, e], 0.99, 0.95, last[e]), atol=1e-12)
    assert np.allclose(R, A + v)
    A1, _ = rl.gae(r, v, d, 0.99, 1.0, last)
    assert np.allclose(A1, rl.returns(r, d, 0.99, last) - v, atol=1e-12)
    A0, _ = rl.gae(r, v, d, 0.99, 0.0, last)
    vn = np.vstack([v[1:], last[None]])
    assert np.allclose(A0, r + 0.99 * (1 - d) * vn - v, atol=1e-12)


def test_baseline():
    x = np.random.default_rng(2).standard_normal(1000) + 3.0
    adv, m = rl.baseline(x)
    assert m == pytest.approx(x.mean())
    assert abs(adv.sum()) < 1e-9


def _tiny(has_value, seed=0, dims=(5, 7, 6, 4)):
    rng = np.random.default_rng(seed)
    dims = list(dims)
    if has_value:
        dims[-1] += 1
    Ws = [rng.standard_normal((n, k)) * 0.5 for k, n in zip(dims[:-1], dims[1:])]
    bs = [rng.standard_normal(n) * 0.1 for n in dims[1:]]
    n = 9
    X = rng.standard_normal((n, dims[0]))
    A = dims[-1] - (1 if has_value else 0)
    a = rng.integers(0, A, n)
    adv = rng.standard_normal(n)
    ret = rng.standard_normal(n)
    logp_old = rng.standard_normal(n) * 0.3 - 1.4
    return Ws, bs, X, a, adv, ret, logp_old


def _torch_loss(Ws, bs, has_value, X, a, logp_old, adv, ret, algo, eps, cv, ce, acts=None):
    torch = pytest.importorskip("torch")
    tW = [torch.tensor(w, dtype=torch.float64, requires_grad=True) for w in Ws]
    tb = [torch.tensor(b, dtype=torch.float64, requires_grad=True) for b in bs]
    h = torch.tensor(X, dtype=torch.float64)
    fns = {rl.TANH: torch.tanh, rl.IDENTITY: lambda z: z,
           rl.GELU: lambda z: torch.nn.functional.gelu(z, approximate="tanh")}
    for l in range(len(Ws)):
        z = h @ tW[l].T + tb[l]
        h = fns[acts[l] if acts else rl.TANH](z) if l + 1 < len(Ws) else z
    A = h.shape[1] - (1 if has_value else 0)
    logpi = torch.log_softmax(h[:, :A], dim=1)
    lpa = logpi[torch.arange(len(a)), torch.tensor(a)]
    advt = torch.tensor(adv)
    if algo == rl.REINFORCE:
        pg = -(advt * lpa).mean()
    else:
        rho = torch.exp(lpa - torch.tensor(logp_old))
        pg = -torch.minimum(rho * advt, torch.clamp(rho, 1 - eps, 1 + eps) * advt).mean()
    ent = -(logpi.exp() * logpi).sum(1).mean()
    loss = pg - ce * ent
    if has_value:
        loss = loss + cv * ((h[:, A] - torch.tensor(ret)) ** 2).mean()
    loss.backward()
    return loss.item(), [(w.grad.numpy(), b.grad.numpy()) for w, b in zip(tW, tb)]


@pytest.mark.parametrize("algo,has_value", [(rl.REINFORCE, False), (rl.REINFORCE, True),
                                            (rl.PPO, True), (rl.PPO, False)])
def test_loss_grad_matches_autograd(algo, has_value):
    Ws, bs, X, a, adv, ret, lpo = _tiny(has_value, seed=algo * 2 + has_value)
    grads, stats = rl.loss_grad(Ws, bs, has_value, X, a, lpo, adv, ret, algo, 0.2, 0.5, 0.01)
    L, tg = _torch_loss(Ws, bs, has_value, X, a, lpo, adv, ret, algo, 0.2, 0.5, 0.01)
    assert stats[0] == pytest.approx(L, rel=1e-12, abs=1e-12)
    for (gW, gb), (tW, tb) in zip(grads, tg):
        assert np.allclose(gW, tW, rtol=1e-10, atol=1e-12)
        assert np.allclose(gb, tb, rtol=1e-10, atol=1e-12)


@pytest.mark.parametrize("acts", [(rl.IDENTITY, rl.GELU), (rl.GELU, rl.TANH), (rl.GELU, rl.GELU)])
def test_loss_grad_with_activations_matches_autograd(acts):
    """Identity and GELU hidden layers (the paper's network shape) against PyTorch autograd
    with its own tanh-form GELU."""
    Ws, bs, X, a, adv, ret, lpo = _tiny(True, seed=11)
    grads, stats = rl.loss_grad(Ws, bs, True, X, a, lpo, adv, ret, rl.PPO, 0.2, 0.5, 0.01,
                                acts=list(acts))
    L, tg = _torch_loss(Ws, bs, True, X, a, lpo, adv, ret, rl.PPO, 0.2, 0.5, 0.01, acts=list(acts))
    assert stats[0] == pytest.approx(L, rel=1e-12, abs=1e-12)
    for (gW, gb), (tW, tb) in zip(grads, tg):
        assert np.allclose(gW, tW, rtol=1e-10, atol=1e-12)
        assert np.allclose(gb, tb, rtol=1e-10, atol=1e-12)


def test_loss_grad_finite_differences():
    Ws, bs, X, a, adv, ret, lpo = _tiny(True, seed=5)
    algo = rl.PPO
    grads, _ = rl.loss_grad(Ws, bs, True, X, a, lpo, adv, ret, algo)
    rng = np.random.default_rng(9)
    h = 1e-6
    for l in range(len(Ws)):
        for _ in range(6):
            j, k = rng.integers(0, Ws[l].shape[0]), rng.integers(0, Ws[l].shape[1])
            Wp = [w.copy() for w in Ws]
            Wm = [w.copy() for w in Ws]
            Wp[l][j, k] += h
            Wm[l][j, k] -= h
            Lp = rl.loss_grad(Wp, bs, True, X, a, lpo, adv, ret, algo)[1][0]
            Lm = rl.loss_grad(Wm, bs, True, X, a, lpo, adv, ret, algo)[1][0]
            assert grads[l][0][j, k] == pytest.approx((Lp - Lm) / (2 * h), rel=1e-5, abs=1e-8)


def test_ppo_at_rho_one_equals_reinforce():
    Ws, bs, X, a, adv, ret, _ = _tiny(False, seed=3)
    inputs, Z = rl.forward(Ws, bs, X)
    m = Z.max(1, keepdims=True)
    logpi = Z - (m + np.log(np.exp(Z - m).sum(1, keepdims=True)))
    lpo = logpi[np.arange(len(a)), a]
    g_ppo, s_ppo = rl.loss_grad(Ws, bs, False, X, a, lpo, adv, ret, rl.PPO, 0.2, 0.0, 0.0)
    g_rf, s_rf = rl.loss_grad(Ws, bs, False, X, a, lpo, adv, ret, rl.REINFORCE, 0.2, 0.0, 0.0)
    assert np.allclose(rl.flat(g_ppo), rl.flat(g_rf), rtol=1e-12, atol=1e-14)
    assert s_ppo[1] == pytest.approx(-np.mean(adv))   # rho = 1: -mean(adv)
    assert s_ppo[4] == 0.0


# adv, rho, whether the clipped branch is the minimum (PPO, eps = 0.2), the policy term
CLIP_CASES = [(1.5, 1.5, True, -1.2 * 1.5), (1.5, 0.5, False, -0.5 * 1.5),
              (-1.5, 0.5, True, 0.8 * 1.5), (-1.5, 1.5, False, 1.5 * 1.5),
              (1.5, 1.1, False, -1.1 * 1.5), (-1.5, 0.9, False, 0.9 * 1.5)]


@pytest.mark.parametrize("adv,rho,clipped,pg", CLIP_CASES)
def test_ppo_clip_cases_by_advantage_sign(adv, rho, clipped, pg):
    """One row, no entropy or value term.  The surrogate min(rho A, clip(rho, 1-eps, 1+eps) A)
    is flat in theta exactly when its clipped branch is the smaller one: rho above 1 + eps with
    A > 0, or below 1 - eps with A < 0.  Then the gradient is 0; otherwise the gradient is that
    of -rho A, i.e. rho times the REINFORCE gradient -A grad log pi(a).  The policy term is the
    tabulated value, and the clip fraction counts |rho - 1| > eps whichever branch wins."""
    Ws, bs, X, a, _, ret, _ = _tiny(False, seed=6)
    X, a, ret = X[:1], a[:1], ret[:1]
    _, Z = rl.forward(Ws, bs, X)
    m = Z.max(1, keepdims=True)
    lpa = (Z - (m + np.log(np.exp(Z - m).sum(1, keepdims=True))))[0, a[0]]
    lpo = np.array([lpa - math.log(rho)])
    A = np.array([adv])
    g_ppo, s = rl.loss_grad(Ws, bs, False, X, a, lpo, A, ret, rl.PPO, 0.2, 0.0, 0.0)
    g_rf, _ = rl.loss_grad(Ws, bs, False, X, a, lpo, A, ret, rl.REINFORCE, 0.2, 0.0, 0.0)
    gp, gr = rl.flat(g_ppo), rl.flat(g_rf)
    assert np.abs(gr).max() > 1e-3
    if clipped:
        assert np.all(gp == 0.0)
    else:
        assert np.allclose(gp, rho * gr, rtol=1e-12, atol=1e-15)
    assert s[1] == pytest.approx(pg, rel=1e-12)
    assert s[4] == (1.0 if abs(rho - 1.0) > 0.2 else 0.0)


def test_entropy_bonus_is_stationary_at_uniform_logits():
    """The entropy of pi = softmax(z) is largest at uniform logits, so with only the entropy
    term (A = 0, no value row) every gradient vanishes there; a sign slip in its derivative
    (pi (log pi - H) for pi (log pi + H)) does not."""
    Ws, bs, X, a, _, ret, lpo = _tiny(False, seed=8)
    Ws[-1][:] = 0.0
    bs[-1][:] = 0.0
    g, s = rl.loss_grad(Ws, bs, False, X, a, lpo, np.zeros(len(a)), ret, rl.REINFORCE, 0.2, 0.0, 1.0)
    assert s[3] == pytest.approx(math.log(Ws[-1].shape[0]), rel=1e-14)
    assert np.abs(rl.flat(g)).max() < 1e-14
    # away from uniform the same term has a gradient
    Ws[-1][0, 0] = 1.0
    g, _ = rl.loss_grad(Ws, bs, False, X, a, lpo, np.zeros(len(a)), ret, rl.REINFORCE, 0.2, 0.0, 1.0)
    assert np.abs(rl.flat(g)).max() > 1e-3


def test_value_term_bias_gradient_closed_form():
    """Only the value term (A = 0, no entropy): L = c_v mean((V - R)^2) with V the last row of
    the last layer, so dL/db_V = 2 c_v mean(V - R), the action rows' bias gradients are 0, and
    the statistic is the mean squared error itself."""
    Ws, bs, X, a, _, ret, lpo = _tiny(True, seed=12)
    cv = 0.5
    _, Z = rl.forward(Ws, bs, X)
    V = Z[:, -1]
    g, s = rl.loss_grad(Ws, bs, True, X, a, lpo, np.zeros(len(a)), ret, rl.REINFORCE, 0.2, cv, 0.0)
    gb = g[-1][1]
    assert gb[-1] == pytest.approx(2.0 * cv * np.mean(V - ret), rel=1e-12)
    assert np.all(gb[:-1] == 0.0)
    assert s[2] == pytest.approx(np.mean((V - ret) ** 2), rel=1e-12)
    assert s[0] == pytest.approx(cv * s[2], rel=1e-12)


def test_uniform_logits_closed_forms():
    # zero last layer: logits all zero, pi uniform over A actions
    Ws, bs, X, a, adv, ret, lpo = _tiny(False, seed=4)
    Ws[-1][:] = 0.0
    bs[-1][:] = 0.0
    A = Ws[-1].shape[0]
    _, s = rl.loss_grad(Ws, bs, False, X, a, lpo, np.ones(len(a)), ret, rl.REINFORCE, 0.2, 0.0, 1.0)
    assert s[3] == pytest.approx(math.log(A))          # entropy of the uniform distribution
    assert s[1] == pytest.approx(math.log(A))          # -mean(log(1/A))
    assert s[0] == pytest.approx(math.log(A) - math.log(A))


def test_gather_rows_layout():
    T, D, E = 3, 2, 4
    obs = np.arange(T * D * E, dtype=np.float32).reshape(T, D, E)
    act = np.arange(T * E).reshape(T, E)
    X, a, _ = rl.gather_rows(obs, act, act, [0, 5, 11], E)
    assert X.tolist() == [[0, 4], [9, 13], [19, 23]]
    assert a.tolist() == [0, 5, 11]


def _adam_case(masked):
    rng = np.random.default_rng(8)
    n = 300
    p0 = rng.standard_normal(n)
    grads = [rng.standard_normal(n) * (0.1 + i) for i in range(5)]
    mask = (rng.random(n) < 0.7).astype(np.uint8) if masked else None
    sel = np.ones(n, bool) if mask is None else mask != 0
    return p0, grads, mask, sel


@pytest.mark.parametrize("masked", [False, True])
def test_adam_matches_torch_optimiser(masked):
    """Five Adam steps against torch.optim.Adam in fp64; masked entries stay put and the
    rest follow torch on the unmasked sub-vector."""
    torch = pytest.importorskip("torch")
    p0, grads, mask, sel = _adam_case(masked)
    n = len(p0)
    tp = torch.tensor(p0[sel], requires_grad=True)
    opt = torch.optim.Adam([tp], lr=3e-3, betas=(0.9, 0.99), eps=1e-6)
    p, m, v = p0.copy(), np.zeros(n), np.zeros(n)
    for t, g in enumerate(grads, start=1):
        tp.grad = torch.tensor(g[sel])
        opt.step()
        p, m, v = rl.adam_step(p, g, m, v, t, 3e-3, 0.9, 0.99, 1e-6, 0.0, mask)
    assert np.allclose(p[sel], tp.detach().numpy(), rtol=1e-12, atol=1e-14)
    assert np.array_equal(p[~sel], p0[~sel]) and np.all(m[~sel] == 0) and np.all(v[~sel] == 0)
    st = opt.state[tp]
    assert np.allclose(m[sel], st["exp_avg"].numpy(), rtol=1e-12, atol=1e-15)
    assert np.allclose(v[sel], st["exp_avg_sq"].numpy(), rtol=1e-12, atol=1e-15)


@pytest.mark.parametrize("masked", [False, True])
def test_adam_clipping_matches_torch_clip_grad_norm(masked):
    """Global-norm clipping over the unmasked entries against torch's clip_grad_norm_,
    whose scale max_norm / (norm + 1e-6) differs from min(1, max_norm / norm) by 1e-6 in
    the denominator: moments and movement equal within 1e-5 of their magnitude (entries
    where m nearly cancels amplify the difference).  A bound above the norm changes
    nothing."""
    torch = pytest.importorskip("torch")
    p0, grads, mask, sel = _adam_case(masked)
    n = len(p0)
    p, m, v = p0.copy(), np.zeros(n), np.zeros(n)
    q, mq, vq = p0.copy(), np.zeros(n), np.zeros(n)
    for t, g in enumerate(grads, start=1):
        tg = torch.tensor(g[sel])
        tg.grad = tg.clone()
        torch.nn.utils.clip_grad_norm_([tg], 0.5)
        gc = g.copy()
        gc[sel] = tg.grad.numpy()
        p, m, v = rl.adam_step(p, g, m, v, t, 3e-3, 0.9, 0.99, 1e-6, 0.5, mask)
        q, mq, vq = rl.adam_step(q, gc, mq, vq, t, 3e-3, 0.9, 0.99, 1e-6, 0.0, mask)
        assert np.max(np.abs(m - mq)) <= 1e-5 * np.max(np.abs(m))
    assert np.max(np.abs(p - q)) <= 1e-5 * np.max(np.abs(p - p0))   # of the total movement
    a = rl.adam_step(p0, grads[0], np.zeros(n), np.zeros(n), 1, 3e-3, max_grad_norm=1e9, mask=mask)
    b = rl.adam_step(p0, grads[0], np.zeros(n), np.zeros(n), 1, 3e-3, mask=mask)
    assert all(np.array_equal(x, y) for x, y in zip(a, b))


def test_adam_first_step_moves_each_entry_by_lr():
    """A textbook property: at t = 1 with eps -> 0 the step is lr sign(g) per entry."""
    g = np.array([3.0, -0.01, 1e-4, -250.0])
    p, _, _ = rl.adam_step(np.zeros(4), g, np.zeros(4), np.zeros(4), 1, 0.01, eps=1e-300)
    assert np.allclose(p, -0.01 * np.sign(g), rtol=1e-12)
