"""Returns, GAE, baseline and loss gradients in numpy fp64 (test infrastructure only).

Written from the paper's Sec. 4.3 (REINFORCE: Monte-Carlo policy gradient with
discounted returns and a baseline; PPO: clipped surrogate with an entropy bonus) and
the GAE estimator of Schulman et al. (2016).  Each function is the plain definition:
a reverse loop over time for the recurrences, explicit forward and backward passes
of the tanh MLP for the gradients.
"""
from __future__ import annotations

import math

import numpy as np

REINFORCE, PPO = 0, 1


def returns(rew, done, gamma, last_value=None):
    """REINFORCE returns G_t = r_t + gamma (1 - d_t) G_{t+1}, G_T = last_value."""
    rew = np.asarray(rew, np.float64)
    done = np.asarray(done, np.float64)
    T, E = rew.shape
    G = np.zeros((T, E))
    nxt = np.zeros(E) if last_value is None else np.asarray(last_value, np.float64).copy()
    for t in range(T - 1, -1, -1):
        nxt = rew[t] + gamma * (1.0 - done[t]) * nxt
        G[t] = nxt
    return G


def gae(rew, val, done, gamma, lam, last_value=None):
    """GAE: delta_t = r_t + gamma (1-d_t) V_{t+1} - V_t; A_t = delta_t + gamma lam (1-d_t) A_{t+1};
    returns (A, R = A + V)."""
    rew = np.asarray(rew, np.float64)
    val = np.asarray(val, np.float64)
    done = np.asarray(done, np.float64)
    T, E = rew.shape
    A = np.zeros((T, E))
    next_v = np.zeros(E) if last_value is None else np.asarray(last_value, np.float64).copy()
    next_a = np.zeros(E)
    for t in range(T - 1, -1, -1):
        mask = 1.0 - done[t]
        delta = rew[t] + gamma * mask * next_v - val[t]
        next_a = delta + gamma * lam * mask * next_a
        A[t] = next_a
        next_v = val[t]
    return A, A + val


def baseline(x):
    """Mean-return baseline: (x - mean(x), mean(x)) with the mean in fp64."""
    x = np.asarray(x, np.float64)
    m = x.sum() / x.size
    return x - m, m


TANH, IDENTITY, GELU = 0, 1, 2
ACT_NAMES = {"tanh": TANH, "identity": IDENTITY, "gelu": GELU}
GELU_C, GELU_A = math.sqrt(2.0 / math.pi), 0.044715


def act_fn(kind, z):
    """Hidden-layer activation (Sec. 4.2): tanh, identity, or GELU in its tanh form
    0.5 z (1 + tanh(sqrt(2/pi) (z + 0.044715 z^3))); kind is a code or a name."""
    kind = ACT_NAMES.get(kind, kind)
    if kind == IDENTITY:
        return z
    if kind == GELU:
        return 0.5 * z * (1.0 + np.tanh(GELU_C * (z + GELU_A * z ** 3)))
    return np.tanh(z)


def act_grad(kind, z):
    """d act / d z."""
    kind = ACT_NAMES.get(kind, kind)
    if kind == IDENTITY:
        return np.ones_like(z)
    if kind == GELU:
        t = np.tanh(GELU_C * (z + GELU_A * z ** 3))
        return 0.5 * (1.0 + t) + 0.5 * z * (1.0 - t * t) * GELU_C * (1.0 + 3.0 * GELU_A * z * z)
    return 1.0 - np.tanh(z) ** 2


def _grid_act(kind, z, e):
    """A grid policy's hidden output: the activation of the fp32 pre-activation by the
    simulator oracle's deterministic fp32 functions, then the grid rounding Q(., e).  The
    rounding turns values into integers, so it is taken in the kernels' precision; the
    fp64 pre-activation of a grid policy is an exact fp32 value, so the cast is exact."""
    from .binding import gridq, map_fn
    kind = ACT_NAMES.get(kind, kind)
    z32 = np.asarray(z, np.float32)
    if kind == IDENTITY:
        a = z32
    else:
        a = map_fn("gelu" if kind == GELU else "tanh", z32.ravel()).reshape(z32.shape)
    return gridq(a.ravel(), e).reshape(z32.shape).astype(np.float64)


def _forward(Ws, bs, X, acts=None, grid=None):
    """grid: the input grid exponent of every layer of a grid policy (the exact policy
    forward): its layer inputs are rounded to their grids, and the backward pass lets the
    gradient through the rounding unchanged (the straight-through estimator)."""
    if grid is None:
        h = np.asarray(X, np.float64)
    else:
        from .binding import gridq
        X32 = np.asarray(X, np.float32)
        h = gridq(X32.ravel(), grid[0]).reshape(X32.shape).astype(np.float64)
    inputs, zs = [], []
    L = len(Ws)
    for l in range(L):
        inputs.append(h)
        z = h @ np.asarray(Ws[l], np.float64).T + np.asarray(bs[l], np.float64)
        zs.append(z)
        if l + 1 == L:
            h = z
        elif grid is None:
            h = act_fn(acts[l] if acts else TANH, z)
        else:
            h = _grid_act(acts[l] if acts else TANH, z, grid[l + 1])
    return inputs, zs, h


def forward(Ws, bs, X, acts=None, grid=None):
    """MLP forward in fp64 (tanh hidden layers unless acts says otherwise); returns the
    list of layer inputs and the last layer's output."""
    inputs, _, h = _forward(Ws, bs, X, acts, grid)
    return inputs, h


def loss_grad(Ws, bs, has_value, X, actions, logp_old, adv, ret, algo, clip_eps=0.2,
              c_value=0.5, c_entropy=0.01, acts=None, grid=None, abs_terms=False):
    """Loss, statistics and the gradient with respect to every W_l, b_l (fp64).

    pi = softmax(logits); policy term REINFORCE -mean(adv log pi(a)) or PPO
    -mean(min(rho adv, clip(rho, 1-eps, 1+eps) adv)) with rho = exp(log pi(a) - logp_old);
    plus c_value mean((V - ret)^2) when a value row exists, minus c_entropy mean(H[pi]).
    Returns (grads [(gW, gb) per layer], stats [L, pg, v, H, clipfrac]); with abs_terms
    also, per layer, the sums over rows of the absolute addends of each gradient entry,
    (|dz|^T |h_in|, sum |dz|): the scale of the rounding error any summation of those
    addends can make (the condition of the sum).
    """
    inputs, zs, Z = _forward(Ws, bs, X, acts, grid)
    n = Z.shape[0]
    A = Z.shape[1] - (1 if has_value else 0)
    logits = Z[:, :A]
    m = logits.max(axis=1, keepdims=True)
    lse = m + np.log(np.exp(logits - m).sum(axis=1, keepdims=True))
    logpi = logits - lse
    pi = np.exp(logpi)
    a = np.asarray(actions, np.int64)
    rows = np.arange(n)
    lpa = logpi[rows, a]
    adv = np.asarray(adv, np.float64)
    onehot = np.zeros_like(logits)
    onehot[rows, a] = 1.0
    if algo == REINFORCE:
        pg = -np.mean(adv * lpa)
        coef = adv
        clipfrac = 0.0
    else:
        rho = np.exp(lpa - np.asarray(logp_old, np.float64))
        s1 = rho * adv
        s2 = np.clip(rho, 1.0 - clip_eps, 1.0 + clip_eps) * adv
        pg = -np.mean(np.minimum(s1, s2))
        coef = np.where(s1 <= s2, adv, 0.0) * rho
        clipfrac = float(np.mean(np.abs(rho - 1.0) > clip_eps))
    dlogits = -(coef[:, None] / n) * (onehot - pi)
    H = -(pi * logpi).sum(axis=1)
    dlogits += (c_entropy / n) * pi * (logpi + H[:, None])
    loss = pg - c_entropy * H.mean()
    vloss = 0.0
    dZ = np.zeros_like(Z)
    dZ[:, :A] = dlogits
    if has_value:
        v = Z[:, A]
        r = np.asarray(ret, np.float64)
        vloss = float(np.mean((v - r) ** 2))
        loss += c_value * vloss
        dZ[:, A] = 2.0 * c_value * (v - r) / n
    grads = [None] * len(Ws)
    absg = [None] * len(Ws)
    dz = dZ
    for l in range(len(Ws) - 1, -1, -1):
        h_in = inputs[l]
        grads[l] = (dz.T @ h_in, dz.sum(axis=0))
        if abs_terms:
            absg[l] = (np.abs(dz).T @ np.abs(h_in), np.abs(dz).sum(axis=0))
        if l > 0:
            dh = dz @ np.asarray(Ws[l], np.float64)
            dz = dh * act_grad(acts[l - 1] if acts else TANH, zs[l - 1])
    stats = np.array([loss, pg, vloss, H.mean(), clipfrac])
    if abs_terms:
        return grads, stats, absg
    return grads, stats


def flat(grads):
    """Concatenate gradients in the library's order W0, b0, W1, b1, ..."""
    return np.concatenate([np.concatenate([g.ravel(), b.ravel()]) for g, b in grads])


def gather_rows(obs, actions, logp, idx, E):
    """Minibatch rows of a [T][D][E] rollout: row r is (t = r // E, e = r % E)."""
    idx = np.asarray(idx, np.int64)
    t, e = idx // E, idx % E
    X = obs[t, :, e]
    return X, np.asarray(actions)[t, e], np.asarray(logp)[t, e]


def adam_step(p, g, m, v, t, lr, beta1=0.9, beta2=0.999, eps=1e-8, max_grad_norm=0.0,
              mask=None):
    """One Adam step (Kingma & Ba 2015, Algorithm 1) in fp64, the optimiser of the
    training loop (Sec. 4.3 names none).  When max_grad_norm > 0 the gradient is first
    scaled by min(1, max_grad_norm / ||g||_2); entries with mask == 0 are left as they
    are and do not count in the norm.  Returns the new (p, m, v)."""
    p, g, m, v = (np.array(x, np.float64) for x in (p, g, m, v))
    sel = np.ones(p.shape, bool) if mask is None else np.asarray(mask) != 0
    s = 1.0
    if max_grad_norm > 0.0:
        norm = math.sqrt(float(np.sum(g[sel] ** 2)))
        if norm > max_grad_norm:
            s = max_grad_norm / norm
    gs = g[sel] * s
    m[sel] = beta1 * m[sel] + (1.0 - beta1) * gs
    v[sel] = beta2 * v[sel] + (1.0 - beta2) * gs * gs
    m_hat = m[sel] / (1.0 - beta1 ** t)
    v_hat = v[sel] / (1.0 - beta2 ** t)
    p[sel] = p[sel] - lr * m_hat / (np.sqrt(v_hat) + eps)
    return p, m, v
