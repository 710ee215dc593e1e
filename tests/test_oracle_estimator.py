"""The policy-gradient estimator (Sec. 4.3 REINFORCE) against exact enumeration.

A single-server env (c1's server: batch time 2000 + 100 n us, batch sizes
{1, 2, 4, 8, 16, 32}, A = 6) fed by a one-entry trace (an arrival every 700 us, the
same for every env), so that the dynamics are deterministic given the actions and the
policy's draws are the only randomness.  Over a horizon of H = 5 decisions all 6^5
action sequences are enumerated with the oracle's simulator (external actions):

    J(theta) = sum_seq P_theta(seq) sum_t r_t,   P_theta(seq) = prod_t pi(a_t | s_t),

with pi the softmax of the tanh MLP (8-32-6) evaluated in fp64 by PyTorch, and
grad J by PyTorch autograd in fp64 (a library routine, independent of the oracle's
hand-written backward pass).  Then the Monte-Carlo side, entirely the oracle's:
many envs sampled by the oracle's rollout (its categorical sampler), undiscounted
returns G_t = sum_{k >= t} r_k by rl.returns, and the REINFORCE loss gradient of
rl.loss_grad, whose expectation is -grad J / H (the loss is a mean over the H rows of
each trajectory).  Checked, over 100 batches of 400 envs (standard errors from the
spread of the batch means):

* the mean of sum_t r_t equals J within 4 standard errors;
* every parameter's estimate -H grad L equals dJ/dtheta within 5.5 standard errors,
  and so do its projections on grad J and on four random directions within 4 (the
  parameters' errors are correlated, so these are tested one direction at a time);
* the same with a constant baseline subtracted from the returns (unbiased too).

A sign-flipped estimator, per-step rewards in place of returns, or a sampler that
does not draw from pi each fail it.
"""
import numpy as np
import pytest

import oracle
from oracle import rl
from paper_2607_05272_gb300 import workloads as W

torch = pytest.importorskip("torch")

EXTERNAL, SAMPLE = 6, 0
H, A = 5, 6
SEED = 0xE57
N_BATCH, BATCH = 100, 400


def _cfg(n_envs):
    return W._base(n_envs=n_envs, arrival_kind=W.ARR_TRACE, episode_len=1 << 30,
                   trace=(np.array([700], np.uint32), None, None))


def _policy():
    Ws, bs = W.mlp_weights([8, 32, 6], 5, sigma=0.6)
    bs = [(np.random.default_rng(9 + l).standard_normal(b.shape) * 0.3).astype(np.float32)
          for l, b in enumerate(bs)]
    return Ws, bs


def _tree():
    """Observations [6^d][8] at every depth d < H and rewards [6^d][6] of each action."""
    e = oracle.OracleEnv(_cfg(1), 0, SEED)
    e.reset()
    states = [e.export()]
    obs, rew = [], []
    for d in range(H):
        o_d, r_d, nxt = [], [], []
        for st in states:
            e.load(st)
            o_d.append(e.observe())
            row = []
            for a in range(A):
                e.load(st)
                row.append(e.step(EXTERNAL, None, a)["reward"])
                nxt.append(e.export())
            r_d.append(row)
        assert e.status() == 0
        obs.append(np.array(o_d, np.float64))
        rew.append(np.array(r_d, np.float64))
        states = nxt
    return obs, rew


def _exact(Ws, bs):
    """J(theta) and dJ/dtheta (flat, W0 b0 W1 b1 order) by enumeration, fp64 autograd."""
    obs, rew = _tree()
    params = []
    for w, b in zip(Ws, bs):
        params += [torch.tensor(w, dtype=torch.float64, requires_grad=True),
                   torch.tensor(b, dtype=torch.float64, requires_grad=True)]

    def logits(x):
        h = torch.tensor(x)
        for l in range(len(Ws)):
            h = h @ params[2 * l].T + params[2 * l + 1]
            if l + 1 < len(Ws):
                h = torch.tanh(h)
        return h

    V = torch.zeros(A ** H, dtype=torch.float64)
    for d in range(H - 1, -1, -1):
        p = torch.softmax(logits(obs[d]), dim=1)
        Q = torch.tensor(rew[d]) + V.reshape(A ** d, A)
        V = (p * Q).sum(dim=1)
    J = V[0]
    J.backward()
    grad = torch.cat([p.grad.reshape(-1) for p in params]).numpy()
    # the deterministic dynamics make the differences between actions matter
    assert np.ptp(rew[-1]) > 0.1
    return float(J.detach()), grad


@pytest.fixture(scope="module")
def mc():
    Ws, bs = _policy()
    J, dJ = _exact(Ws, bs)
    E = N_BATCH * BATCH
    out = oracle.rollout(_cfg(E), (Ws, bs, False), SEED, SAMPLE, list(range(E)), H)
    assert not out["done"].any()
    G = rl.returns(out["reward"], out["done"], 1.0)
    return Ws, bs, J, dJ, out, G


def _batch_grads(Ws, bs, out, G, shift):
    E = N_BATCH * BATCH
    g = []
    for b in range(N_BATCH):
        envs = np.arange(b * BATCH, (b + 1) * BATCH)
        rows = (np.arange(H)[:, None] * E + envs[None, :]).ravel()
        X, a, lpo = rl.gather_rows(out["obs"], out["action"], out["logp"], rows, E)
        adv = G[rows // E, rows % E] - shift
        grads, _ = rl.loss_grad(Ws, bs, False, X, a, lpo, adv, adv, rl.REINFORCE, 0.2, 0.0, 0.0)
        g.append(-H * rl.flat(grads))
    return np.array(g)


def test_mean_return_is_the_enumerated_value(mc):
    Ws, bs, J, dJ, out, G = mc
    per_batch = G[0].reshape(N_BATCH, BATCH).mean(axis=1)
    se = per_batch.std(ddof=1) / np.sqrt(N_BATCH)
    assert abs(per_batch.mean() - J) < 4.0 * se, (per_batch.mean(), J, se)


@pytest.mark.parametrize("shift", [0.0, 1.7])
def test_reinforce_gradient_is_unbiased(mc, shift):
    Ws, bs, J, dJ, out, G = mc
    g = _batch_grads(Ws, bs, out, G, shift)
    mean = g.mean(axis=0)
    se = g.std(axis=0, ddof=1) / np.sqrt(N_BATCH)
    live = se > 1e-12 * (np.abs(dJ).max() + 1.0)
    # parameters no trajectory moves (a feature that is always 0) are exactly 0 on both sides
    assert np.all(np.abs(mean[~live]) <= 1e-9) and np.all(np.abs(dJ[~live]) <= 1e-9)
    z = (mean[live] - dJ[live]) / se[live]
    assert live.sum() > 100
    assert np.max(np.abs(z)) < 5.5, np.max(np.abs(z))
    dirs = [dJ / np.linalg.norm(dJ)] + \
        [v / np.linalg.norm(v) for v in np.random.default_rng(3).standard_normal((4, dJ.size))]
    for u in dirs:
        proj = g @ u
        zp = (proj.mean() - dJ @ u) / (proj.std(ddof=1) / np.sqrt(N_BATCH))
        assert abs(zp) < 4.0, zp
    # the check has power: the exact gradient is far from zero in standard errors
    assert np.sqrt(np.mean((dJ[live] / se[live]) ** 2)) > 5.0
