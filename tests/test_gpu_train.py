"""The on-device training loop (Sec. 4.3) against the oracle's pipeline, and learning.

One REINFORCE iteration (rollout -> returns -> mean baseline -> loss gradient -> Adam)
through the library matches the same steps on the oracle: the rollout bit for bit
(checked elsewhere), the updated parameters within the loss gradient's 1e-5 and
Adam's arithmetic.  A PPO iteration and the learned-baseline REINFORCE iteration run
end to end and move the parameters.  Training on the heterogeneous two-server router
raises its mean reward per decision above Round-Robin's.
"""
import numpy as np
import pytest

import oracle
from oracle import rl
from paper_2607_05272_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _train():
    from paper_2607_05272_gb300 import build as B
    B.build()
    from paper_2607_05272_gb300 import train
    return train


def test_reinforce_iteration_matches_oracle():
    train = _train()
    name, E, H, lr, seed = "c2", 33, 64, 1e-3, 5
    cfg = W.CONFIGS[name](E)
    dims, hv = W.mlp_dims(name)
    Ws, bs = W.mlp_weights(dims, 3)
    tr = train.Trainer(cfg, dims, hv, weights=(Ws, bs), algo="reinforce", horizon=H, lr=lr,
                       gamma=0.99, c_entropy=0.01, max_grad_norm=0.5, seed=seed)
    tr.iteration()
    torch.cuda.synchronize()
    got = tr.params.cpu().numpy().astype(np.float64)
    out = oracle.rollout(cfg, (Ws, bs, hv), seed, 0, list(range(E)), H)
    G = rl.returns(out["reward"], out["done"], 0.99, np.zeros(E))
    adv, _ = rl.baseline(G)
    rows = np.arange(E * H)
    X, a, lpo = rl.gather_rows(out["obs"], out["action"], out["logp"], rows, E)
    grads, _ = rl.loss_grad(Ws, bs, hv, X, a, lpo, adv.ravel(), G.ravel(), rl.REINFORCE,
                            0.2, 0.0, 0.01)
    g = rl.flat(grads)
    p0 = rl.flat(list(zip(Ws, bs)))
    ref, _, _ = rl.adam_step(p0, g, np.zeros_like(g), np.zeros_like(g), 1, lr, max_grad_norm=0.5)
    # Adam's first step is lr * g / (|g| + eps), about lr sign(g): the gradient's relative
    # error moves it by a small fraction of lr, except for entries whose gradient is
    # within fp32 noise of zero, where the sign itself may differ (at most 2 lr)
    err = np.abs(got - ref)
    tiny = np.abs(g) <= 1e-4 * np.sqrt(np.mean(g * g))
    assert np.all(err[~tiny] <= 1e-6 * np.abs(p0[~tiny]) + 2e-3 * lr)
    assert np.all(err[tiny] <= 1e-6 * np.abs(p0[tiny]) + 2.0 * lr)
    assert np.median(np.abs(ref - p0)) > 0.5 * lr


@pytest.mark.parametrize("name,algo", [("c3", "ppo"), ("c3s", "reinforce"), ("c1p", "reinforce")])
def test_iteration_runs_and_moves_the_policy(name, algo):
    train = _train()
    cfg = W.CONFIGS[name](64)
    dims, hv = W.mlp_dims(name)
    weights = W.policy_weights(name, dims, 2)
    mask = W.param_mask(name, dims)
    tr = train.Trainer(cfg, dims, hv, W.mlp_acts(name), weights, mask, algo=algo, horizon=64,
                       minibatch=1024, epochs=2, lr=1e-3)
    before = tr.params.clone()
    s = tr.iteration()
    torch.cuda.synchronize()
    assert np.isfinite(s["loss"]) and s["updates"] == (8 if algo == "ppo" else 1)
    moved = (tr.params != before).cpu().numpy()
    if mask is None:
        assert moved.mean() > 0.5
    else:   # frozen entries stay, the rest move
        assert not moved[mask == 0].any() and moved[mask != 0].mean() > 0.5


@pytest.mark.parametrize("algo", ["ppo", "reinforce"])
def test_graph_replay_equals_eager_iterations(algo):
    """Four iterations replayed from one captured CUDA graph give the eager iterations'
    parameters bit for bit (same kernels, same minibatch draws, device step counter)."""
    train = _train()
    name = "c3s"
    cfg = W.CONFIGS[name](96)
    dims, hv = W.mlp_dims(name)
    out = []
    for graph in (False, True):
        tr = train.Trainer(cfg, dims, hv, None, W.policy_weights(name, dims, 2),
                           W.param_mask(name, dims), algo=algo, horizon=64, minibatch=2048,
                           epochs=2, lr=1e-3, graph=graph)
        for _ in range(4):
            s = tr.iteration()
        torch.cuda.synchronize()
        out.append((tr.params.cpu().numpy(), tr.t_dev.item(), s["updates"], tr.graph is not None))
    (pe, te, ue, ge), (pg, tg, ug, gg) = out
    assert np.array_equal(pe, pg) and te == tg == ue == ug and gg and not ge


def test_training_beats_round_robin_on_heterogeneous_routing():
    """The segregation result in miniature (Sec. 5): 40 PPO iterations on the two-server
    fast/slow router lift the mean reward per decision well above its start and the
    trained policy above Round-Robin on fresh envs (all seeds fixed, kernels
    deterministic)."""
    train = _train()
    res = train.main(["--workload", "c3s", "--envs", "1024", "--iters", "40", "--every", "1000",
                      "--algo", "ppo"])
    assert res["last10_reward"] > res["first_iter_reward"] + 1.0
    assert res["eval"]["trained_argmax"]["reward"] > res["eval"]["rr"]["reward"]
