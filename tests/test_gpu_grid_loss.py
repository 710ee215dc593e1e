"""The loss gradient of grid policies (Sec. 4.3 REINFORCE / PPO over the exact policy
forward) on the fused FP32 kernel, against the loss oracle's grid path.

The kernel rounds the gathered observations and every hidden output to their grids as the
rollout does (so the forward reproduces the rollout's logits) and lets the gradient through
each rounding unchanged (the straight-through estimator: the activation's derivative at the
pre-activation, the weight gradients over the rounded layer inputs).  The oracle
(`oracle/rl.py`, grid=) computes the same forward with exact sums and the straight-through
backward in fp64; it is pinned to the simulator oracle's logits bit for bit and to PyTorch
autograd of h = a + (q - a).detach() (test_oracle_grid_policy.py).  Checked:

* c2 (16-64-64-12, tanh), c3 (13-128-128-17 with a value row) and the paper's network c1p
  (identity and GELU layers), REINFORCE and PPO, whole buffers and minibatches: every
  gradient entry within 1e-5 of the oracle (relative to the entry plus the tensor's rms),
  the statistics within 1e-5;
* the forward inside the loss is the rollout's: with the old log-probabilities equal to
  the rollout's, no PPO ratio leaves 1 (clip fraction 0) and PPO's gradient is
  REINFORCE's to 1e-6 (the ratios are 1 up to the rounding of the softmax sums);
* a TF32 request gives the FP32 path's bits (grid policies have only that path);
* a grid policy of c4's size (too large for the fused kernel) is rejected.
"""
import numpy as np
import pytest

from oracle import rl
from paper_2607_05272_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _simx():
    from paper_2607_05272_gb300 import build as B
    B.build()
    from paper_2607_05272_gb300 import simx
    return simx


def _grid_host(name, seed=31):
    dims, hv = W.mlp_dims(name)
    acts = W.mlp_acts(name)
    gx = [5] + [7] * (len(dims) - 2)
    ew = [8] * (len(dims) - 1)
    Ws, bs = W.grid_weights(dims, seed, gx, ew)
    W.grid_check(Ws, bs, gx, ew)
    return Ws, bs, hv, acts, gx


def _rollout(simx, name, E, H, host):
    Ws, bs, hv, acts, gx = host
    pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws],
                      [torch.from_numpy(b).cuda() for b in bs], hv, acts, grid=gx)
    sim = simx.Sim(W.CONFIGS[name](E))
    sim.reset(W.SEED[name] + 7)
    buf = simx.alloc_rollout(E, sim.D, H, has_value=hv)
    sim.rollout("sample", H, buf, pol)
    torch.cuda.synchronize()
    st, code = sim.last_status()
    sim.close()
    assert st == 0 and code == 0
    return pol, buf


def _call(simx, pol, buf, ret, adv, idx, n, algo, precision):
    grad = torch.empty(pol.n_params, device="cuda")
    stats = torch.empty(5, device="cuda")
    ws = torch.empty(simx.ppo_loss_grad_workspace_size(pol, n), dtype=torch.uint8, device="cuda")
    simx.ppo_loss_grad(pol, buf, torch.from_numpy(ret).cuda(), torch.from_numpy(adv).cuda(),
                       None if idx is None else torch.from_numpy(idx).cuda(), n, algo, 0.2, 0.5,
                       0.01, grad, stats, ws, precision=precision)
    torch.cuda.synchronize()
    return grad.cpu().numpy(), stats.cpu().numpy()


def _check_grad(g, g_ref, layers, tol=1e-5):
    off = 0
    for (W_, b_) in layers:
        for size in (W_.size, b_.size):
            gg, rr = g[off:off + size], g_ref[off:off + size]
            off += size
            assert np.linalg.norm(gg - rr) <= tol * np.linalg.norm(rr) + 1e-12
            rms = np.sqrt(np.mean(rr ** 2))
            assert np.all(np.abs(gg - rr) <= tol * (np.abs(rr) + rms) + 1e-12)


CASES = [("c2", "reinforce", 40, 128, None), ("c2", "ppo", 33, 200, 3001),
         ("c3", "ppo", 64, 128, 8192), ("c3", "reinforce", 9, 50, None),
         ("c1p", "reinforce", 40, 200, None), ("c1p", "ppo", 17, 300, 2001)]


@pytest.mark.parametrize("name,algo,E,H,nmb", CASES,
                         ids=["%s-%s-%s" % (c[0], c[1], c[4] or "all") for c in CASES])
def test_grid_loss_gradient_matches_oracle(name, algo, E, H, nmb):
    simx = _simx()
    host = _grid_host(name)
    Ws, bs, hv, acts, gx = host
    pol, buf = _rollout(simx, name, E, H, host)
    rng = np.random.default_rng(5)
    adv = (rng.standard_normal((H, E)) * 2.0).astype(np.float32)
    ret = rng.standard_normal((H, E)).astype(np.float32)
    logp = buf["logp"].cpu().numpy()
    if algo == "ppo":
        shift = rng.choice([0.0, 0.35, -0.35], size=(H, E)).astype(np.float32)
        logp = (logp + shift).astype(np.float32)
        buf["logp"] = torch.from_numpy(logp).cuda()
    n_rows = E * H
    idx = None if nmb is None else rng.permutation(n_rows)[:nmb].astype(np.int64)
    n = n_rows if idx is None else nmb
    g, st = _call(simx, pol, buf, ret, adv, idx, n, algo, "fp32")
    obs = buf["obs"].cpu().numpy()
    act = buf["action"].cpu().numpy()
    rows = np.arange(n_rows) if idx is None else idx
    X, a, lpo = rl.gather_rows(obs, act, logp, rows, E)
    t, e = rows // E, rows % E
    grads, st_ref = rl.loss_grad(Ws, bs, hv, X, a, lpo, adv[t, e], ret[t, e],
                                 rl.PPO if algo == "ppo" else rl.REINFORCE, 0.2, 0.5, 0.01, acts,
                                 grid=gx)
    _check_grad(g.astype(np.float64), rl.flat(grads), list(zip(Ws, bs)))
    assert np.allclose(st, st_ref, rtol=1e-5, atol=1e-6), (st, st_ref)
    # a TF32 request takes the same (only) path: the same bits
    g32, st32 = _call(simx, pol, buf, ret, adv, idx, n, algo, "tf32")
    assert np.array_equal(g32.view(np.uint32), g.view(np.uint32))
    assert np.array_equal(st32.view(np.uint32), st.view(np.uint32))


def test_grid_loss_forward_is_the_rollouts():
    """With logp_old the rollout's own log-probabilities every ratio is 1 up to the
    rounding of the softmax sums: the loss kernel's grid forward gives the rollout's
    logits (an off-grid forward would move them by whole grid steps)."""
    simx = _simx()
    host = _grid_host("c3", seed=4)
    pol, buf = _rollout(simx, "c3", 48, 64, host)
    H, E = 64, 48
    rng = np.random.default_rng(9)
    adv = rng.standard_normal((H, E)).astype(np.float32)
    ret = rng.standard_normal((H, E)).astype(np.float32)
    g, st = _call(simx, pol, buf, ret, adv, None, E * H, "ppo", "fp32")
    assert st[4] == 0.0   # clip fraction: no row's ratio moved from 1
    # PPO with rho = 1 is REINFORCE's gradient (the surrogate's gradient at rho = 1)
    g_r, _ = _call(simx, pol, buf, ret, adv, None, E * H, "reinforce", "fp32")
    assert np.allclose(g, g_r, rtol=1e-6, atol=1e-9)


def test_grid_policy_too_large_for_the_loss_is_rejected():
    simx = _simx()
    dims, hv = W.mlp_dims("c4")
    gx, ew = [5, 7, 7], [8, 8, 8]
    Ws, bs = W.grid_weights(dims, 2, gx, ew)
    pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws],
                      [torch.from_numpy(b).cuda() for b in bs], hv, grid=gx)
    sim = simx.Sim(W.c4(5))
    buf = simx.alloc_rollout(5, sim.D, 4, has_value=hv)
    sim.close()
    grad = torch.empty(pol.n_params, device="cuda")
    stats = torch.empty(5, device="cuda")
    ws = torch.empty(max(simx.ppo_loss_grad_workspace_size(pol, 20), 16), dtype=torch.uint8,
                     device="cuda")
    with pytest.raises(simx.SimxError) as e:
        simx.ppo_loss_grad(pol, buf, torch.zeros((4, 5), device="cuda"),
                           torch.zeros((4, 5), device="cuda"), None, 20, "reinforce", 0.2, 0.5,
                           0.0, grad, stats, ws)
    assert e.value.status == simx.EINVAL
