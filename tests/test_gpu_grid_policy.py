"""GPU parity of the grid policy (the exact policy forward) against the oracle's definition
(the exact dot product, an fp64 sum rounded once to fp32), through the C ABI.

* Rollouts bit for bit (actions, log-probabilities, values, observations, rewards, final
  state): c2 on the warp-local forward (16-64-64-12), c1p's GELU network on the block-wide
  forward, and the c3 router; ragged env counts.
* policy_forward at the premise's worst case: a hidden layer saturated at +-255 units
  feeding a fan-in-256 output layer with every mantissa at +-255 and the largest bias, so
  the kernel's fp32 FMA chains run up to 2^24 product units.
* Validation: out-of-range grid exponents and too-wide layers are refused; the loss
  gradient takes a grid policy (its parity is test_gpu_grid_loss.py's).
"""
import numpy as np
import pytest

import oracle
from paper_2607_05272_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ORC_MODE = {"sample": 0, "argmax": 1}


def _simx():
    from paper_2607_05272_gb300 import build as B
    B.build()
    from paper_2607_05272_gb300 import simx
    return simx


def _dev(simx, Ws, bs, hv, gx, acts=None):
    return simx.Policy([torch.from_numpy(w).cuda() for w in Ws],
                       [torch.from_numpy(b).cuda() for b in bs], hv, acts, grid=gx)


@pytest.mark.parametrize("name,E", [("c2", 1000), ("c1p", 301), ("c3", 517)])
def test_grid_rollout_matches_oracle(name, E):
    simx = _simx()
    cfg = W.CONFIGS[name](E)
    dims, hv = W.mlp_dims(name)
    acts = W.mlp_acts(name)
    gx = [5] + [7] * (len(dims) - 2)
    ew = [8] * (len(dims) - 1)
    Ws, bs = W.grid_weights(dims, 21, gx, ew)
    W.grid_check(Ws, bs, gx, ew)
    pol = _dev(simx, Ws, bs, hv, gx, acts)
    H, seed = 48, 0x6A1D
    sim = simx.Sim(cfg)
    sim.reset(seed)
    buf = simx.alloc_rollout(E, sim.D, H, has_value=hv, trace=True)
    sim.rollout("sample", H, buf, pol)
    torch.cuda.synchronize()
    got = {k: v.cpu().numpy() for k, v in buf.items()}
    state = sim.save()
    st, code = sim.last_status()
    sim.close()
    assert st == 0 and code == 0
    ref = oracle.rollout(cfg, (Ws, bs, hv, acts, gx), seed, ORC_MODE["sample"], list(range(E)), H)
    assert np.array_equal(got["action"], ref["action"].astype(np.uint8))
    assert np.array_equal(got["trace"], ref["trace"])
    for k in ("obs", "reward", "logp") + (("value",) if hv else ()):
        assert np.array_equal(got[k].view(np.uint32), ref[k].view(np.uint32)), k
    assert np.array_equal(state, ref["state"])
    # the policy is not trivial: several actions are taken
    assert len(np.unique(got["action"])) > 2


def test_grid_policy_forward_worst_case():
    simx = _simx()
    D, Hd, A = 28, 256, 17
    gx, ew = [5, 8], [8, 8]
    rng = np.random.default_rng(8)
    sgn = rng.choice([-1, 1], Hd)
    W0 = np.zeros((Hd, D), np.float32)
    # bias 2^16 product units = 8.0: tanh(+-8) rounds to +-256 units, clamped to +-255
    b0 = np.ldexp(sgn.astype(np.float64) * (1 << 16), -(gx[0] + ew[0])).astype(np.float32)
    m1 = rng.integers(-255, 256, (A + 1, Hd))
    m1[0] = sgn * 255
    m1[1] = -sgn * 255
    mb1 = rng.integers(-(1 << 16), (1 << 16) + 1, A + 1)
    mb1[0], mb1[1] = 1 << 16, -(1 << 16)
    W1 = np.ldexp(m1.astype(np.float64), -ew[1]).astype(np.float32)
    b1 = np.ldexp(mb1.astype(np.float64), -(gx[1] + ew[1])).astype(np.float32)
    Ws, bs = [W0, W1], [b0, b1]
    W.grid_check(Ws, bs, gx, ew)
    pol = _dev(simx, Ws, bs, True, gx)
    n = 133
    obs = (rng.standard_normal((D, n)) * 3.0).astype(np.float32)
    logits = torch.empty((A, n), device="cuda")
    val = torch.empty(n, device="cuda")
    act = torch.empty(n, dtype=torch.uint8, device="cuda")
    lp = torch.empty(n, device="cuda")
    simx.policy_forward(pol, torch.from_numpy(obs).cuda(), n, "sample", 7, 3, env_base=50,
                        logits=logits, value=val, action=act, logp=lp)
    torch.cuda.synchronize()
    lg_all = logits.cpu().numpy()
    top = np.float32(np.ldexp(256.0 * 255 * 255 + (1 << 16), -(gx[1] + ew[1])))
    assert np.all(lg_all[0] == top) and np.all(lg_all[1] == -top)
    for i in range(0, n, 7):
        lg, v, a, l = oracle.policy((Ws, bs, True, None, gx), obs[:, i], ORC_MODE["sample"], 7, 3,
                                    50 + i)
        assert np.array_equal(lg_all[:, i].view(np.uint32), lg.view(np.uint32))
        assert np.float32(val[i].item()) == np.float32(v)
        assert int(act[i]) == a and np.float32(lp[i].item()) == np.float32(l)


def test_grid_policy_validation():
    simx = _simx()
    dims, hv = W.mlp_dims("c2")
    gx, ew = [5, 7, 7], [8, 8, 8]
    Ws, bs = W.grid_weights(dims, 2, gx, ew)
    obs = torch.zeros((dims[0], 4), device="cuda")
    for bad in ([5, 25, 7], [-1, 7, 7]):
        pol = _dev(simx, Ws, bs, hv, bad)
        with pytest.raises(simx.SimxError) as e:
            simx.policy_forward(pol, obs, 4, "argmax", 1, 0)
        assert e.value.status == simx.EINVAL
    wide, wb = W.grid_weights([dims[0], 300, dims[-1]], 2, gx, ew)
    with pytest.raises(simx.SimxError) as e:
        simx.policy_forward(_dev(simx, wide, wb, hv, gx), obs, 4, "argmax", 1, 0)
    assert e.value.status == simx.EINVAL
    # the loss gradient takes grid policies on its fused FP32 path (checked against the
    # oracle in test_gpu_grid_loss.py)
    pol = _dev(simx, Ws, bs, hv, gx)
    cfg = W.c2(5)
    sim = simx.Sim(cfg)
    sim.reset(3)
    buf = simx.alloc_rollout(5, sim.D, 4, has_value=hv)
    sim.rollout("sample", 4, buf, pol)
    sim.close()
    grad = torch.empty(pol.n_params, device="cuda")
    stats = torch.empty(5, device="cuda")
    ws = torch.empty(simx.ppo_loss_grad_workspace_size(pol, 20), dtype=torch.uint8, device="cuda")
    simx.ppo_loss_grad(pol, buf, torch.zeros((4, 5), device="cuda"),
                       torch.ones((4, 5), device="cuda"), None, 20, "reinforce", 0.2, 0.0,
                       0.0, grad, stats, ws)
    torch.cuda.synchronize()
    assert torch.isfinite(grad).all() and torch.isfinite(stats).all()
