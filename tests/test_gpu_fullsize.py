"""Parity at the benchmark's full sizes, in the launch configurations bench.py times.

* c2 as the benchmark runs it (4096 envs x 512 steps, 16 lanes per env, 64-thread blocks,
  the benchmark's seed and weights): sampled envs, which the oracle reproduces one by one,
  bit for bit (records and final state).
* The benchmark step's returns and mean baseline over all 2,097,152 rows against the fp64
  recurrence (within 1e-5 of the recurrence on absolute values), and its REINFORCE loss
  gradient and loss value against the fp64 oracle (computed in row chunks) on the same
  advantages and returns: TF32 within 1e-2, FP32 within 1e-5 per tensor in norm, and per
  element against the condition of each entry's sum over the rows: |g - g_ref| <=
  tol |g_ref| + eps_sum (sum of the absolute values of its per-row addends), eps_sum the
  rounding bound of such a sum (1e-2 TF32, 1e-3 FP32).
* The policy-free router step at 65,536 envs (the thread-per-env kernel's
  configuration): sampled envs' records and final state bit for bit.
"""
import numpy as np
import pytest

import oracle
from oracle import rl
from paper_2607_05272_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

SEED_BENCH = 0x5EED0002  # bench.py's replica seed of rank 0


def _simx():
    from paper_2607_05272_gb300 import build as B
    B.build()
    from paper_2607_05272_gb300 import simx
    return simx


def _c2_rollout(simx):
    E, H = 4096, W.HORIZON["c2"]
    cfg = W.c2(E)
    dims, hv = W.mlp_dims("c2")
    Ws, bs = W.mlp_weights(dims, 1)
    pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws],
                      [torch.from_numpy(b).cuda() for b in bs], hv)
    sim = simx.Sim(cfg)
    sim.reset(SEED_BENCH)
    buf = simx.alloc_rollout(E, sim.D, H, trace=True)
    sim.rollout("sample", H, buf, pol)
    torch.cuda.synchronize()
    return cfg, (Ws, bs, hv), pol, sim, buf, E, H


def _sample(E, k, seed):
    rng = np.random.default_rng(seed)
    return sorted(set([0, 1, E // 2 - 1, E // 2, E - 2, E - 1] +
                      rng.choice(E, k, replace=False).tolist()))


def test_c2_benchmark_rollout_sampled_envs_bit_exact():
    simx = _simx()
    cfg, host, pol, sim, buf, E, H = _c2_rollout(simx)
    envs = _sample(E, 10, 5)
    state = sim.save()
    st, code = sim.last_status()
    sim.close()
    assert st == 0 and code == 0
    ref = oracle.rollout(cfg, host, SEED_BENCH, 0, envs, H)
    got = {k: v.cpu().numpy()[..., envs] for k, v in buf.items()}
    assert np.array_equal(got["action"], ref["action"].astype(np.uint8))
    assert np.array_equal(got["done"], ref["done"])
    assert np.array_equal(got["trace"], ref["trace"])
    for k in ("obs", "reward", "logp"):
        assert np.array_equal(got[k].view(np.uint32), ref[k].view(np.uint32)), k
    assert np.array_equal(state[envs], ref["state"])


def _oracle_loss_chunked(Ws, bs, obs, act, logp, adv, G, n, chunk=262144):
    """REINFORCE loss gradient over all n rows, in row chunks (each chunk's mean weighted
    by its share of the rows), with the sum of absolute addends of every entry."""
    E = obs.shape[2]
    total, scale, stats = None, None, np.zeros(5)
    for r0 in range(0, n, chunk):
        rows = np.arange(r0, min(n, r0 + chunk))
        X, a, lpo = rl.gather_rows(obs, act, logp, rows, E)
        t, e = rows // E, rows % E
        g, st, ab = rl.loss_grad(Ws, bs, False, X, a, lpo, adv[t, e], G[t, e], rl.REINFORCE,
                                 0.2, 0.0, 0.0, abs_terms=True)
        w = len(rows) / n
        f, fa = rl.flat(g) * w, rl.flat(ab) * w
        total = f if total is None else total + f
        scale = fa if scale is None else scale + fa
        stats += np.asarray(st, np.float64) * w
    return total, scale, stats


def test_c2_benchmark_step_full_size_loss_gradient():
    simx = _simx()
    cfg, host, pol, sim, buf, E, H = _c2_rollout(simx)
    sim.close()
    n = E * H
    ret = torch.empty((H, E), device="cuda")
    adv = torch.empty((H, E), device="cuda")
    mean = torch.empty(1, device="cuda")
    simx.compute_returns_gae(buf["reward"], buf["done"], 0.99, -1.0, ret)
    ws_b = torch.empty(simx.returns_baseline_workspace_size(n), dtype=torch.uint8, device="cuda")
    simx.returns_baseline(ret, adv, mean, ws_b)
    grads = {}
    for prec in ("tf32", "fp32"):
        grad = torch.empty(pol.n_params, device="cuda")
        stats = torch.empty(5, device="cuda")
        ws = torch.empty(simx.ppo_loss_grad_workspace_size(pol, n), dtype=torch.uint8,
                         device="cuda")
        simx.ppo_loss_grad(pol, buf, ret, adv, None, n, "reinforce", 0.2, 0.0, 0.0, grad, stats,
                           ws, precision=prec)
        torch.cuda.synchronize()
        grads[prec] = (grad.cpu().numpy().astype(np.float64), stats.cpu().numpy())
    reward = buf["reward"].cpu().numpy()
    done = buf["done"].cpu().numpy()
    G = rl.returns(reward, done, 0.99)
    scale = rl.returns(np.abs(reward), done, 0.99)
    G_gpu = ret.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(G_gpu - G) <= 1e-5 * (np.abs(G) + scale))
    _, m = rl.baseline(G)
    # the mean of values each within the bound above, plus its own fp32 rounding
    assert abs(mean.item() - m) <= 1e-5 * np.mean(np.abs(G) + scale) + 1e-7 * abs(m)
    # the loss on the advantages and returns both sides are given (the GPU's fp32 values)
    A_gpu = adv.cpu().numpy().astype(np.float64)
    Ws, bs, _ = host
    g_ref, g_abs, st_ref = _oracle_loss_chunked(Ws, bs, buf["obs"].cpu().numpy(),
                                         buf["action"].cpu().numpy(), buf["logp"].cpu().numpy(),
                                         A_gpu, G_gpu, n)
    # per element: tol |g_ref| + eps_sum (sum of |addends|).  eps_sum bounds the rounding
    # of a sum over the rows: TF32 inputs (2^-11 relative each) within 1e-2; FP32
    # accumulation of depth below 16,384 (rows per block plus blocks) within
    # 16,384 x 2^-24 < 1e-3 of the absolute sum
    for prec, tol, eps_sum in (("tf32", 1e-2, 1e-2), ("fp32", 1e-5, 1e-3)):
        g, st = grads[prec]
        off = 0
        for w, b in zip(Ws, bs):
            for size in (w.size, b.size):
                gg, rr = g[off:off + size], g_ref[off:off + size]
                off += size
                assert np.linalg.norm(gg - rr) <= tol * np.linalg.norm(rr) + 1e-12, prec
                # per element, against the condition of the sum over 2M rows: the sum
                # of its absolute addends
                sc = g_abs[off - size:off]
                ratio = np.abs(gg - rr) / (tol * np.abs(rr) + eps_sum * sc + 1e-12)
                worst = int(np.argmax(ratio))
                assert ratio[worst] <= 1.0, (prec, off - size, worst, gg[worst], rr[worst], sc[worst])
        assert abs(st[0] - st_ref[0]) <= tol * (abs(st_ref[0]) + 1.0), prec


def test_router_policy_free_step_65536_envs_sampled():
    simx = _simx()
    E, H = 65536, 64
    cfg = W.c5(E)
    sim = simx.Sim(cfg)
    sim.reset(W.SEED["c5"])
    buf = simx.alloc_rollout(E, sim.D, H, trace=True)
    sim.rollout("sq", H, buf)
    torch.cuda.synchronize()
    state = sim.save()
    st, code = sim.last_status()
    sim.close()
    assert st == 0
    envs = _sample(E, 10, 7)
    ref = oracle.rollout(cfg, None, W.SEED["c5"], 4, envs, H)
    got = {k: v.cpu().numpy()[..., envs] for k, v in buf.items()}
    assert np.array_equal(got["action"], ref["action"].astype(np.uint8))
    assert np.array_equal(got["trace"], ref["trace"])
    for k in ("obs", "reward"):
        assert np.array_equal(got[k].view(np.uint32), ref[k].view(np.uint32)), k
    assert np.array_equal(state[envs], ref["state"])
