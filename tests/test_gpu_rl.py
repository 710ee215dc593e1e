"""GPU parity of returns, GAE, the mean baseline and the loss gradients (Sec. 4.3).

The oracle computes in fp64; the CUDA path in fp32 with a different association
order, so these compare within tolerances derived from the arithmetic:
* returns / GAE, per element: |x - x_ref| <= 1e-5 * (|x_ref| + s) where s is the
  same recurrence run on absolute values (the sum of |terms| it adds), and per
  tensor ||x - x_ref|| <= 1e-5 ||x_ref||;
* loss gradients, per tensor: ||g - g_ref|| <= 1e-5 ||g_ref||, per element:
  |g - g_ref| <= 1e-5 (|g_ref| + rms(g_ref)); the tensor-core (TF32-input) path is held
  to 1e-2 under the same definitions.
Sizes span several blocks with ragged tails, plus the full c1 returns shape; every env
count here (up to 40,000) takes the chunked two-pass returns kernel.  Env counts from
65,536 that are a multiple of 4 take the one-pass four-envs-per-thread kernel instead;
test_gpu_launch_shapes.py covers it at 65,536 and 262,144 envs (and 262,145, which
falls back to the chunked one).
"""
import numpy as np
import pytest

import oracle
from oracle import rl
from paper_2607_05272_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _simx():
    from paper_2607_05272_gb300 import build as B
    B.build()
    from paper_2607_05272_gb300 import simx
    return simx


def _check_recurrence(x, ref, scale):
    x = x.astype(np.float64)
    assert np.all(np.abs(x - ref) <= 1e-5 * (np.abs(ref) + scale) + 1e-30)
    assert np.linalg.norm(x - ref) <= 1e-5 * np.linalg.norm(ref)


@pytest.mark.parametrize("T,E,seg", [(10000, 64, 1000), (512, 4096, 512), (257, 333, 50), (1, 5, 1),
                                     (77, 33001, 20), (5, 40000, 3)])
def test_reinforce_returns(T, E, seg):
    simx = _simx()
    rng = np.random.default_rng(T + E)
    r = (rng.standard_normal((T, E)) * 3.0 - 1.0).astype(np.float32)
    d = np.zeros((T, E), np.uint8)
    d[seg - 1::seg] = 1
    last = rng.standard_normal(E).astype(np.float32)
    ret = torch.empty((T, E), device="cuda")
    simx.compute_returns_gae(torch.from_numpy(r).cuda(), torch.from_numpy(d).cuda(), 0.99, -1.0,
                             ret, last_val=torch.from_numpy(last).cuda())
    torch.cuda.synchronize()
    ref = rl.returns(r, d, 0.99, last)
    scale = rl.returns(np.abs(r), d, 0.99, np.abs(last))
    _check_recurrence(ret.cpu().numpy(), ref, scale)


@pytest.mark.parametrize("T,E", [(256, 16384), (512, 1000), (1024, 97), (3, 40), (301, 40000),
                                 (1, 32768)])
def test_gae(T, E):
    simx = _simx()
    rng = np.random.default_rng(T * 7 + E)
    r = rng.standard_normal((T, E)).astype(np.float32)
    v = rng.standard_normal((T, E)).astype(np.float32)
    d = (rng.random((T, E)) < 0.02).astype(np.uint8)
    d[-1] = 1
    last = rng.standard_normal(E).astype(np.float32)
    adv = torch.empty((T, E), device="cuda")
    ret = torch.empty((T, E), device="cuda")
    simx.compute_returns_gae(torch.from_numpy(r).cuda(), torch.from_numpy(d).cuda(), 0.99, 0.95,
                             ret, adv=adv, val=torch.from_numpy(v).cuda(),
                             last_val=torch.from_numpy(last).cuda())
    torch.cuda.synchronize()
    A, R = rl.gae(r, v, d, 0.99, 0.95, last)
    # condition: the GAE recurrence on |delta| terms (|r| + gamma |V'| + |V|)
    vn = np.vstack([v[1:], last[None]]).astype(np.float64)
    absd = np.abs(r) + 0.99 * np.abs(vn) + np.abs(v)
    scale = rl.returns(absd, d, 0.99 * 0.95)
    _check_recurrence(adv.cpu().numpy(), A, scale)
    _check_recurrence(ret.cpu().numpy(), R, scale + np.abs(v))


@pytest.mark.parametrize("n", [1, 1000, 2_097_152])
def test_mean_baseline(n):
    simx = _simx()
    rng = np.random.default_rng(n)
    x = (rng.standard_normal(n) * 50.0 - 300.0).astype(np.float32)
    xt = torch.from_numpy(x).cuda()
    adv = torch.empty_like(xt)
    mean = torch.empty(1, device="cuda")
    ws = torch.empty(simx.returns_baseline_workspace_size(n), dtype=torch.uint8, device="cuda")
    simx.returns_baseline(xt, adv, mean, ws)
    torch.cuda.synchronize()
    a_ref, m_ref = rl.baseline(x)
    assert abs(mean.item() - m_ref) <= 1e-6 * abs(m_ref)
    assert np.all(np.abs(adv.cpu().numpy() - a_ref) <= 1e-6 * (np.abs(x) + abs(m_ref)))


def _rollout_for_loss(simx, name, E, H, hidden=None):
    cfg = W.CONFIGS[name](E)
    dims, hv = W.mlp_dims(name)
    if hidden is not None:
        dims = [dims[0]] + [hidden] * (len(dims) - 2) + [dims[-1]]
    Ws, bs = W.policy_weights(name, dims, 21)
    bs = [(np.random.default_rng(l).standard_normal(b.shape) * 0.05).astype(np.float32)
          for l, b in enumerate(bs)]
    acts = W.mlp_acts(name)
    pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws],
                      [torch.from_numpy(b).cuda() for b in bs], hv, acts)
    sim = simx.Sim(cfg)
    sim.reset(W.SEED[name])
    buf = simx.alloc_rollout(E, sim.D, H, has_value=hv)
    sim.rollout("sample", H, buf, pol)
    torch.cuda.synchronize()
    sim.close()
    return cfg, pol, (Ws, bs, hv, acts), buf


def _check_grad(g, g_ref, layers, tol=1e-5):
    off = 0
    for (W_, b_) in layers:
        for size in (W_.size, b_.size):
            gg, rr = g[off:off + size], g_ref[off:off + size]
            off += size
            assert np.linalg.norm(gg - rr) <= tol * np.linalg.norm(rr) + 1e-12
            rms = np.sqrt(np.mean(rr ** 2))
            assert np.all(np.abs(gg - rr) <= tol * (np.abs(rr) + rms) + 1e-12)


def _loss_case(simx, name, algo, E, H, nmb, precision="fp32", hidden=None):
    cfg, pol, host, buf = _rollout_for_loss(simx, name, E, H, hidden)
    n_rows = E * H
    rng = np.random.default_rng(3)
    adv = (rng.standard_normal((H, E)) * 2.0).astype(np.float32)
    ret = rng.standard_normal((H, E)).astype(np.float32)
    logp = buf["logp"].cpu().numpy()
    if algo == "ppo":
        # move half the rows' old log-probabilities so clipping is exercised, keeping
        # rho away from the clip edges by more than the arithmetic's noise
        shift = rng.choice([0.0, 0.35, -0.35], size=(H, E)).astype(np.float32)
        logp = (logp + shift).astype(np.float32)
        buf["logp"] = torch.from_numpy(logp).cuda()
    idx = None if nmb is None else rng.permutation(n_rows)[:nmb].astype(np.int64)
    n = n_rows if idx is None else len(idx)
    grad = torch.empty(pol.n_params, device="cuda")
    stats = torch.empty(5, device="cuda")
    ws = torch.empty(simx.ppo_loss_grad_workspace_size(pol, n), dtype=torch.uint8, device="cuda")
    simx.ppo_loss_grad(pol, buf, torch.from_numpy(ret).cuda(), torch.from_numpy(adv).cuda(),
                       None if idx is None else torch.from_numpy(idx).cuda(), n, algo, 0.2, 0.5,
                       0.01, grad, stats, ws, precision=precision)
    torch.cuda.synchronize()
    obs = buf["obs"].cpu().numpy()
    act = buf["action"].cpu().numpy()
    rows = np.arange(n_rows) if idx is None else idx
    X, a, lpo = rl.gather_rows(obs, act, logp, rows, E)
    t, e = rows // E, rows % E
    Ws, bs, hv, acts = host
    grads, st = rl.loss_grad(Ws, bs, hv, X, a, lpo, adv[t, e], ret[t, e],
                             rl.PPO if algo == "ppo" else rl.REINFORCE, 0.2, 0.5, 0.01, acts)
    return grad.cpu().numpy().astype(np.float64), stats.cpu().numpy().astype(np.float64), \
        rl.flat(grads), st, list(zip(Ws, bs)), n


@pytest.mark.parametrize("name,algo,E,H,nmb", [
    ("c3", "ppo", 64, 256, 8192),
    ("c4", "ppo", 33, 128, 3000),
    ("c2", "reinforce", 40, 512, None),
    ("c1", "reinforce", 16, 700, 5000),
    ("c3", "ppo", 8, 64, 333),
    ("c2", "reinforce", 3, 7, None),
    ("c1p", "reinforce", 40, 300, None),   # the paper's network: identity and GELU layers
    ("c1p", "ppo", 17, 500, 4001),
])
def test_loss_gradient_matches_oracle(name, algo, E, H, nmb):
    simx = _simx()
    g, s, g_ref, st, layers, n = _loss_case(simx, name, algo, E, H, nmb)
    _check_grad(g, g_ref, layers)
    assert np.all(np.abs(s[:4] - st[:4]) <= 1e-5 * (np.abs(st[:4]) + 1.0))
    assert abs(s[4] - st[4]) <= 1.0 / n  # clip fraction: at most one row on an fp32 edge


@pytest.mark.parametrize("name,algo,E,H,nmb,hidden", [
    ("c2", "reinforce", 40, 512, None, None),   # 160 full 128-row tiles
    ("c2", "reinforce", 3, 7, None, None),      # one partial tile
    ("c1", "reinforce", 16, 700, 5000, None),   # minibatch, ragged last tile
    ("c2", "ppo", 37, 300, 9001, None),
    ("c3", "ppo", 64, 256, 8192, 64),           # value head, 13-64-64-17
    ("c3", "reinforce", 21, 50, None, 32),
    # the streamed kernels of wide policies (layers up to 256)
    ("c3", "ppo", 64, 256, 8192, None),         # 13-128-128-17, a full minibatch
    ("c3", "ppo", 8, 64, 333, None),            # three tiles, the last ragged
    ("c4", "ppo", 33, 128, 3000, None),         # 28-256-256-49
    ("c4", "reinforce", 9, 100, None, None),    # every row, 8 tiles
    ("c3", "ppo", 16, 256, 4001, 100),          # 13-100-100-17: widths off the 16 / 32 grid
    ("c3s", "ppo", 32, 256, 8192, None),        # 10-128-128-9, two-tower policy
])
def test_tensor_core_loss_gradient_matches_oracle(name, algo, E, H, nmb, hidden):
    """TF32 tensor-core loss gradient against the fp64 oracle, within 1e-2."""
    simx = _simx()
    g, s, g_ref, st, layers, n = _loss_case(simx, name, algo, E, H, nmb, "tf32", hidden)
    _check_grad(g, g_ref, layers, tol=1e-2)
    assert np.all(np.abs(s[:4] - st[:4]) <= 1e-2 * (np.abs(st[:4]) + 1.0))
    assert abs(s[4] - st[4]) <= 1.0 / n


@pytest.mark.parametrize("name,hidden", [("c1p", None), ("c1p", 256)])
def test_tensor_core_request_falls_back(name, hidden):
    """A policy the tensor-core kernels do not take (identity / GELU layers) gives the
    FP32 path's exact bits."""
    simx = _simx()
    a = _loss_case(simx, name, "ppo", 16, 64, 700, "tf32", hidden)
    b = _loss_case(simx, name, "ppo", 16, 64, 700, "fp32", hidden)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


@pytest.mark.parametrize("name,algo,E,H,nmb,hidden", [
    ("c1p", "ppo", 24, 200, 3001, 256),     # 8-256-256-256-256-34: identity and GELU layers
    ("c4", "reinforce", 9, 100, None, None),  # 28-256-256-49 tanh
])
def test_gemm_pipeline_loss_gradient_matches_oracle(name, algo, E, H, nmb, hidden):
    """Policies too wide for the fused one-kernel path take the GEMM pipeline."""
    simx = _simx()
    g, s, g_ref, st, layers, n = _loss_case(simx, name, algo, E, H, nmb, "fp32", hidden)
    _check_grad(g, g_ref, layers)
    assert np.all(np.abs(s[:4] - st[:4]) <= 1e-5 * (np.abs(st[:4]) + 1.0))
    assert abs(s[4] - st[4]) <= 1.0 / n


@pytest.mark.parametrize("n,clip,masked", [(1, 0.0, False), (1000, 0.0, False), (100003, 0.5, False),
                                           (77777, 0.0, True), (5102, 1.0, True)])
def test_adam_matches_oracle(n, clip, masked):
    """Six Adam steps on fp32 device vectors against the fp64 oracle: parameters within
    1e-6 of their size plus 1e-4 of the total step length, moments within 1e-5."""
    f32 = lambda x: float(np.float32(x))
    simx = _simx()
    rng = np.random.default_rng(n)
    p0 = rng.standard_normal(n).astype(np.float32)
    mask = (rng.random(n) < 0.6).astype(np.uint8) if masked else None
    p, m, v = (torch.from_numpy(x).cuda() for x in (p0.copy(), np.zeros(n, np.float32),
                                                    np.zeros(n, np.float32)))
    tm = None if mask is None else torch.from_numpy(mask).cuda()
    ws = torch.empty(simx.adam_workspace_size(n), dtype=torch.uint8, device="cuda")
    rp, rm, rv = p0.astype(np.float64), np.zeros(n), np.zeros(n)
    lr = 1e-3
    for t in range(1, 7):
        g = (rng.standard_normal(n) * 10.0 ** rng.uniform(-3, 1, n)).astype(np.float32)
        simx.adam_step(p, torch.from_numpy(g).cuda(), m, v, t, lr, 0.9, 0.999, 1e-8, clip, tm, ws)
        # the oracle takes the hyper-parameters the ABI carries: fp32 values
        rp, rm, rv = rl.adam_step(rp, g, rm, rv, t, *map(f32, (lr, 0.9, 0.999, 1e-8, clip)), mask)
    torch.cuda.synchronize()
    gp, gm, gv = (x.cpu().numpy().astype(np.float64) for x in (p, m, v))
    assert np.all(np.abs(gp - rp) <= 1e-6 * np.abs(rp) + 1e-4 * 6 * lr)
    assert np.all(np.abs(gm - rm) <= 1e-5 * np.abs(rm) + 1e-7 * np.abs(rm).max())
    assert np.all(np.abs(gv - rv) <= 1e-5 * np.abs(rv) + 1e-7 * np.abs(rv).max())
    if masked:
        sel = mask == 0
        assert np.array_equal(gp[sel], p0[sel]) and not gm[sel].any() and not gv[sel].any()


def test_adam_rejects_bad_arguments():
    simx = _simx()
    x = torch.zeros(8, device="cuda")
    for kw in (dict(t=0, lr=1e-3), dict(t=1, lr=-1.0), dict(t=1, lr=1e-3, beta1=1.0),
               dict(t=1, lr=1e-3, eps=0.0), dict(t=1, lr=1e-3, max_grad_norm=1.0)):
        with pytest.raises(simx.SimxError) as e:   # the last: clipping without a workspace
            simx.adam_step(x, x, x, x, **kw)
        assert e.value.status == simx.EINVAL


def test_empty_inputs():
    """Empty inputs: returns over T = 0 or E = 0 and a policy forward of 0 columns are
    no-ops; a loss over 0 rows, a baseline over 0 returns and an Adam step over 0
    parameters are refused with EINVAL."""
    simx = _simx()
    ret = torch.full((4, 8), 7.0, device="cuda")
    simx.compute_returns_gae(torch.zeros((0, 8), device="cuda"),
                             torch.zeros((0, 8), dtype=torch.uint8, device="cuda"), 0.99, -1.0,
                             ret[:0])
    simx.compute_returns_gae(torch.zeros((4, 0), device="cuda"),
                             torch.zeros((4, 0), dtype=torch.uint8, device="cuda"), 0.99, -1.0,
                             ret[:, :0])
    torch.cuda.synchronize()
    assert torch.all(ret == 7.0)
    ws = torch.empty(64, dtype=torch.uint8, device="cuda")
    with pytest.raises(simx.SimxError) as e:
        simx.returns_baseline(torch.zeros(0, device="cuda"), torch.zeros(0, device="cuda"),
                              torch.zeros(1, device="cuda"), ws)
    assert e.value.status == simx.EINVAL
    x = torch.zeros(0, device="cuda")
    with pytest.raises(simx.SimxError) as e:
        simx.adam_step(x, x, x, x, 1, 1e-3)
    assert e.value.status == simx.EINVAL
    cfg, pol, host, buf = _rollout_for_loss(simx, "c2", 5, 4)
    grad = torch.empty(pol.n_params, device="cuda")
    stats = torch.empty(5, device="cuda")
    lws = torch.empty(simx.ppo_loss_grad_workspace_size(pol, 1), dtype=torch.uint8, device="cuda")
    with pytest.raises(simx.SimxError) as e:
        simx.ppo_loss_grad(pol, buf, torch.zeros((4, 5), device="cuda"),
                           torch.zeros((4, 5), device="cuda"), None, 0, "reinforce", 0.2, 0.0, 0.0,
                           grad, stats, lws)
    assert e.value.status == simx.EINVAL
    obs = torch.zeros((pol.Ws[0].shape[1], 4), device="cuda")
    simx.policy_forward(pol, obs, 0, "argmax", 1, 0)
    torch.cuda.synchronize()
