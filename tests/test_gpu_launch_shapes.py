"""Parity at the launch shapes the large configurations run (Sec. 3.1, 3.2, 4.1-4.3).

The fused step's lanes per env and threads per block follow the env count; the
library reports the choice (simx_launch_shape) and each case asserts the shape it
means to cover before comparing:

* c3 at 16,384 envs: 8 lanes per env, 128-thread blocks (16 envs per block), the
  block-wide policy forward over 13-128-128-17 with its weights staged in shared memory
  (as in every fused case here: their weights are 82 KB and more);
* c4 at 65,536 envs: 8 lanes, 256-thread blocks (32 envs per block), 28-256-256-49,
  diurnal x lognormal arrivals and Pareto costs, the full 512-step horizon;
* c5 (argmax) at 262,144 and 1,048,576 envs x 1024 steps, 8 lanes, 256 threads; at
  1,048,576 envs the observation buffer holds more than 2^32 floats;
* the thread-per-env policy-free step (Shortest-Queue router) at 262,144 and
  1,048,576 envs;
* the one-pass four-envs-per-thread returns kernel at 65,536 and 262,144 envs
  (REINFORCE and GAE, horizons that are not a multiple of its 8-step lookahead, done
  flags and bootstrap values), and 262,145 envs, which takes the chunked kernel.

The oracle reproduces any single env from (seed, env id), so the rollouts are
compared on sampled envs: {0, 1, 31, 32, 33, E/2 - 1, E/2, E - 1} (block and warp
edges) and 64 ids drawn from Philox, bit for bit on actions, per-step traces, done
flags, observations, rewards, log-probabilities, values and the final env state.
The returns are compared on every element under the recurrence bound of
test_gpu_rl.py.
"""
import numpy as np
import pytest

import oracle
from oracle import rl
from paper_2607_05272_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ORC_MODE = {"sample": 0, "argmax": 1, "sq": 4}


def _simx():
    from paper_2607_05272_gb300 import build as B
    B.build()
    from paper_2607_05272_gb300 import simx
    return simx


def _env_sample(E, seed):
    edges = [0, 1, 31, 32, 33, E // 2 - 1, E // 2, E - 1]
    drawn = (oracle.philox_n(0, 0, 7, seed, 16).ravel().astype(np.int64) % E).tolist()
    return sorted(set(e for e in edges + drawn if 0 <= e < E))


def _policy(simx, name):
    dims, hv = W.mlp_dims(name)
    Ws, bs = W.policy_weights(name, dims, 7)
    pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws],
                      [torch.from_numpy(b).cuda() for b in bs], hv)
    return pol, (Ws, bs, hv, None)


def _run_sampled(name, E, H, mode, shape, with_state=True):
    simx = _simx()
    cfg = W.CONFIGS[name](E)
    net = mode in ("sample", "argmax")
    pol, host = _policy(simx, name) if net else (None, None)
    sim = simx.Sim(cfg)
    assert sim.launch_shape(mode, pol) == shape
    sim.reset(W.SEED[name])
    buf = simx.alloc_rollout(E, sim.D, H, has_value=bool(net and host[2]), trace=True)
    sim.rollout(mode, H, buf, pol)
    torch.cuda.synchronize()
    st, code = sim.last_status()
    assert st == 0 and code == 0
    envs = _env_sample(E, W.SEED[name])
    sel = torch.tensor(envs, device="cuda")
    got = {k: v.index_select(v.dim() - 1, sel).cpu().numpy() for k, v in buf.items()}
    del buf
    state = sim.save()[envs] if with_state else None
    sim.close()
    torch.cuda.empty_cache()
    ref = oracle.rollout(cfg, host, W.SEED[name], ORC_MODE[mode], envs, H)
    assert np.array_equal(got["action"], ref["action"].astype(np.uint8))
    assert np.array_equal(got["trace"], ref["trace"])
    assert np.array_equal(got["done"], ref["done"])
    keys = ["obs", "reward"] + (["logp"] if net else []) + (["value"] if net and host[2] else [])
    for k in keys:
        assert np.array_equal(got[k].view(np.uint32), ref[k].view(np.uint32)), k
    if with_state:
        assert np.array_equal(state, ref["state"])


FUSED = dict(kernel="fused", lanes=8, mlp_warp=False, tensor_cores=False, staged=True)


def test_c3_16384_envs_128_thread_blocks():
    _run_sampled("c3", 16384, W.HORIZON["c3"], "sample", dict(FUSED, threads=128))


def test_c4_65536_envs_256_thread_blocks():
    _run_sampled("c4", 65536, W.HORIZON["c4"], "sample", dict(FUSED, threads=256))


def test_c5_argmax_262144_envs():
    _run_sampled("c5", 262144, W.HORIZON["c5"], "argmax", dict(FUSED, threads=256))


def test_c5_argmax_1048576_envs():
    # the final state image of a million envs is 8.8 GB: records and traces only
    _run_sampled("c5", 1048576, W.HORIZON["c5"], "argmax", dict(FUSED, threads=256),
                 with_state=False)


THREAD = dict(kernel="thread", lanes=1, threads=128, mlp_warp=False, tensor_cores=False,
              staged=False)


@pytest.mark.parametrize("E,H,state", [(262144, 256, True), (1048576, 64, False)])
def test_policy_free_step_large(E, H, state):
    _run_sampled("c5", E, H, "sq", THREAD, with_state=state)


def _check_recurrence(x, ref, scale):
    x = x.astype(np.float64)
    assert np.all(np.abs(x - ref) <= 1e-5 * (np.abs(ref) + scale) + 1e-30)
    assert np.linalg.norm(x - ref) <= 1e-5 * np.linalg.norm(ref)


@pytest.mark.parametrize("T,E", [(13, 65536), (101, 262144), (7, 262145)])
@pytest.mark.parametrize("gae", [False, True], ids=["reinforce", "gae"])
def test_returns_wide_sizes(T, E, gae):
    simx = _simx()
    rng = np.random.default_rng(T * 31 + E + gae)
    r = (rng.standard_normal((T, E)) * 2.0 - 0.5).astype(np.float32)
    v = rng.standard_normal((T, E)).astype(np.float32)
    d = (rng.random((T, E)) < 0.05).astype(np.uint8)
    last = rng.standard_normal(E).astype(np.float32)
    ret = torch.empty((T, E), device="cuda")
    adv = torch.empty((T, E), device="cuda")
    dev = lambda x: torch.from_numpy(x).cuda()
    if gae:
        simx.compute_returns_gae(dev(r), dev(d), 0.99, 0.95, ret, adv=adv, val=dev(v),
                                 last_val=dev(last))
    else:
        simx.compute_returns_gae(dev(r), dev(d), 0.99, -1.0, ret, last_val=dev(last))
    torch.cuda.synchronize()
    if gae:
        A, R = rl.gae(r, v, d, 0.99, 0.95, last)
        vn = np.vstack([v[1:], last[None]]).astype(np.float64)
        absd = np.abs(r) + 0.99 * np.abs(vn) + np.abs(v)
        scale = rl.returns(absd, d, 0.99 * 0.95)
        _check_recurrence(adv.cpu().numpy(), A, scale)
        _check_recurrence(ret.cpu().numpy(), R, scale + np.abs(v))
    else:
        G = rl.returns(r, d, 0.99, last)
        scale = rl.returns(np.abs(r), d, 0.99, np.abs(last))
        _check_recurrence(ret.cpu().numpy(), G, scale)
