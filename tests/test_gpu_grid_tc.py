"""The grid policy's forward on the tensor cores inside the fused step (the exact policy
forward: tcgen05.mma kind::f16 with bf16 operands and FP32 accumulation), against the
oracle's definition (the exact dot product) and against the FP32 FMA tiles.

On the grid every operand is exact in bf16 and every partial sum stays below 2^24
product units, so the tensor core's sums must be the exact ones: the same bits as the
FP32 chains and as the oracle's fp64 sums rounded once.  Checked at the launch shapes
that take it (blocks of 128 or 256 threads, the block-wide forward):

* c3's router at 16,384 envs (16 envs per block) and c5 (argmax) at 65,536 envs (32 per
  block): sampled envs bit for bit against the oracle (actions, traces, observations,
  rewards, log-probabilities, values, final state), and every env of the rollout bit for
  bit against the same launch on the FP32 tiles (SIMX_TC_FORWARD=0);
* the paper's network (identity and GELU layers, 8-4-4-4-128-34) in blocks of 256;
* the premise's worst case in a rollout: a 13-256-17 policy whose hidden layer is
  saturated at +-255 units feeding an output layer with every mantissa at +-255 and the
  largest bias, so the tensor core sums 256 products of 255 x 255 units to
  256 x 255^2 + 2^16 < 2^24 units: the value row must be that sum exactly at every step.
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


def _env_sample(E, seed):
    edges = [0, 1, 15, 16, 31, 32, 33, E // 2 - 1, E // 2, E - 1]
    drawn = (oracle.philox_n(0, 0, 9, seed, 8).ravel().astype(np.int64) % E).tolist()
    return sorted(set(e for e in edges + drawn if 0 <= e < E))


def _grid_policy(name, seed=21):
    dims, hv = W.mlp_dims(name)
    acts = W.mlp_acts(name)
    gx = [5] + [7] * (len(dims) - 2)
    ew = [8] * (len(dims) - 1)
    Ws, bs = W.grid_weights(dims, seed, gx, ew)
    W.grid_check(Ws, bs, gx, ew)
    return Ws, bs, hv, acts, gx


def _rollout(simx, cfg, host, mode, H, seed, tc, monkeypatch):
    Ws, bs, hv, acts, gx = host
    monkeypatch.setenv("SIMX_TC_FORWARD", "1" if tc else "0")
    pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws],
                      [torch.from_numpy(b).cuda() for b in bs], hv, acts, grid=gx)
    sim = simx.Sim(cfg)
    shape = sim.launch_shape(mode, pol)
    sim.reset(seed)
    buf = simx.alloc_rollout(cfg["n_envs"], sim.D, H, has_value=hv, trace=True)
    sim.rollout(mode, H, buf, pol)
    torch.cuda.synchronize()
    st, code = sim.last_status()
    state = sim.save()
    sim.close()
    assert st == 0 and code == 0
    return shape, buf, state


CASES = [("c3", 16384, 64, "sample", None, 128), ("c5", 65536, 48, "argmax", None, 256),
         ("c1p", 4096, 200, "sample", "256", 256)]


@pytest.mark.parametrize("name,E,H,mode,threads,expect", CASES, ids=[c[0] for c in CASES])
def test_tensor_core_grid_rollout(name, E, H, mode, threads, expect, monkeypatch):
    simx = _simx()
    if threads:
        monkeypatch.setenv("SIMX_THREADS", threads)
    cfg = W.CONFIGS[name](E)
    host = _grid_policy(name)
    seed = 0x6A1D + E
    shape, buf, state = _rollout(simx, cfg, host, mode, H, seed, True, monkeypatch)
    assert shape["tensor_cores"] and shape["threads"] == expect and not shape["mlp_warp"]
    shape0, buf0, state0 = _rollout(simx, cfg, host, mode, H, seed, False, monkeypatch)
    assert not shape0["tensor_cores"]
    # every env: the tensor-core sums are the FP32 chains' bits
    for k in buf:
        assert torch.equal(buf[k], buf0[k]), k
    assert np.array_equal(state, state0)
    # sampled envs: the oracle's exact dot products
    envs = _env_sample(E, seed)
    sel = torch.tensor(envs, device="cuda")
    got = {k: v.index_select(v.dim() - 1, sel).cpu().numpy() for k, v in buf.items()}
    ref = oracle.rollout(cfg, host, seed, ORC_MODE[mode], envs, H)
    assert np.array_equal(got["action"], ref["action"].astype(np.uint8))
    assert np.array_equal(got["trace"], ref["trace"])
    for k in ("obs", "reward", "logp") + (("value",) if host[2] else ()):
        assert np.array_equal(got[k].view(np.uint32), ref[k].view(np.uint32)), k
    assert np.array_equal(state[envs], ref["state"])
    assert len(np.unique(got["action"])) > 1


def test_tensor_core_grid_worst_case(monkeypatch):
    simx = _simx()
    E, H, D, Hd, A = 65536, 32, 13, 256, 16
    gx, ew = [5, 8], [8, 8]
    rng = np.random.default_rng(8)
    sgn = rng.choice([-1, 1], Hd)
    W0 = np.zeros((Hd, D), np.float32)
    # bias 2^16 product units = 8.0: tanh(+-8) rounds to +-256 units, clamped to +-255
    b0 = np.ldexp(sgn.astype(np.float64) * (1 << 16), -(gx[0] + ew[0])).astype(np.float32)
    m1 = rng.integers(-255, 256, (A + 1, Hd))
    m1[0] = sgn * 255
    m1[A] = sgn * 255                 # the value row: +255 x 255 units in every term
    mb1 = rng.integers(-(1 << 16), (1 << 16) + 1, A + 1)
    mb1[0] = mb1[A] = 1 << 16
    W1 = np.ldexp(m1.astype(np.float64), -ew[1]).astype(np.float32)
    b1 = np.ldexp(mb1.astype(np.float64), -(gx[1] + ew[1])).astype(np.float32)
    Ws, bs = [W0, W1], [b0, b1]
    W.grid_check(Ws, bs, gx, ew)
    host = (Ws, bs, True, None, gx)
    cfg = W.c5(E)
    shape, buf, state = _rollout(simx, cfg, host, "argmax", H, 77, True, monkeypatch)
    assert shape["tensor_cores"]
    top = np.float32(np.ldexp(256.0 * 255 * 255 + (1 << 16), -(gx[1] + ew[1])))
    assert 256 * 255 * 255 + (1 << 16) < 1 << 24
    assert torch.all(buf["value"] == float(top))
    assert torch.all(buf["action"] == 0)          # row 0 holds the largest logit
    envs = _env_sample(E, 77)
    sel = torch.tensor(envs, device="cuda")
    got = {k: v.index_select(v.dim() - 1, sel).cpu().numpy() for k, v in buf.items()}
    ref = oracle.rollout(cfg, host, 77, ORC_MODE["argmax"], envs, H)
    for k in ("obs", "reward", "logp", "value"):
        assert np.array_equal(got[k].view(np.uint32), ref[k].view(np.uint32)), k
    assert np.array_equal(state[envs], ref["state"])
