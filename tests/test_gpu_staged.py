"""The block-wide FP32 policy forward with its weights streamed through shared memory
(Sec. 4.2 policy inside the fused step): one thread keeps two stages of weight rows in
flight with bulk copies, every thread runs a register tile of up to 4 envs x 8 outputs.

Every output is still the fma chain from 0 over k in order, then + bias, the activation
and (grid policies) the grid rounding, so the staged launch must give the unstaged
launch's bits (SIMX_STAGE=0) on every env, and the oracle's on sampled envs (actions,
traces, done flags, observations, rewards, log-probabilities, values, final state).
Each case asserts the launch shape it means to cover:

* c4 at 65,536 envs (4x8 tiles for the 256-wide layers, 2x4 for the 49 outputs; 256-thread
  blocks), 64 steps;
* c3 at 16,384 envs (2x8 tiles, 1x4 for the 17 outputs; 128-thread blocks);
* the paper's network (c1p: identity and GELU layers, five layers down to 4 wide) with
  staging forced on small weights, in 256-thread blocks;
* a c3 grid policy with staging forced and the tensor-core forward off: the grid
  rounding in the staged epilogue;
* c4 at 1,003 envs in 128-thread blocks (8 lanes, 4 KB stages): a last block with 11
  envs;
* c4 at 65,536 envs with 16 lanes per env (2x8 tiles, 1x4 for the 49 outputs, 16 envs per
  256-thread block);
* c3t, trace replay (gaps, types and costs from a trace), at 16,384 envs;
* single steps (sim_step_batched: one launch per step, so the weight pipeline starts and
  drains every launch) against rollout_collect, c4 at 4,096 envs in 256-thread blocks.
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
    edges = [0, 1, 7, 8, 31, 32, 33, E // 2 - 1, E // 2, E - 1]
    drawn = (oracle.philox_n(0, 0, 11, seed, 8).ravel().astype(np.int64) % E).tolist()
    return sorted(set(e for e in edges + drawn if 0 <= e < E))


def _host(name, grid):
    dims, hv = W.mlp_dims(name)
    acts = W.mlp_acts(name)
    if grid:
        gx = [5] + [7] * (len(dims) - 2)
        ew = [8] * (len(dims) - 1)
        Ws, bs = W.grid_weights(dims, 23, gx, ew)
        W.grid_check(Ws, bs, gx, ew)
        return Ws, bs, hv, acts, gx
    Ws, bs = W.policy_weights(name, dims, 7)
    return Ws, bs, hv, acts, None


def _rollout(simx, cfg, host, mode, H, seed, stage, monkeypatch):
    Ws, bs, hv, acts, gx = host
    if stage:
        monkeypatch.setenv("SIMX_STAGE", stage)
    else:
        monkeypatch.delenv("SIMX_STAGE", raising=False)
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


# name, envs, steps, mode, grid policy, SIMX_THREADS, SIMX_LANES, SIMX_STAGE, threads
CASES = [
    ("c4", 65536, 64, "sample", False, None, None, "", 256),
    ("c3", 16384, 96, "sample", False, None, None, "", 128),
    ("c1p", 4096, 300, "sample", False, "256", None, "1", 256),
    ("c3", 16384, 64, "argmax", True, None, None, "1", 128),
    ("c4", 1003, 200, "sample", False, "128", "8", "", 128),
    ("c4", 65536, 32, "sample", False, None, "16", "", 256),
    ("c3t", 16384, 64, "sample", False, None, None, "", 128),
]


@pytest.mark.parametrize("name,E,H,mode,grid,threads,lanes,stage,expect", CASES,
                         ids=["c4", "c3", "c1p-forced", "c3-grid-forced", "c4-ragged", "c4-16-lanes",
                              "c3t"])
def test_staged_forward(name, E, H, mode, grid, threads, lanes, stage, expect, monkeypatch):
    simx = _simx()
    if threads:
        monkeypatch.setenv("SIMX_THREADS", threads)
    if lanes:
        monkeypatch.setenv("SIMX_LANES", lanes)
    monkeypatch.setenv("SIMX_TC_FORWARD", "0")
    cfg = W.CONFIGS[name](E)
    host = _host(name, grid)
    seed = 0x57A6 + E
    shape, buf, state = _rollout(simx, cfg, host, mode, H, seed, stage, monkeypatch)
    assert shape["kernel"] == "fused" and shape["threads"] == expect and not shape["mlp_warp"]
    assert shape["staged"] and not shape["tensor_cores"]
    shape0, buf0, state0 = _rollout(simx, cfg, host, mode, H, seed, "0", monkeypatch)
    assert not shape0["staged"]
    # every env: the unstaged forward's bits
    for k in buf:
        assert torch.equal(buf[k], buf0[k]), k
    assert np.array_equal(state, state0)
    # sampled envs: the oracle's fma chains
    envs = _env_sample(E, seed)
    sel = torch.tensor(envs, device="cuda")
    got = {k: v.index_select(v.dim() - 1, sel).cpu().numpy() for k, v in buf.items()}
    ref = oracle.rollout(cfg, host, seed, ORC_MODE[mode], envs, H)
    assert np.array_equal(got["action"], ref["action"].astype(np.uint8))
    assert np.array_equal(got["trace"], ref["trace"])
    assert np.array_equal(got["done"], ref["done"])
    for k in ("obs", "reward", "logp") + (("value",) if host[2] else ()):
        assert np.array_equal(got[k].view(np.uint32), ref[k].view(np.uint32)), k
    assert np.array_equal(state[envs], ref["state"])
    assert len(np.unique(got["action"])) > 1


def test_staged_single_steps_equal_the_rollout(monkeypatch):
    simx = _simx()
    monkeypatch.setenv("SIMX_LANES", "8")
    monkeypatch.setenv("SIMX_THREADS", "256")
    monkeypatch.delenv("SIMX_STAGE", raising=False)
    E, H = 4096, 24
    cfg = W.c4(E)
    Ws, bs, hv, acts, _ = _host("c4", False)
    pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws],
                      [torch.from_numpy(b).cuda() for b in bs], hv, acts)
    seed = 0x57E9
    sim = simx.Sim(cfg)
    shape = sim.launch_shape("sample", pol)
    assert shape["staged"] and shape["threads"] == 256 and shape["lanes"] == 8
    sim.reset(seed)
    buf = simx.alloc_rollout(E, sim.D, H, has_value=hv)
    sim.rollout("sample", H, buf, pol)
    torch.cuda.synchronize()
    state_r = sim.save()
    sim.close()
    sim = simx.Sim(cfg)
    sim.reset(seed)
    rew = torch.empty((H, E), device="cuda")
    done = torch.empty((H, E), dtype=torch.uint8, device="cuda")
    act = torch.empty((H, E), dtype=torch.uint8, device="cuda")
    lp = torch.empty((H, E), device="cuda")
    obs = torch.empty((H, sim.D, E), device="cuda")
    for t in range(H):
        sim.step("sample", pol, obs=obs[t], reward=rew[t], done=done[t], action=act[t], logp=lp[t])
    torch.cuda.synchronize()
    st, code = sim.last_status()
    assert st == 0 and code == 0
    assert torch.equal(act, buf["action"]) and torch.equal(done, buf["done"])
    assert torch.equal(rew.view(torch.int32), buf["reward"].view(torch.int32))
    assert torch.equal(lp.view(torch.int32), buf["logp"].view(torch.int32))
    # a step writes the observation after it, the rollout the one before each step
    assert torch.equal(obs[:-1].view(torch.int32), buf["obs"][1:].view(torch.int32))
    assert np.array_equal(sim.save(), state_r)
    sim.close()
