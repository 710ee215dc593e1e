"""Edge cases against the oracle: the largest configuration the ABI accepts, and the
simulated clock running past its limit.

* Maximum sizes: 8 servers, 2 request types, rings of 4096, 8 batch sizes (64 routing
  actions plus a value row), a 6-layer policy at the widest hidden layer (256), ragged
  env count: bit for bit, sampled policy and the Shortest-Queue step.
* Clock overflow (a degenerate case of the integer-time simulator): candidate gaps
  saturate at 2^26 us, so a 400 s mean gap carries the clock past 2^31 us within about 33
  arrivals; both sides raise the same time flag, freeze the same envs and keep the same
  state, on the MLP kernel and on the policy-free kernel.
"""
import numpy as np
import pytest

import oracle
from paper_2607_05272_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ORC_MODE = {"sample": 0, "argmax": 1, "static": 2, "rr": 3, "sq": 4, "random": 5}


def _simx():
    from paper_2607_05272_gb300 import build as B
    B.build()
    from paper_2607_05272_gb300 import simx
    return simx


def _run(simx, cfg, mode, H, seed, host=None):
    E = cfg["n_envs"]
    pol = None
    if host is not None:
        Ws, bs, hv = host
        pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws],
                          [torch.from_numpy(b).cuda() for b in bs], hv)
    sim = simx.Sim(cfg)
    sim.reset(seed)
    buf = simx.alloc_rollout(E, sim.D, H, has_value=bool(host and host[2]), trace=True)
    sim.rollout(mode, H, buf, pol)
    torch.cuda.synchronize()
    got = {k: v.cpu().numpy() for k, v in buf.items()}
    got["state"] = sim.save()
    st, code = sim.last_status()
    sim.close()
    ref = oracle.rollout(cfg, host, seed, ORC_MODE[mode], list(range(E)), H)
    return got, ref, st, code


def _same(got, ref, has_value):
    assert np.array_equal(got["action"], ref["action"].astype(np.uint8))
    assert np.array_equal(got["trace"], ref["trace"])
    assert np.array_equal(got["done"], ref["done"])
    for k in ("obs", "reward", "logp") + (("value",) if has_value else ()):
        assert np.array_equal(got[k].view(np.uint32), ref[k].view(np.uint32)), k
    assert np.array_equal(got["state"], ref["state"])


def _max_cfg(E):
    c = W.c4(E)
    c.update(queue_cap=4096, n_bsizes=8, bsizes=[1, 2, 4, 8, 16, 32, 48, 64], static_bi=3)
    return c


@pytest.mark.parametrize("mode", ["sample", "sq"])
def test_largest_configuration_matches_oracle(mode):
    simx = _simx()
    cfg = _max_cfg(37)
    host = None
    if mode == "sample":
        A = cfg["n_servers"] * cfg["n_bsizes"]
        dims = [cfg["obs_dim"], 256, 256, 256, 256, 256, A + 1]
        Ws, bs = W.mlp_weights(dims, 4)
        host = (Ws, bs, True)
    got, ref, st, code = _run(simx, cfg, mode, 128, 0xED6E, host)
    assert st == 0 and code == 0
    _same(got, ref, host is not None)


@pytest.mark.parametrize("mode", ["sample", "static"])
def test_clock_overflow_is_flagged_identically(mode):
    simx = _simx()
    cfg = W.c1(21)
    cfg.update(cand_mean_gap_us=4.0e8, episode_len=1 << 30)
    host = None
    if mode == "sample":
        dims, hv = W.mlp_dims("c1")
        Ws, bs = W.mlp_weights(dims, 6)
        host = (Ws, bs, hv)
    got, ref, st, code = _run(simx, cfg, mode, 60, 0x0F10, host)
    assert st == simx.EOVERFLOW and code & 1          # the time flag
    flags = got["state"][:, 28]
    assert np.all(flags & 1)                          # every env ran out of clock
    _same(got, ref, False)
