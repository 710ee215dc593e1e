"""c1's fixed-batch-1 variant on the GPU against the M/D/1 closed form (Sec. 3.1).

c1's server (batch time 2000 + 100 n us) serving one request at a time is an M/D/1
queue with D = 2100 us; the Pollaczek-Khinchine mean wait in queue is
W_q = lambda D^2 / (2 (1 - rho)).  c1's own rate (800 req/s, rho = 1.68) is unstable, so
the check runs at 200 and 400 req/s (rho = 0.42 and 0.84) with a queue of 4096 (drops
negligible).  The whole rollout runs through rollout_collect (Static policy, the
thread-per-env step); sampled envs match the oracle bit for bit, and the mean wait over
every env after a 2000-decision warm-up is within 4 standard errors (across envs) and
3 % of W_q.
"""
import math

import numpy as np
import pytest

import oracle
from paper_2607_05272_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _simx():
    from paper_2607_05272_gb300 import build as B
    B.build()
    from paper_2607_05272_gb300 import simx
    return simx


@pytest.mark.parametrize("lam,H", [(200.0, 12000), (400.0, 40000)])
def test_md1_mean_wait_on_gpu(lam, H):
    simx = _simx()
    E, seed, warm = 1024, 0x3D1 + int(lam), 2000
    cfg = W.md1(lam, E)
    sim = simx.Sim(cfg)
    assert sim.launch_shape("static")["kernel"] == "thread"
    sim.reset(seed)
    buf = simx.alloc_rollout(E, sim.D, H, trace=True)
    sim.rollout("static", H, buf)
    torch.cuda.synchronize()
    st, code = sim.last_status()
    assert st == 0 and code == 0
    envs = [0, 1, 511, 1023]
    sel = torch.tensor(envs, device="cuda")
    got = {k: v.index_select(v.dim() - 1, sel).cpu().numpy() for k, v in buf.items()}
    state = sim.save()[envs]
    tr = buf["trace"][warm:, 1:3, :].to(torch.float64)
    n = tr[:, 0, :].sum(0)                  # requests dispatched (batch 1: 0 or 1 per step)
    w = tr[:, 1, :].sum(0)                  # their summed queueing microseconds
    per_env = (w / n).cpu().numpy()
    sim.close()
    ref = oracle.rollout(cfg, None, seed, 2, envs, H)
    assert np.array_equal(got["action"], ref["action"].astype(np.uint8))
    assert np.array_equal(got["trace"], ref["trace"])
    for k in ("obs", "reward"):
        assert np.array_equal(got[k].view(np.uint32), ref[k].view(np.uint32)), k
    assert np.array_equal(state, ref["state"])
    D = 2100.0
    rho = lam * D * 1e-6
    Wq = (lam * 1e-6) * D * D / (2.0 * (1.0 - rho))
    est, se = per_env.mean(), per_env.std(ddof=1) / math.sqrt(per_env.size)
    assert abs(est - Wq) < 4.0 * se, (est, Wq, se)
    assert abs(est - Wq) < 0.03 * Wq
