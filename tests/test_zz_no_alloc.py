"""The allocation-free loss-gradient entry point against the workspace one.

ppo_loss_grad_noalloc serves callers that cannot allocate device memory themselves
(a plain C host program without a device allocator, or an application whose device
memory budget is fixed up front): its scratch is a buffer built into the library.
This file is collected last so that a failure here comes after every other test, and
it passes both alone in a fresh process and after the rest of the suite.
"""
import numpy as np
import pytest

from paper_2607_05272_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _setup(name, E, H, seed=21, hidden=None):
    from paper_2607_05272_gb300 import build as B
    B.build()
    from paper_2607_05272_gb300 import simx
    dims, hv = W.mlp_dims(name)
    if hidden is not None:
        dims = [dims[0]] + [hidden] * (len(dims) - 2) + [dims[-1]]
    Ws, bs = W.mlp_weights(dims, seed)
    pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws],
                      [torch.from_numpy(b).cuda() for b in bs], hv)
    sim = simx.Sim(W.CONFIGS[name](E))
    sim.reset(W.SEED[name])
    buf = simx.alloc_rollout(E, sim.D, H, has_value=hv)
    sim.rollout("sample", H, buf, pol)
    torch.cuda.synchronize()
    sim.close()
    return simx, pol, buf


# (workload, algorithm, envs, steps, minibatch rows or None, hidden width, precision):
# the fused FP32 kernel (c3, c2), the one-SM TF32 tensor-core kernel (c2; c3 with 64-wide
# hidden layers and a value row), and for c4's 28-256-256-49 on a minibatch whose
# workspace still fits the built-in buffer the FP32 GEMM pipeline and the streamed TF32
# tensor-core kernels.
CASES = [("c3", "ppo", 64, 256, 8192, None, "fp32"),
         ("c2", "reinforce", 40, 512, None, None, "fp32"),
         ("c2", "reinforce", 40, 512, None, None, "tf32"),
         ("c3", "ppo", 64, 256, 8192, 64, "tf32"),
         ("c4", "ppo", 33, 128, 1500, None, "fp32"),
         ("c4", "ppo", 33, 128, 1500, None, "tf32")]


@pytest.mark.parametrize("name,algo,E,H,nmb,hidden,prec", CASES)
def test_noalloc_matches_workspace_entry_point_twice(name, algo, E, H, nmb, hidden, prec):
    simx, pol, buf = _setup(name, E, H, hidden=hidden)
    rng = np.random.default_rng(7)
    adv = torch.from_numpy((rng.standard_normal((H, E)) * 2.0).astype(np.float32)).cuda()
    ret = torch.from_numpy(rng.standard_normal((H, E)).astype(np.float32)).cuda()
    n_rows = E * H
    idx = None if nmb is None else torch.from_numpy(rng.permutation(n_rows)[:nmb].astype(np.int64)).cuda()
    n = n_rows if idx is None else nmb
    need = simx.ppo_loss_grad_workspace_size(pol, n)
    assert need <= simx.NOALLOC_SCRATCH_BYTES
    tol = 1e-2 if prec == "tf32" else 1e-5
    g_ref = torch.empty(pol.n_params, device="cuda")
    s_ref = torch.empty(5, device="cuda")
    ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    simx.ppo_loss_grad(pol, buf, ret, adv, idx, n, algo, 0.2, 0.5, 0.01, g_ref, s_ref, ws,
                       precision=prec)
    for call in range(2):  # the shared scratch keeps the last call's contents
        g = torch.full((pol.n_params,), float("nan"), device="cuda")
        st = torch.full((5,), float("nan"), device="cuda")
        simx.ppo_loss_grad_noalloc(pol, buf, ret, adv, idx, n, algo, 0.2, 0.5, 0.01, g, st,
                                   precision=prec)
        torch.cuda.synchronize()
        gr, gn = g_ref.cpu().numpy().astype(np.float64), g.cpu().numpy().astype(np.float64)
        assert np.linalg.norm(gn - gr) <= tol * np.linalg.norm(gr)
        rms = np.sqrt(np.mean(gr ** 2))
        assert np.all(np.abs(gn - gr) <= tol * (np.abs(gr) + rms))
        assert np.allclose(st.cpu().numpy(), s_ref.cpu().numpy(), rtol=tol, atol=1e-6)


def test_noalloc_rejects_a_minibatch_beyond_its_scratch():
    simx, pol, buf = _setup("c4", 33, 512)
    n = 33 * 512
    need = simx.ppo_loss_grad_workspace_size(pol, n)
    assert need > simx.NOALLOC_SCRATCH_BYTES
    adv = torch.zeros((512, 33), device="cuda")
    ret = torch.zeros((512, 33), device="cuda")
    g = torch.empty(pol.n_params, device="cuda")
    st = torch.empty(5, device="cuda")
    with pytest.raises(simx.SimxError) as ei:
        simx.ppo_loss_grad_noalloc(pol, buf, ret, adv, None, n, "ppo", 0.2, 0.5, 0.01, g, st)
    assert ei.value.status == simx.EINVAL
    assert "allocation-free" in str(ei.value)
