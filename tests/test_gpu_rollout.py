"""GPU parity of the simulator and fused policy (Sec. 3.1, 3.2, 4.1, 4.2) with the oracle.

Every case runs the CUDA path through the C ABI and the oracle on the same seeded
inputs; integer state (decision times, queue contents, per-step dispatch counts and
queueing sums, counters, RNG positions) and actions must match bit for bit, and so
must the fp32 observations, log-probabilities, values and rewards, because both
sides evaluate them with the same operation order.  Env counts are ragged (not a
multiple of the 32 envs a block owns) so partial blocks and warps are covered.
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


def _policy(simx, name, seed=7):
    dims, hv = W.mlp_dims(name)
    Ws, bs = W.policy_weights(name, dims, seed)
    acts = W.mlp_acts(name)
    pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws],
                      [torch.from_numpy(b).cuda() for b in bs], hv, acts)
    return pol, (Ws, bs, hv, acts)


def _run(name, cfg, H, mode, seed=None, trace=True):
    simx = _simx()
    seed = W.SEED[name] if seed is None else seed
    E = cfg["n_envs"]
    pol, host = _policy(simx, name) if mode in ("sample", "argmax") else (None, None)
    sim = simx.Sim(cfg)
    sim.reset(seed)
    buf = simx.alloc_rollout(E, sim.D, H, has_value=bool(host and host[2]), trace=trace)
    sim.rollout(mode, H, buf, pol)
    torch.cuda.synchronize()
    got = {k: v.cpu().numpy() for k, v in buf.items()}
    got["state"] = sim.save()
    st, code = sim.last_status()
    sim.close()
    ref = oracle.rollout(cfg, host, seed, ORC_MODE[mode], list(range(E)), H)
    return got, ref, st, code


def _assert_same(got, ref, has_value):
    assert np.array_equal(got["action"], ref["action"].astype(np.uint8))
    assert np.array_equal(got["trace"], ref["trace"])
    assert np.array_equal(got["done"], ref["done"])
    assert np.array_equal(got["obs"].view(np.uint32), ref["obs"].view(np.uint32))
    assert np.array_equal(got["reward"].view(np.uint32), ref["reward"].view(np.uint32))
    assert np.array_equal(got["logp"].view(np.uint32), ref["logp"].view(np.uint32))
    if has_value:
        assert np.array_equal(got["value"].view(np.uint32), ref["value"].view(np.uint32))
    assert np.array_equal(got["state"], ref["state"])


CASES = [
    ("c1", lambda: W.c1(64), 10000, "sample"),   # the full c1 workload
    ("c2", lambda: W.c2(37), 512, "sample"),
    ("c3", lambda: W.c3(45), 256, "sample"),
    ("c4", lambda: W.c4(21), 512, "sample"),
    ("c5", lambda: W.c5(40), 1024, "argmax"),
    ("burst", lambda: W.burst(37), 2000, "sample"),  # square-wave arrivals (fixed dwell)
    ("c3h", lambda: W.c3h(45), 256, "sample"),        # heterogeneous server speeds
    ("c1w", lambda: W.c1w(33), 2000, "sample"),       # Wait + batch 1..32: 33 actions
    ("c2w", lambda: W.c2w(37), 512, "sample"),        # Wait + (type, batch 1..32): 65
    ("c1p", lambda: W.c1p(41), 2000, "sample"),       # the paper's network (GELU heads)
    ("c2t", lambda: W.c2t(37), 512, "sample"),        # trace replay: gaps and types
    ("c3t", lambda: W.c3t(45), 256, "sample"),        # trace replay: gaps, types, costs
]


@pytest.mark.parametrize("name,mk,H,mode", CASES, ids=[c[0] for c in CASES])
def test_rollout_matches_oracle(name, mk, H, mode):
    got, ref, st, code = _run(name, mk(), H, mode)
    assert st == 0 and code == 0
    _assert_same(got, ref, W.MLP_SHAPES[name][1])


@pytest.mark.parametrize("lanes", [8, 16, 32])
@pytest.mark.parametrize("name,mk,H,mode", [c for c in CASES if c[0] != "c1"] +
                         [("c1", lambda: W.c1(23), 1500, "sample")],
                         ids=[c[0] for c in CASES if c[0] != "c1"] + ["c1"])
def test_rollout_every_lane_width(name, mk, H, mode, lanes, monkeypatch):
    """The same results whichever number of lanes (8, 16, 32) serves an env."""
    monkeypatch.setenv("SIMX_LANES", str(lanes))
    got, ref, st, code = _run(name, mk(), min(H, 300), mode)
    assert st == 0 and code == 0
    _assert_same(got, ref, W.MLP_SHAPES[name][1])


BASELINES = [
    ("c1", lambda: W.c1(33), 2000, "static"),
    ("c2", lambda: W.c2(33), 512, "static"),
    ("c2", lambda: W.c2(35), 256, "random"),
    ("c3", lambda: W.c3(70), 256, "sq"),
    ("c3", lambda: W.c3(33), 256, "rr"),
    ("c3", lambda: W.c3(33), 256, "random"),
    ("c4", lambda: W.c4(33), 512, "sq"),
    ("burst", lambda: W.burst(35), 2000, "static"),
    ("c3h", lambda: W.c3h(41), 256, "sq"),
    ("c3h", lambda: W.c3h(39), 256, "rr"),
    ("c2w", lambda: W.c2w(34), 512, "static"),
    ("c1w", lambda: W.c1w(30), 2000, "random"),
    ("c2t", lambda: W.c2t(33), 512, "static"),
    ("c3t", lambda: W.c3t(41), 256, "sq"),
    ("c3t", lambda: W.c3t(35), 256, "random"),
]


@pytest.mark.parametrize("name,mk,H,mode", BASELINES, ids=["%s-%s" % (c[0], c[3]) for c in BASELINES])
def test_policy_free_baselines_match_oracle(name, mk, H, mode):
    got, ref, st, code = _run(name, mk(), H, mode)
    assert st == 0
    _assert_same(got, ref, False)


def test_single_env_and_zero_horizon():
    simx = _simx()
    got, ref, st, _ = _run("c3", W.c3(1), 200, "sample")
    _assert_same(got, ref, True)
    sim = simx.Sim(W.c2(5))
    sim.reset(3)
    before = sim.save()
    buf = simx.alloc_rollout(5, sim.D, 1)
    sim.rollout("static", 0, buf)
    assert np.array_equal(sim.save(), before)


@pytest.mark.parametrize("name,mk", [("c2", lambda: W.c2(36)), ("c4", lambda: W.c4(13)),
                                     ("c3h", lambda: W.c3h(17)), ("c1p", lambda: W.c1p(19))])
def test_step_batched_equals_rollout(name, mk):
    """H single-step launches with the internal policy give the rollout's records."""
    simx = _simx()
    cfg = mk()
    E, H = cfg["n_envs"], 40
    pol, host = _policy(simx, name)
    sim = simx.Sim(cfg)
    sim.reset(W.SEED[name])
    D = sim.D
    obs0 = torch.empty((D, E), device="cuda")
    sim.observe(obs0)
    obs = torch.empty((H, D, E), device="cuda")
    rew = torch.empty((H, E), device="cuda")
    done = torch.empty((H, E), dtype=torch.uint8, device="cuda")
    act = torch.empty((H, E), dtype=torch.uint8, device="cuda")
    lp = torch.empty((H, E), device="cuda")
    for t in range(H):
        sim.step("sample", pol, obs=obs[t], reward=rew[t], done=done[t], action=act[t], logp=lp[t])
    torch.cuda.synchronize()
    ref = oracle.rollout(cfg, host, W.SEED[name], 0, list(range(E)), H + 1)
    assert np.array_equal(obs0.cpu().numpy(), ref["obs"][0])
    assert np.array_equal(obs.cpu().numpy(), ref["obs"][1:])
    assert np.array_equal(act.cpu().numpy(), ref["action"][:H].astype(np.uint8))
    assert np.array_equal(rew.cpu().numpy().view(np.uint32), ref["reward"][:H].view(np.uint32))
    assert np.array_equal(lp.cpu().numpy().view(np.uint32), ref["logp"][:H].view(np.uint32))
    assert np.array_equal(done.cpu().numpy(), ref["done"][:H])
    sim.close()


@pytest.mark.parametrize("name,mk", [("c1", lambda: W.c1(9)), ("c2", lambda: W.c2(17)),
                                     ("c3", lambda: W.c3(19)), ("c4", lambda: W.c4(11)),
                                     ("c2w", lambda: W.c2w(15)), ("c3t", lambda: W.c3t(13))])
def test_external_actions_match_oracle(name, mk):
    simx = _simx()
    cfg = mk()
    E, H = cfg["n_envs"], 60
    A = (cfg["n_types"] if cfg["mode"] == 0 else cfg["n_servers"]) * cfg["n_bsizes"] + cfg["action_layout"]
    rng = np.random.default_rng(5)
    acts = rng.integers(0, A, size=(H, E)).astype(np.int32)
    sim = simx.Sim(cfg)
    sim.reset(11)
    rew = torch.empty((H, E), device="cuda")
    obs = torch.empty((H, sim.D, E), device="cuda")
    for t in range(H):
        sim.step("external", actions=torch.from_numpy(acts[t]).cuda(), obs=obs[t], reward=rew[t])
    torch.cuda.synchronize()
    st = sim.save()
    envs = [oracle.OracleEnv(cfg, e, 11) for e in range(E)]
    for e in envs:
        e.reset()
    r_ref = np.zeros((H, E), np.float32)
    o_ref = np.zeros((H, sim.D, E), np.float32)
    for t in range(H):
        for i, e in enumerate(envs):
            r_ref[t, i] = e.step(6, None, int(acts[t, i]))["reward"]
            o_ref[t, :, i] = e.observe()
    assert np.array_equal(rew.cpu().numpy().view(np.uint32), r_ref.view(np.uint32))
    assert np.array_equal(obs.cpu().numpy(), o_ref)
    for i, e in enumerate(envs):
        assert np.array_equal(st[i], e.export())
    sim.close()


def test_bad_external_action_sets_status():
    simx = _simx()
    sim = simx.Sim(W.c3(8))
    sim.reset(1)
    a = torch.zeros(8, dtype=torch.int32, device="cuda")
    a[3] = 99
    sim.step("external", actions=a)
    st, code = sim.last_status()
    assert st == simx.EOVERFLOW and code & 4
    assert sim.stats()["envs_flagged"] == 1
    sim.close()


@pytest.mark.parametrize("name,mk,H", [("c2", lambda: W.c2(21), 300), ("c4", lambda: W.c4(19), 300),
                                      ("c3t", lambda: W.c3t(23), 200)])
def test_save_load_resume_is_bit_exact(name, mk, H):
    simx = _simx()
    cfg = mk()
    E = cfg["n_envs"]
    pol, host = _policy(simx, name)
    hv = bool(host[2])
    a = simx.Sim(cfg)
    a.reset(77)
    full = simx.alloc_rollout(E, a.D, H, has_value=hv, trace=True)
    a.rollout("sample", H, full, pol)
    torch.cuda.synchronize()
    b = simx.Sim(cfg)
    b.reset(77)
    h1 = simx.alloc_rollout(E, b.D, H // 2, has_value=hv, trace=True)
    b.rollout("sample", H // 2, h1, pol)
    img = b.save()
    b.close()
    c = simx.Sim(cfg)
    c.reset(77)
    c.load(img)
    h2 = simx.alloc_rollout(E, c.D, H - H // 2, has_value=hv, trace=True)
    c.rollout("sample", H - H // 2, h2, pol)
    torch.cuda.synchronize()
    for k in full:
        joined = torch.cat([h1[k], h2[k]], 0)
        assert torch.equal(full[k], joined), k
    assert np.array_equal(a.save(), c.save())


def _tiny_trace_cfg(E, with_costs):
    gap = np.array([5, 0, 12, 3, 100, 7, 1, 0, 0, 40, 2], np.uint32)
    typ = np.array([0, 1, 1, 0, 5, 0, 1, 1, 0, 0, 1], np.uint8)   # 5: the last type
    cost = np.array([11, 22, 33, 44, 55, 66, 77, 88, 99, 1, 0], np.uint32)
    cfg = W.c3t(E)
    cfg["trace"] = (gap, typ, cost if with_costs else None)
    return cfg


@pytest.mark.parametrize("mode", ["sample", "sq"])
@pytest.mark.parametrize("with_costs", [True, False])
def test_short_trace_wraps_like_the_oracle(mode, with_costs):
    """An 11-entry trace with zero gaps and an out-of-range type, replayed hundreds of
    times over by every env from its own starting entry."""
    got, ref, st, code = _run("c3t", _tiny_trace_cfg(43, with_costs), 300, mode)
    assert st == 0 and code == 0
    _assert_same(got, ref, mode == "sample")


def test_trace_call_order_and_arguments():
    simx = _simx()
    g = torch.ones(4, dtype=torch.int32, device="cuda")
    plain = simx.Sim(W.c3(8))
    with pytest.raises(simx.SimxError) as e:   # not a trace workload
        plain.set_trace(g)
    assert e.value.status == simx.EINVAL
    plain.close()
    cfg = W.c3t(8)
    cfg["trace"] = None
    sim = simx.Sim(cfg)
    with pytest.raises(simx.SimxError) as e:   # reset before any trace
        sim.reset(1)
    assert e.value.status == simx.ESTATE
    with pytest.raises(simx.SimxError) as e:   # empty trace
        sim.set_trace(g[:0])
    assert e.value.status == simx.EINVAL
    sim.set_trace(g)
    sim.reset(1)
    sim.close()


@pytest.mark.parametrize("with_ws", [False, True])
def test_policy_forward_matches_oracle(with_ws):
    """Both entries (the library's repack buffer, or a caller workspace) against the oracle."""
    simx = _simx()
    for name, mode in (("c3", "sample"), ("c4", "argmax"), ("c2", "sample"), ("c1p", "sample")):
        pol, host = _policy(simx, name, seed=3)
        D = host[0][0].shape[1]
        n = 77
        rng = np.random.default_rng(2)
        obs = rng.standard_normal((D, n)).astype(np.float32)
        A = pol.n_actions
        logits = torch.empty((A, n), device="cuda")
        act = torch.empty(n, dtype=torch.uint8, device="cuda")
        lp = torch.empty(n, device="cuda")
        val = torch.empty(n, device="cuda") if host[2] else None
        ws = None
        if with_ws:
            ws = torch.empty(simx.policy_forward_workspace_size(pol), dtype=torch.uint8,
                             device="cuda")
            with pytest.raises(simx.SimxError) as e:   # one byte short
                simx.policy_forward(pol, torch.from_numpy(obs).cuda(), n, mode, 99, 5,
                                    env_base=100, logits=logits, workspace=ws[:-1])
            assert e.value.status == simx.EINVAL
        simx.policy_forward(pol, torch.from_numpy(obs).cuda(), n, mode, 99, 5, env_base=100,
                            logits=logits, value=val, action=act, logp=lp, workspace=ws)
        torch.cuda.synchronize()
        for i in range(n):
            lg, v, a, l = oracle.policy(host, obs[:, i], ORC_MODE[mode], 99, 5, 100 + i)
            assert np.array_equal(logits[:, i].cpu().numpy(), lg)
            assert int(act[i]) == a
            assert np.float32(lp[i].item()) == np.float32(l)
            if val is not None:
                assert np.float32(val[i].item()) == np.float32(v)
