#!/usr/bin/env python
"""Throughput benchmark of the batched rollout engine (one JSON line on rank 0).

Workload: the single-server bursty heterogeneous environment (4096 envs x 512
decision steps, two-state MMPP 300/3000 req/s, 80/20 short/long requests, per-type
queues of 256, MLP 16-64-64-12, REINFORCE with a mean-return baseline), inputs
synthetic and seeded.  One step is one pass of the whole hot path over one batch:
rollout_collect (simulation + fused policy) -> REINFORCE returns -> mean baseline
-> loss gradient over all 2,097,152 rows, every stage a kernel of libsimx.so.

metric: simulated decision steps per second (envs x horizon x ranks / step time).
--impl reference times the oracle (the plain CPU reference) on a bounded sample of
the same workload on the host cores.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "simulated decision steps/sec"
UNIT = "steps/s"
WORKLOAD = "c2"
SEED_BASE = 0x5EED0002
GAMMA = 0.99
L2_FLUSH_BYTES = 256 << 20


def _args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=100)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", default="gpu", choices=["gpu", "reference"])
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-hbm-step", action="store_true")
    p.add_argument("--sweep", action="store_true",
                   help="every configuration (c1-c5, c5 at every env count): one JSON line each")
    p.add_argument("--sweep-configs", default="c1,c2,c3,c4,c5,c1p,c3s,c3t",
                   help="comma-separated subset of the sweep's configurations")
    p.add_argument("--sweep-child", default=None, help=argparse.SUPPRESS)
    p.add_argument("--loss-precision", default="tf32", choices=["tf32", "fp32"],
                   help="loss-gradient products: tf32 tensor cores (parity 1e-2) or fp32 (1e-5)")
    p.add_argument("--cpu-child", default=None, help=argparse.SUPPRESS)
    p.add_argument("--minibatch-loss", default=None, metavar="WORKLOAD",
                   help="time the PPO loss gradient on 8192-row minibatches of a workload's "
                        "rollout (both precisions) and exit")
    return p.parse_args()


# --------------------------------------------------------------------------- #
# CPU reference (the oracle), run in a child process with single-threaded BLAS
# --------------------------------------------------------------------------- #
def _oracle_step(n_envs: int, env0: int, H: int):
    """One oracle pass of the hot path over envs [env0, env0 + n_envs): rollout,
    returns, mean baseline, REINFORCE loss gradient (fp64).  Returns seconds."""
    import numpy as np

    import oracle
    from oracle import rl
    from paper_2607_05272_gb300 import workloads as W
    cfg = W.c2(n_envs)
    dims, hv = W.mlp_dims(WORKLOAD)
    Ws, bs = W.mlp_weights(dims, 1)
    t0 = time.perf_counter()
    out = oracle.rollout(cfg, (Ws, bs, hv), SEED_BASE, 0, list(range(env0, env0 + n_envs)), H)
    G = rl.returns(out["reward"], out["done"], GAMMA)
    adv, _ = rl.baseline(G)
    X = out["obs"].transpose(0, 2, 1).reshape(-1, dims[0])
    rl.loss_grad(Ws, bs, hv, X, out["action"].ravel(), out["logp"].ravel(), adv.ravel(),
                 G.ravel(), rl.REINFORCE, 0.2, 0.0, 0.0)
    return time.perf_counter() - t0


def _cpu_child(spec: str):
    kind, n_envs, steps, warm = spec.split(",")
    n_envs, steps, warm = int(n_envs), int(steps), int(warm)
    H = 512
    times = []
    for i in range(warm + steps):
        dt = _oracle_step(n_envs, (i * n_envs) % 4096, H)
        if i >= warm:
            times.append(dt)
    print(json.dumps({"times": times, "env_steps": n_envs * H}))


def _run_cpu(n_envs: int, steps: int, warm: int) -> dict:
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    r = subprocess.run([sys.executable, os.path.abspath(__file__), "--cpu-child",
                        "x,%d,%d,%d" % (n_envs, steps, warm)], capture_output=True, text=True,
                       env=env, cwd=ROOT)
    if r.returncode != 0:
        raise RuntimeError("oracle child failed:\n" + r.stderr[-2000:])
    return json.loads(r.stdout.strip().splitlines()[-1])


def cpu_baseline() -> dict:
    """The oracle as it stands, single-threaded, on a bounded sample (~10-20 s)."""
    import oracle
    oracle.build()
    probe = _run_cpu(16, 1, 0)
    per_env = probe["times"][0] / 16.0
    n = int(max(16, min(4096, 12.0 / max(per_env, 1e-6))))
    res = _run_cpu(n, 1, 0)
    v = res["env_steps"] / res["times"][0]
    return {"value": v, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": "%d envs x 512 steps of the same workload (rollout + returns + baseline + "
                      "loss gradient), single-threaded" % n}


def run_reference(a) -> None:
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import oracle
    oracle.build()
    probe = _run_cpu(16, 1, 0)
    per_env = probe["times"][0] / 16.0
    budget = min(6.0, 150.0 / max(1, a.steps + a.warmup))  # whole run within a few minutes
    n = int(max(4, min(4096, budget / max(per_env, 1e-6))))
    res = _run_cpu(n, a.steps, a.warmup)
    t = statistics.mean(res["times"])
    v = res["env_steps"] / t
    sample = ("%d envs x 512 steps per step (rollout + returns + baseline + loss gradient), "
              "single-threaded" % n)
    line = {
        "impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": a.gpus,
        "steps": a.steps, "warmup": a.warmup, "ms_per_step": t * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": "c2: 4096 envs x 512 steps, MMPP 300/3000 req/s, 80/20 short/long, "
                               "MLP 16-64-64-12, REINFORCE + mean baseline",
                   "sample_envs": n},
        "cpu_baseline": {"value": v, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": sample},
        "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def _sweep_child(spec: str):
    """Oracle rollout of one configuration over envs [env0, env0 + n) for H steps."""
    import oracle
    from paper_2607_05272_gb300 import workloads as W
    name, E, env0, n, H = spec.split(",")
    E, env0, n, H = int(E), int(env0), int(n), int(H)
    cfg = W.CONFIGS[name](E)
    dims, hv = W.mlp_dims(name)
    Ws, bs = W.policy_weights(name, dims, 1)
    mode = 1 if name == "c5" else 0
    t0 = time.perf_counter()
    oracle.rollout(cfg, (Ws, bs, hv, W.mlp_acts(name)), W.SEED[name], mode,
                   list(range(env0, env0 + n)), H)
    print(json.dumps({"seconds": time.perf_counter() - t0, "env_steps": n * H}))


def _oracle_rate(name: str, E: int, H: int, budget_s: float = 3.0) -> dict:
    """Oracle rollout env-steps/s on one core and on every host core (one fresh process per
    core over disjoint env ranges); each sample sized to about budget_s seconds."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")

    def child(env0, n, h):
        return subprocess.Popen([sys.executable, os.path.abspath(__file__), "--sweep-child",
                                 "%s,%d,%d,%d,%d" % (name, E, env0, n, h)], stdout=subprocess.PIPE,
                                stderr=subprocess.PIPE, text=True, env=env, cwd=ROOT)

    def result(p):
        out, err = p.communicate()
        if p.returncode != 0:
            raise RuntimeError("oracle child failed:\n" + err[-2000:])
        return json.loads(out.strip().splitlines()[-1])

    h = min(H, 64)
    probe = result(child(0, 1, h))
    per_step = probe["seconds"] / probe["env_steps"]
    target = max(h, int(budget_s / max(per_step, 1e-9)))  # env-steps for about budget_s
    h = min(H, max(h, target // E))                        # whole-E samples grow the horizon
    n = max(1, min(E, target // h))
    one = result(child(0, n, h))
    cores = os.cpu_count() or 1
    n_each = max(1, min(n, -(-E // cores)))
    h_each = min(H, max(h, target // n_each))
    procs = [child((i * n_each) % E, n_each, h_each) for i in range(cores)]
    res = [result(p) for p in procs]
    # every process runs concurrently; the rate uses each one's own compute time (process
    # start-up excluded), bounded by the slowest
    wall = max(r["seconds"] for r in res)
    return {"oracle_1core_steps_per_s": one["env_steps"] / one["seconds"],
            "oracle_ncore_steps_per_s": sum(r["env_steps"] for r in res) / wall,
            "oracle_cores": cores,
            "oracle_sample": "%d envs x %d steps (1 core); %d processes x %d envs x %d steps"
                             % (n, h, cores, n_each, h_each)}


def measure_fp32_peak(simx, torch) -> dict:
    """FP32 FMA rate of this GPU from the library's probe kernel (best of 5 launches)."""
    sink = torch.empty(simx.fma_probe_sink_floats(), device="cuda")
    simx.fma_probe(1000, sink)
    best = 0.0
    for _ in range(5):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        fl = simx.fma_probe(20000, sink)
        e1.record()
        torch.cuda.synchronize()
        best = max(best, fl / (e0.elapsed_time(e1) * 1e-3) / 1e12)
    props = torch.cuda.get_device_properties(torch.cuda.current_device())
    return {"tflops": best, "sms": props.multi_processor_count}


def run_sweep(a) -> None:
    """Every configuration on one GPU (rollout steps/s and FP32 fraction; GAE samples/s and
    HBM fraction; PPO loss minibatches/s) beside the oracle's 1-core and all-core rates."""
    import numpy as np
    import torch

    from paper_2607_05272_gb300 import build as B
    from paper_2607_05272_gb300 import workloads as W
    B.build()
    import oracle
    oracle.build()
    from paper_2607_05272_gb300 import simx
    peaks, src = _peaks()
    fp = measure_fp32_peak(simx, torch)
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    tf32_peak = float(peaks.get("bf16_tflops", 1900.0)) * 0.5
    print(json.dumps({"fp32_fma_probe_tflops": fp["tflops"], "sms": fp["sms"], "hbm_gbs": hbm,
                      "hbm_source": src}), flush=True)
    cases = [("c1", 64, 10000, "sample"), ("c2", 4096, 512, "sample"), ("c3", 16384, 256, "sample"),
             ("c4", 65536, 512, "sample"), ("c1p", 4096, 2000, "sample"),
             ("c3s", 4096, 256, "sample"), ("c3t", 16384, 256, "sample")]
    cases += [("c5", e, 1024, "argmax") for e in (1024, 4096, 16384, 65536, 262144, 1048576)]
    keep = set(a.sweep_configs.split(","))
    cases = [c for c in cases if c[0] in keep]
    oracle_cache = {}
    for name, E, H, mode in cases:
        cfg = W.CONFIGS[name](E)
        dims, hv = W.mlp_dims(name)
        Ws, bs = W.policy_weights(name, dims, 1)
        pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws],
                          [torch.from_numpy(b).cuda() for b in bs], hv, W.mlp_acts(name))
        sim = simx.Sim(cfg)
        sim.reset(W.SEED[name])
        warm = simx.alloc_rollout(E, sim.D, 4, has_value=hv)
        sim.rollout(mode, 4, warm, pol)
        del warm
        buf = simx.alloc_rollout(E, sim.D, H, has_value=hv)
        arr0 = sim.stats()["arrived"]
        reps = 3 if E * H <= 50_000_000 else 1
        ts = []
        for _ in range(reps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            sim.rollout(mode, H, buf, pol)
            e1.record()
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1))
        st, code = sim.last_status()
        arrivals = (sim.stats()["arrived"] - arr0) / reps
        ms = statistics.median(ts)
        P = sum(dims[l] * dims[l + 1] for l in range(len(dims) - 1))
        A = dims[-1] - (1 if hv else 0)
        flop = E * H * (2.0 * P + 20.0 * sum(dims[1:-1]) + 20.0 * A) + 15.0 * arrivals
        line = {"config": name, "envs": E, "horizon": H, "policy": mode,
                "rollout_ms": ms, "decision_steps_per_s": E * H / (ms * 1e-3),
                "fp32_tflops": flop / (ms * 1e-3) / 1e12,
                "fp32_frac": flop / (ms * 1e-3) / 1e12 / fp["tflops"], "status": st}
        n = E * H
        if hv:  # GAE over the rollout buffer: reward, value, done in; advantage, return out
            adv = torch.empty((H, E), device="cuda")
            ret = torch.empty((H, E), device="cuda")
            last = torch.zeros(E, device="cuda")
            gts = []
            for _ in range(3):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                simx.compute_returns_gae(buf["reward"], buf["done"], 0.99, 0.95, ret, adv=adv,
                                         val=buf["value"], last_val=last)
                e1.record()
                torch.cuda.synchronize()
                gts.append(e0.elapsed_time(e1))
            g = min(gts)
            line.update({"gae_ms": g, "gae_samples_per_s": n / (g * 1e-3),
                         "gae_gbs": 17.0 * n / (g * 1e-3) / 1e9,
                         "gae_hbm_frac": 17.0 * n / (g * 1e-3) / 1e9 / hbm})
            # PPO loss gradient on one minibatch of 8192 rows, both precisions
            rng = np.random.default_rng(1)
            idx = torch.from_numpy(rng.permutation(n)[:8192].astype(np.int64)).cuda()
            grad = torch.empty(pol.n_params, device="cuda")
            stats = torch.empty(5, device="cuda")
            ws = torch.empty(simx.ppo_loss_grad_workspace_size(pol, 8192), dtype=torch.uint8,
                             device="cuda")
            lflop = 8192 * (6.0 * P - 2.0 * dims[0] * dims[1])
            for prec in ("fp32", "tf32"):
                lts = []
                for _ in range(6):
                    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    e0.record()
                    simx.ppo_loss_grad(pol, buf, ret, adv, idx, 8192, "ppo", 0.2, 0.5, 0.01, grad,
                                       stats, ws, precision=prec)
                    e1.record()
                    torch.cuda.synchronize()
                    lts.append(e0.elapsed_time(e1))
                lm = statistics.median(lts[1:])
                line["loss8192_%s_ms" % prec] = lm
                line["loss8192_%s_minibatches_per_s" % prec] = 1e3 / lm
                line["loss8192_%s_tflops" % prec] = lflop / (lm * 1e-3) / 1e12
            del adv, ret, grad, ws
        key = name if name != "c5" else "c5"
        if key not in oracle_cache:
            oracle_cache[key] = _oracle_rate(name, E, H)
        line.update(oracle_cache[key])
        line["gpu_vs_oracle_ncore"] = line["decision_steps_per_s"] / line["oracle_ncore_steps_per_s"]
        print(json.dumps(line), flush=True)
        sim.close()
        del buf, sim, pol
        torch.cuda.empty_cache()


# --------------------------------------------------------------------------- #
# GPU arm
# --------------------------------------------------------------------------- #
class Clocks:
    """nvidia-smi sampling during the timed region."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.p = None
        try:
            self.p = subprocess.Popen(["nvidia-smi", "-i", str(index), "--query-gpu=" + self.Q,
                                       "--format=csv,noheader,nounits", "-lms", "200"],
                                      stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.p = None

    def stop(self):
        if self.p is None:
            return None
        self.p.terminate()
        try:
            out, _ = self.p.communicate(timeout=10)
        except subprocess.TimeoutExpired:
            self.p.kill()
            out, _ = self.p.communicate()
        rows = []
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 7:
                continue
            try:
                rows.append((float(f[0]), float(f[1]), f[3:7]))
            except ValueError:
                continue
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, r in rows for i in range(4) if r[i].lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


# DRAM bytes (read + write) of one k_rollout launch of the benchmark workload, from an
# ncu capture of the current kernel; to be re-measured (or set to None) whenever the
# rollout kernel changes.
ROLLOUT_DRAM_BYTES = 123.8e6


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except (OSError, ValueError):
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "sm_max_mhz": 2070.0}, "fallback"


def hbm_step_measure(simx, W, torch, E=65536, steps=100, warm=10) -> dict:
    """sim_step_batched with the Shortest-Queue baseline on the 4-server environment.

    The timed steps are replayed from a CUDA graph (launch-bound otherwise: one step is a
    few microseconds).  Counted bytes per env-step: the structure-of-arrays state read and
    written (29 header words, 2K server words, 2KT queue words), the records written (next
    observation, reward, done, action) and 8 B per routed request (one ring write and one
    ring read)."""
    cfg = W.c5(E)
    K, T, D = cfg["n_servers"], cfg["n_types"], cfg["obs_dim"]
    sim = simx.Sim(cfg)
    sim.reset(SEED_BASE + 5)
    obs = torch.empty((D, E), device="cuda")
    rew = torch.empty(E, device="cuda")
    done = torch.empty(E, dtype=torch.uint8, device="cuda")
    act = torch.empty(E, dtype=torch.uint8, device="cuda")
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for _ in range(warm):
            sim.step("sq", obs=obs, reward=rew, done=done, action=act)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        for _ in range(steps):
            sim.step("sq", obs=obs, reward=rew, done=done, action=act)
    graph.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = 3
    e0.record()
    for _ in range(reps):
        graph.replay()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / (reps * steps)
    st, code = sim.last_status()
    sim.close()
    if st != 0:
        raise RuntimeError("device status 0x%x in the HBM step" % code)
    state = (29 + 2 * K + 2 * K * T) * 4
    per = 2 * state + (D * 4 + 4 + 1 + 1) + 8
    gbs = per * E / (ms * 1e-3) / 1e9
    peaks, src = _peaks()
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    l2 = "state (%.0f MB) %s the 129 MB L2" % (state * E / 1e6, "fits in" if state * E < 100e6 else "exceeds")
    return {"kernel": "k_step_thread (policy-free step, SoA state round trip)", "envs": E,
            "us_per_step": ms * 1e3, "env_steps_per_s": E / (ms * 1e-3),
            "bytes_per_env_step": per, "achieved": gbs, "peak": hbm, "unit": "GB/s",
            "frac": gbs / hbm, "peak_source": "%s hbm_gbs" % src, "l2": l2,
            "timing": "CUDA graph of %d steps, replayed %d times, CUDA events" % (steps, reps)}


def run_minibatch_loss(name: str, E: int = 256, steps: int = 20) -> None:
    """The PPO loss gradient (Sec. 4.3) on 8192-row minibatches drawn from a rollout of
    `name` (E envs x its horizon): median of `steps` timed calls per precision after 3
    warm-up calls, CUDA events on the stream; one JSON line."""
    import numpy as np
    import torch

    from paper_2607_05272_gb300 import build as B
    from paper_2607_05272_gb300 import workloads as W
    B.build()
    from paper_2607_05272_gb300 import simx
    cfg = W.CONFIGS[name](E)
    H = W.HORIZON[name]
    dims, hv = W.mlp_dims(name)
    Ws, bs = W.policy_weights(name, dims, 1)
    pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws],
                      [torch.from_numpy(b).cuda() for b in bs], hv, W.mlp_acts(name))
    sim = simx.Sim(cfg)
    sim.reset(W.SEED[name])
    buf = simx.alloc_rollout(E, sim.D, H, has_value=hv)
    sim.rollout("sample", H, buf, pol)
    n = E * H
    rng = np.random.default_rng(1)
    ret = torch.from_numpy(rng.standard_normal((H, E)).astype(np.float32)).cuda()
    adv = torch.from_numpy(rng.standard_normal((H, E)).astype(np.float32)).cuda()
    idx = torch.from_numpy(rng.permutation(n)[:8192].astype(np.int64)).cuda()
    grad = torch.empty(pol.n_params, device="cuda")
    stats = torch.empty(5, device="cuda")
    ws = torch.empty(simx.ppo_loss_grad_workspace_size(pol, 8192), dtype=torch.uint8, device="cuda")
    P = sum(w.size for w in Ws)
    flop = 8192 * (6.0 * P - 2.0 * dims[0] * dims[1])
    line = {"workload": name, "rows": 8192, "mlp": dims, "flop_per_call": flop}
    for prec in ("fp32", "tf32"):
        ts = []
        for i in range(3 + steps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            simx.ppo_loss_grad(pol, buf, ret, adv, idx, 8192, "ppo", 0.2, 0.5, 0.01, grad, stats,
                               ws, precision=prec)
            e1.record()
            torch.cuda.synchronize()
            if i >= 3:
                ts.append(e0.elapsed_time(e1))
        ms = statistics.median(ts)
        line[prec] = {"ms": ms, "minibatches_per_s": 1e3 / ms, "tflops": flop / (ms * 1e-3) / 1e12}
    print(json.dumps(line), flush=True)


# --- replicas (N > 1): every rank simulates its own envs, no data-path collective -------

def replica_seed(rank: int) -> int:
    """Seed of rank `rank`'s replica: envs are keyed by (seed, env id), so replicas with
    different seeds are independent problems (weak scaling)."""
    return SEED_BASE + rank


def max_over_ranks(x: float, dist=None, device="cpu") -> float:
    """The largest of the ranks' values (the step time the job is charged)."""
    if dist is None:
        return x
    import torch
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(world: int, units_per_rank: int, ms: float) -> float:
    """Whole-job throughput: the units all ranks processed over the slowest rank's time."""
    return world * units_per_rank / (ms * 1e-3)


def run_gpu(a) -> None:
    import numpy as np
    import torch

    from paper_2607_05272_gb300 import build as B
    from paper_2607_05272_gb300 import workloads as W
    B.build()
    from paper_2607_05272_gb300 import simx

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")

    # Replicas: every rank simulates its own 4096 envs (seed offset by rank); no
    # data-path collective, only the timing barrier and max-reduction.
    E, H = 4096, W.HORIZON[WORKLOAD]
    cfg = W.c2(E)
    dims, hv = W.mlp_dims(WORKLOAD)
    Ws, bs = W.mlp_weights(dims, 1)
    dWs = [torch.from_numpy(w).cuda() for w in Ws]
    dbs = [torch.from_numpy(b).cuda() for b in bs]
    pol = simx.Policy(dWs, dbs, hv)
    sim = simx.Sim(cfg, device=local)
    sim.reset(replica_seed(rank))
    D = sim.D
    n = E * H
    buf = simx.alloc_rollout(E, D, H)
    ret = torch.empty((H, E), device="cuda")
    adv = torch.empty((H, E), device="cuda")
    mean = torch.empty(1, device="cuda")
    ws_b = torch.empty(simx.returns_baseline_workspace_size(n), dtype=torch.uint8, device="cuda")
    grad = torch.empty(pol.n_params, device="cuda")
    stats = torch.empty(5, device="cuda")
    ws_l = torch.empty(simx.ppo_loss_grad_workspace_size(pol, n), dtype=torch.uint8, device="cuda")
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    fp = measure_fp32_peak(simx, torch)  # FP32 roofline denominator, measured on this GPU
    stream = torch.cuda.current_stream()

    def step(ev=None):
        if ev:
            ev[0].record(stream)
        sim.rollout("sample", H, buf, pol)
        if ev:
            ev[1].record(stream)
        simx.compute_returns_gae(buf["reward"], buf["done"], GAMMA, -1.0, ret)
        if ev:
            ev[2].record(stream)
        simx.returns_baseline(ret, adv, mean, ws_b)
        if ev:
            ev[3].record(stream)
        simx.ppo_loss_grad(pol, buf, ret, adv, None, n, "reinforce", 0.2, 0.0, 0.0, grad, stats,
                           ws_l, precision=a.loss_precision)
        if ev:
            ev[4].record(stream)

    for _ in range(a.warmup):
        step()
    torch.cuda.synchronize()

    # candidates generated per rollout launch (for the algorithmic FLOP count)
    cj0 = sim.save()[:, 2].astype(np.int64)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(a.steps)]
    clocks = Clocks(local) if rank == 0 else None
    l0 = simx.launches()
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    t_wall = time.perf_counter()
    for k in range(a.steps):
        flush.zero_()  # evict L2 between steps (outside the timed events)
        step(evs[k])
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    t_wall = time.perf_counter() - t_wall
    launches = simx.launches() - l0
    clk = clocks.stop() if clocks else None
    cj1 = sim.save()[:, 2].astype(np.int64)
    cand_per_launch = float((cj1 - cj0).sum()) / a.steps

    phase_ms = [[evs[k][i].elapsed_time(evs[k][i + 1]) for i in range(4)] for k in range(a.steps)]
    step_ms = [evs[k][0].elapsed_time(evs[k][4]) for k in range(a.steps)]
    ms = statistics.mean(step_ms)
    ph = [statistics.mean(p[i] for p in phase_ms) for i in range(4)]
    ms = max_over_ranks(ms, dist, "cuda")
    value = job_value(world, n, ms)
    st, code = sim.last_status()
    if st != 0:
        raise RuntimeError("device status 0x%x after the timed region" % code)

    # end to end through the public API: policy in from pinned host memory, gradient and
    # statistics back to the host, every step
    e2e = None
    if not a.no_e2e:
        hW = [torch.from_numpy(w).pin_memory() for w in Ws]
        hb = [torch.from_numpy(b).pin_memory() for b in bs]
        hg = torch.empty(pol.n_params, dtype=torch.float32).pin_memory()
        hs = torch.empty(5, dtype=torch.float32).pin_memory()
        h2d = sum(w.numel() * 4 for w in hW) + sum(b.numel() * 4 for b in hb)
        d2h = hg.numel() * 4 + hs.numel() * 4
        k_e2e = max(3, min(a.steps, 50))
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(k_e2e):
            for d, h in zip(dWs + dbs, hW + hb):
                d.copy_(h, non_blocking=True)
            step()
            hg.copy_(grad, non_blocking=True)
            hs.copy_(stats, non_blocking=True)
            torch.cuda.synchronize()
        t_e2e = (time.perf_counter() - t0) / k_e2e
        t_e2e = max_over_ranks(t_e2e, dist, "cuda")
        e2e = {"value": job_value(world, n, t_e2e * 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h}

    # the loss gradient in the other precision, on the same buffer, for comparison
    other = "fp32" if a.loss_precision == "tf32" else "tf32"
    lo_ms = []
    for _ in range(5):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        simx.ppo_loss_grad(pol, buf, ret, adv, None, n, "reinforce", 0.2, 0.0, 0.0, grad, stats,
                           ws_l, precision=other)
        e1.record(stream)
        torch.cuda.synchronize()
        lo_ms.append(e0.elapsed_time(e1))
    loss_other_ms = statistics.median(lo_ms[1:])

    # the policy-free batched step (Sec. 5.1 Shortest-Queue router) of the multi-server
    # environment at 65,536 envs: state read and written every step, HBM-bound
    hbm_step = None if a.no_hbm_step else [hbm_step_measure(simx, W, torch, E=e)
                                            for e in (65536, 1048576)]

    # roofline of the dominant kernel
    peaks, src = _peaks()
    sm_mhz = float(peaks.get("sm_max_mhz", 2070.0))
    fp32_nominal = fp["sms"] * 128 * 2 * sm_mhz * 1e6 / 1e12  # FMA lanes x clock
    fp32_peak = fp["tflops"]
    fp32_src = ("measured FMA probe (libsimx k_fma_probe, best of 5): %.1f TFLOP/s; nominal "
                "%d SMs x 128 lanes x 2 x %.0f MHz = %.1f" % (fp32_peak, fp["sms"], sm_mhz,
                                                            fp32_nominal))
    P = sum(dims[l] * dims[l + 1] for l in range(len(dims) - 1))
    hidden = sum(dims[1:-1])
    A = dims[-1] - (1 if hv else 0)
    flop_rollout = n * (2.0 * P + 20.0 * hidden + 20.0 * A) + 15.0 * cand_per_launch
    flop_loss = n * (6.0 * P - 2.0 * dims[0] * dims[1])
    phases = {"rollout_ms": ph[0], "returns_ms": ph[1], "baseline_ms": ph[2], "loss_grad_ms": ph[3],
              "loss_grad_%s_ms" % other: loss_other_ms}
    # the loss kernel against its own bound: FP32 lanes, or the TF32 tensor pipe (nominally
    # half the bf16 rate; the measured bf16 GEMM peak x 0.5)
    if a.loss_precision == "tf32":
        tf32_peak = float(peaks.get("bf16_tflops", 1900.0)) * 0.5
        ach_l = flop_loss / (ph[3] * 1e-3) / 1e12
        roof_loss = {"kernel": "k_loss_tc (tcgen05 kind::tf32)", "bound": "tensor", "achieved": ach_l,
                     "peak": tf32_peak, "unit": "TFLOP/s", "frac": ach_l / tf32_peak, "traffic": None,
                     "peak_source": "%s bf16_tflops x 0.5 (nominal tf32 / bf16 rate)" % src}
    else:
        ach_l = flop_loss / (ph[3] * 1e-3) / 1e12
        roof_loss = {"kernel": "k_loss_fused (FP32 SIMT)", "bound": "alu", "achieved": ach_l,
                     "peak": fp32_peak, "unit": "TFLOP/s", "frac": ach_l / fp32_peak, "traffic": None,
                     "peak_source": fp32_src}
    dom = max(range(4), key=lambda i: ph[i])
    if dom == 0:
        ach = flop_rollout / (ph[0] * 1e-3) / 1e12
        roof = {"kernel": "k_rollout (simulation + fused policy)", "bound": "alu", "achieved": ach,
                "peak": fp32_peak, "unit": "TFLOP/s", "frac": ach / fp32_peak,
                "traffic": ROLLOUT_DRAM_BYTES,
                "traffic_source": "ncu dram__bytes_read.sum + dram__bytes_write.sum of one "
                                  "k_rollout launch of this workload (10.0 MB + 113.8 MB)",
                "peak_source": fp32_src}
    elif dom == 3:
        roof = roof_loss
    else:
        hbm = float(peaks.get("hbm_gbs", 6800.0))
        byts = n * 13.0 if dom == 1 else n * 12.0
        ach = byts / (ph[dom] * 1e-3) / 1e9
        roof = {"kernel": "returns" if dom == 1 else "baseline", "bound": "hbm", "achieved": ach,
                "peak": hbm, "unit": "GB/s", "frac": ach / hbm, "traffic": None,
                "peak_source": "%s hbm_gbs" % src}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": a.steps,
            "warmup": a.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32+tf32" if a.loss_precision == "tf32" else "f32",
            "data": "synthetic",
            "config": {"workload": "c2: 4096 envs x 512 steps per GPU, MMPP 300/3000 req/s, "
                                   "80/20 short/long, MLP 16-64-64-12, REINFORCE + mean baseline",
                       "envs_per_gpu": E, "horizon": H, "l2": "flushed (256 MB write) before every "
                       "timed step", "parallelism": "replicas" if world > 1 else "single GPU",
                       "loss_precision": "tf32 tensor cores, split tf32 first layer, fp32 "
                       "accumulation (parity 1e-2)" if a.loss_precision == "tf32" else
                       "fp32 (parity 1e-5)"},
            "phases_ms": phases,
            "roofline": roof,
            "roofline_loss": roof_loss,
            "e2e": e2e,
            "hbm_step": hbm_step,
            "gpu_launches": launches,
            "clocks": clk,
            "wall_s": t_wall,
        }
        if world == 1 and not a.no_cpu_baseline:
            line["cpu_baseline"] = cpu_baseline()
        print(json.dumps(line), flush=True)
    sim.close()
    if dist:
        dist.destroy_process_group()


def main():
    a = _args()
    if a.cpu_child:
        _cpu_child(a.cpu_child)
        return
    if a.sweep_child:
        _sweep_child(a.sweep_child)
        return
    if a.minibatch_loss:
        run_minibatch_loss(a.minibatch_loss)
        return
    if a.sweep:
        run_sweep(a)
        return
    if a.impl == "reference":
        run_reference(a)
    else:
        run_gpu(a)


if __name__ == "__main__":
    main()
