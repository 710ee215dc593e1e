#!/usr/bin/env python
"""Throughput benchmark of the batched rollout engine (one JSON line on rank 0).

Workload: the trace-shaped multi-server environment (65,536 envs x 512 decision steps
per GPU, 8 simulated servers, diurnal 1000-8000 req/s x lognormal(0, 1) burst factors
per 500 ms, Pareto(1.5, 10 ms) long-request costs, 85/15 short/long, action = server x
batch size (48), MLP 28-256-256-48 plus a value row, PPO with GAE(0.99, 0.95)), the
largest configuration that fits one GPU, inputs synthetic and seeded.  One step is one
pass of the whole hot path over one batch, every numeric stage a kernel of libsimx.so:
rollout_collect (simulation + fused policy) -> bootstrap value -> GAE -> one PPO epoch
over the 33,554,432 rows in 4096 minibatches of 8192 (loss gradient + Adam update
each, replayed from a CUDA graph).  --epochs 4 runs the four epochs of the full PPO
update.  The minibatch permutation is drawn on the device by torch.randperm.

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
WORKLOAD = "c4"
ENVS, HORIZON, MINIBATCH = 65536, 512, 8192
SEED_BASE = 0x5EED0004
GAMMA, LAMBDA = 0.99, 0.95
CLIP, C_VALUE, C_ENTROPY, LR, MAX_NORM = 0.2, 0.5, 0.01, 3e-4, 0.5
L2_FLUSH_BYTES = 256 << 20
WORKLOAD_TEXT = ("c4: 65,536 envs x 512 steps per GPU, 8 servers, diurnal 1000-8000 req/s x "
                 "lognormal(0,1) per 500 ms, Pareto(1.5, 10 ms) long costs, 85/15 short/long, "
                 "MLP 28-256-256-48+V, PPO (GAE 0.99/0.95, clip 0.2, minibatches of 8192, Adam)")


def _args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=10)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--epochs", type=int, default=1,
                   help="PPO epochs per step (passes of minibatches over the rollout buffer)")
    p.add_argument("--impl", default="gpu", choices=["gpu", "reference"])
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-hbm-step", action="store_true")
    p.add_argument("--no-extras", action="store_true", help="skip the c2 and 1M-env c5 extra lines")
    p.add_argument("--sweep", action="store_true",
                   help="every configuration (c1-c5, c5 at every env count): one JSON line each")
    p.add_argument("--sweep-configs", default="c1,c2,c3,c4,c5,c1p,c3s,c3t",
                   help="comma-separated subset of the sweep's configurations")
    p.add_argument("--sweep-child", default=None, help=argparse.SUPPRESS)
    p.add_argument("--loss-precision", default="tf32", choices=["tf32", "fp32"],
                   help="loss-gradient products: tf32 tensor cores (parity 1e-2) or fp32 (1e-5)")
    p.add_argument("--cpu-child", default=None, help=argparse.SUPPRESS)
    p.add_argument("--grid-rollout", default=None, metavar="WORKLOAD",
                   help="time a grid policy's rollout with the forward on the tensor cores and on "
                        "the FP32 tiles (the exact policy forward) and exit")
    p.add_argument("--grid-envs", type=int, default=65536)
    p.add_argument("--rollout-only", default=None, metavar="WORKLOAD",
                   help="time rollout_collect alone (its fp32 policy) with the forward's weights "
                        "staged in shared memory and read through L1, and exit")
    p.add_argument("--rollout-envs", type=int, default=None)
    p.add_argument("--rollout-steps", type=int, default=None)
    p.add_argument("--hbm-step-only", type=int, default=None, metavar="ENVS",
                   help="time only the policy-free batched step at this env count and exit")
    p.add_argument("--minibatch-loss", default=None, metavar="WORKLOAD",
                   help="time the PPO loss gradient on 8192-row minibatches of a workload's "
                        "rollout (both precisions) and exit")
    return p.parse_args()


# --------------------------------------------------------------------------- #
# CPU reference (the oracle), run in a child process with single-threaded BLAS
# --------------------------------------------------------------------------- #
def _oracle_step(n_envs: int, env0: int, H: int, epochs: int):
    """One oracle pass of the hot path over envs [env0, env0 + n_envs) of the workload:
    rollout, bootstrap value, GAE, then `epochs` PPO epochs over the sample's rows in
    minibatches of up to 8192 (fp64 loss gradient and Adam on each).  Returns seconds."""
    import numpy as np

    import oracle
    from oracle import rl
    from paper_2607_05272_gb300 import workloads as W
    cfg = W.CONFIGS[WORKLOAD](ENVS)
    dims, hv = W.mlp_dims(WORKLOAD)
    Ws, bs = W.policy_weights(WORKLOAD, dims, 1)
    t0 = time.perf_counter()
    ids = list(range(env0, env0 + n_envs))
    # H + 1 decisions: the first H are the rollout, the last one's observation is each
    # env's state after it, whose value row bootstraps GAE
    full = oracle.rollout(cfg, (Ws, bs, hv), SEED_BASE, 0, ids, H + 1)
    out = {k: full[k][:H] for k in ("obs", "action", "logp", "value", "reward", "done")}
    _, Z = rl.forward(Ws, bs, full["obs"][H].T)
    last = Z[:, -1].astype(np.float32)
    A, R = rl.gae(out["reward"], out["value"], out["done"], GAMMA, LAMBDA, last)
    n = n_envs * H
    flat = np.concatenate([np.concatenate([w.ravel(), b.ravel()]) for w, b in zip(Ws, bs)])
    p, m, v = flat.astype(np.float64), np.zeros(flat.size), np.zeros(flat.size)
    rng = np.random.default_rng(env0)
    t = 0
    for _ in range(epochs):
        perm = rng.permutation(n)
        for i in range(0, n, MINIBATCH):
            rows = perm[i:i + MINIBATCH]
            X, a, lpo = rl.gather_rows(out["obs"], out["action"], out["logp"], rows, n_envs)
            tt, ee = rows // n_envs, rows % n_envs
            g, _ = rl.loss_grad(Ws, bs, hv, X, a, lpo, A[tt, ee], R[tt, ee], rl.PPO, CLIP, C_VALUE,
                                C_ENTROPY)
            t += 1
            p, m, v = rl.adam_step(p, rl.flat(g), m, v, t, LR, max_grad_norm=MAX_NORM)
    return time.perf_counter() - t0


def _cpu_child(spec: str):
    kind, n_envs, steps, warm, epochs = spec.split(",")
    n_envs, steps, warm, epochs = int(n_envs), int(steps), int(warm), int(epochs)
    times = []
    for i in range(warm + steps):
        dt = _oracle_step(n_envs, (i * n_envs) % ENVS, HORIZON, epochs)
        if i >= warm:
            times.append(dt)
    print(json.dumps({"times": times, "env_steps": n_envs * HORIZON}))


def _run_cpu(n_envs: int, steps: int, warm: int, epochs: int) -> dict:
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    r = subprocess.run([sys.executable, os.path.abspath(__file__), "--cpu-child",
                        "x,%d,%d,%d,%d" % (n_envs, steps, warm, epochs)], capture_output=True,
                       text=True, env=env, cwd=ROOT)
    if r.returncode != 0:
        raise RuntimeError("oracle child failed:\n" + r.stderr[-2000:])
    return json.loads(r.stdout.strip().splitlines()[-1])


def _sample_text(n: int, epochs: int) -> str:
    return ("%d envs x %d steps of the same workload (rollout, bootstrap value, GAE, %d PPO "
            "epoch(s) of loss gradient + Adam over those rows), single-threaded"
            % (n, HORIZON, epochs))


def cpu_baseline(epochs: int) -> dict:
    """The oracle as it stands, single-threaded, on a bounded sample (~10-20 s)."""
    import oracle
    oracle.build()
    probe = _run_cpu(2, 1, 0, epochs)
    per_env = probe["times"][0] / 2.0
    n = int(max(2, min(4096, 12.0 / max(per_env, 1e-6))))
    res = _run_cpu(n, 1, 0, epochs)
    v = res["env_steps"] / res["times"][0]
    return {"value": v, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": _sample_text(n, epochs)}


def run_reference(a) -> None:
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import oracle
    oracle.build()
    probe = _run_cpu(2, 1, 0, a.epochs)
    per_env = probe["times"][0] / 2.0
    budget = min(6.0, 150.0 / max(1, a.steps + a.warmup))  # whole run within a few minutes
    n = int(max(2, min(4096, budget / max(per_env, 1e-6))))
    res = _run_cpu(n, a.steps, a.warmup, a.epochs)
    t = statistics.mean(res["times"])
    v = res["env_steps"] / t
    line = {
        "impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": a.gpus,
        "steps": a.steps, "warmup": a.warmup, "ms_per_step": t * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD_TEXT, "ppo_epochs_per_step": a.epochs, "sample_envs": n},
        "cpu_baseline": {"value": v, "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": _sample_text(n, a.epochs)},
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
# ncu capture of the current kernel; None until one is taken, and to be re-measured (or
# set back to None) whenever the rollout kernel changes.
ROLLOUT_DRAM_BYTES = 389046528.0 + 4584373504.0
ROLLOUT_DRAM_SOURCE = ("ncu dram__bytes_read.sum + dram__bytes_write.sum of one k_rollout launch "
                       "of this workload (389.0 MB + 4584.4 MB; profiles/k_rollout_c4_bench.md)")


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


def run_grid_rollout(name: str, E: int, reps: int = 3) -> None:
    """A grid policy (the exact policy forward) on `name`'s env: rollout_collect with the
    forward on the tensor cores, then on the FP32 tiles (SIMX_TC_FORWARD=0), CUDA events
    around each launch after a warm-up; the two buffers must be equal bit for bit."""
    import torch

    from paper_2607_05272_gb300 import build as B
    from paper_2607_05272_gb300 import workloads as W
    B.build()
    from paper_2607_05272_gb300 import simx
    cfg = W.CONFIGS[name](E)
    H = W.HORIZON[name]
    dims, hv = W.mlp_dims(name)
    gx = [5] + [7] * (len(dims) - 2)
    ew = [8] * (len(dims) - 1)
    Ws, bs = W.grid_weights(dims, 21, gx, ew)
    pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws], [torch.from_numpy(b).cuda() for b in bs],
                      hv, W.mlp_acts(name), grid=gx)
    mode = "argmax" if name == "c5" else "sample"
    line = {"workload": name, "envs": E, "horizon": H, "mlp": dims}
    bufs = []
    for tc in ("1", "0"):
        os.environ["SIMX_TC_FORWARD"] = tc
        sim = simx.Sim(cfg)
        shape = sim.launch_shape(mode, pol)
        sim.reset(W.SEED[name])
        warm = simx.alloc_rollout(E, sim.D, 4, has_value=hv)
        sim.rollout(mode, 4, warm, pol)
        del warm
        buf = simx.alloc_rollout(E, sim.D, H, has_value=hv)
        ts = []
        for _ in range(reps):
            sim.reset(W.SEED[name])
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            sim.rollout(mode, H, buf, pol)
            e1.record()
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1))
        st, _ = sim.last_status()
        sim.close()
        ms = statistics.median(ts)
        key = "tensor_cores" if tc == "1" else "fp32_tiles"
        line[key] = {"ms": ms, "decision_steps_per_s": E * H / (ms * 1e-3), "status": st,
                     "launch": shape}
        bufs.append(buf)
    os.environ.pop("SIMX_TC_FORWARD", None)
    line["bit_identical"] = all(torch.equal(bufs[0][k], bufs[1][k]) for k in bufs[0])
    line["speedup"] = line["fp32_tiles"]["ms"] / line["tensor_cores"]["ms"]
    print(json.dumps(line), flush=True)


def run_rollout_only(name: str, E: int, H: int, reps: int = 3) -> None:
    """rollout_collect of `name`'s fp32 policy over E envs x H steps, with the policy's
    weights staged in shared memory (SIMX_STAGE=1) and read through L1 (SIMX_STAGE=0):
    CUDA events around each launch after a warm-up; the two buffers must be equal bit for
    bit.  One JSON line."""
    import torch

    from paper_2607_05272_gb300 import build as B
    from paper_2607_05272_gb300 import workloads as W
    B.build()
    from paper_2607_05272_gb300 import simx
    cfg = W.CONFIGS[name](E)
    dims, hv = W.mlp_dims(name)
    Ws, bs = W.policy_weights(name, dims, 1)
    pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws], [torch.from_numpy(b).cuda() for b in bs],
                      hv, W.mlp_acts(name))
    mode = "argmax" if name == "c5" else "sample"
    line = {"workload": name, "envs": E, "horizon": H, "mlp": dims}
    bufs = []
    for stage in ("1", "0"):
        os.environ["SIMX_STAGE"] = stage
        sim = simx.Sim(cfg)
        shape = sim.launch_shape(mode, pol)
        sim.reset(W.SEED[name])
        warm = simx.alloc_rollout(E, sim.D, 4, has_value=hv)
        sim.rollout(mode, 4, warm, pol)
        del warm
        buf = simx.alloc_rollout(E, sim.D, H, has_value=hv)
        ts = []
        for _ in range(reps):
            sim.reset(W.SEED[name])
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            sim.rollout(mode, H, buf, pol)
            e1.record()
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1))
        st, _ = sim.last_status()
        sim.close()
        ms = statistics.median(ts)
        key = "staged" if stage == "1" else "through_l1"
        line[key] = {"ms": ms, "us_per_step": 1000.0 * ms / H,
                     "decision_steps_per_s": E * H / (ms * 1e-3), "status": st, "launch": shape}
        bufs.append(buf)
    os.environ.pop("SIMX_STAGE", None)
    line["bit_identical"] = all(torch.equal(bufs[0][k], bufs[1][k]) for k in bufs[0])
    line["speedup"] = line["through_l1"]["ms"] / line["staged"]["ms"]
    print(json.dumps(line), flush=True)


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


class PPOStep:
    """One step of the benchmark on this GPU: rollout -> bootstrap value -> GAE -> PPO
    epochs (loss gradient + Adam per minibatch, the minibatch loop replayed from a CUDA
    graph captured on the first call after a warm eager one)."""

    def __init__(self, simx, W, torch, seed: int, epochs: int, precision: str, device: int):
        import numpy as np
        self.simx, self.torch = simx, torch
        self.E, self.H, self.mb, self.epochs, self.precision = ENVS, HORIZON, MINIBATCH, epochs, precision
        cfg = W.CONFIGS[WORKLOAD](self.E)
        self.dims, hv = W.mlp_dims(WORKLOAD)
        Ws, bs = W.policy_weights(WORKLOAD, self.dims, 1)
        self.host_params = np.concatenate([np.concatenate([w.ravel(), b.ravel()])
                                           for w, b in zip(Ws, bs)]).astype(np.float32)
        self.params = torch.from_numpy(self.host_params.copy()).cuda()
        self.policy = simx.Policy.from_flat(self.params, self.dims, hv)
        n = self.params.numel()
        self.m = torch.zeros(n, device="cuda")
        self.v = torch.zeros(n, device="cuda")
        self.grad = torch.empty(n, device="cuda")
        self.stats = torch.empty(5, device="cuda")
        self.adam_ws = torch.empty(simx.adam_workspace_size(n), dtype=torch.uint8, device="cuda")
        self.t_dev = torch.zeros(1, dtype=torch.int64, device="cuda")
        self.sim = simx.Sim(cfg, device=device)
        self.sim.reset(seed)
        self.D = self.sim.D
        self.buf = simx.alloc_rollout(self.E, self.D, self.H, has_value=True)
        self.ret = torch.empty((self.H, self.E), device="cuda")
        self.adv = torch.empty((self.H, self.E), device="cuda")
        self.last = torch.empty(self.E, device="cuda")
        self.obs_next = torch.empty((self.D, self.E), device="cuda")
        self.pf_ws = torch.empty(simx.policy_forward_workspace_size(self.policy),
                                 dtype=torch.uint8, device="cuda")
        self.n_rows = self.E * self.H
        self.n_mb = self.n_rows // self.mb
        self.loss_ws = torch.empty(simx.ppo_loss_grad_workspace_size(self.policy, self.mb),
                                   dtype=torch.uint8, device="cuda")
        self.perm = torch.empty((epochs, self.n_rows), dtype=torch.int64, device="cuda")
        self.gen = torch.Generator(device="cuda")
        self.gen.manual_seed(seed)
        self.graph = None
        self.graph_launches = 0
        self.replays = 0

    def _updates(self):
        s = self.simx
        for e in range(self.epochs):
            for i in range(self.n_mb):
                s.ppo_loss_grad(self.policy, self.buf, self.ret, self.adv,
                                self.perm[e, i * self.mb:(i + 1) * self.mb], self.mb, "ppo", CLIP,
                                C_VALUE, C_ENTROPY, self.grad, self.stats, self.loss_ws,
                                precision=self.precision)
                s.adam_step(self.params, self.grad, self.m, self.v, self.t_dev, LR,
                            max_grad_norm=MAX_NORM, workspace=self.adam_ws)

    def run(self, ev=None):
        """One step; ev: five CUDA events bracketing the permutation draw, the rollout, the
        bootstrap + GAE and the PPO updates."""
        torch, s, stream = self.torch, self.simx, self.torch.cuda.current_stream()

        def mark(i):
            if ev:
                ev[i].record(stream)
        mark(0)
        for e in range(self.epochs):
            self.perm[e] = torch.randperm(self.n_rows, device="cuda", generator=self.gen)
        mark(1)
        self.sim.rollout("sample", self.H, self.buf, self.policy)
        mark(2)
        self.sim.observe(self.obs_next)
        s.policy_forward(self.policy, self.obs_next, self.E, "argmax", 0, 0, value=self.last,
                         workspace=self.pf_ws)
        s.compute_returns_gae(self.buf["reward"], self.buf["done"], GAMMA, LAMBDA, self.ret,
                              adv=self.adv, val=self.buf["value"], last_val=self.last)
        mark(3)
        if self.graph is None:
            self._updates()          # eager: sizes every library-side buffer first
            self.graph = torch.cuda.CUDAGraph()
            l0 = s.launches()
            with torch.cuda.graph(self.graph, capture_error_mode="relaxed"):
                self._updates()
            self.graph_launches = s.launches() - l0   # library kernels in one replay
        else:
            self.graph.replay()
            self.replays += 1
        mark(4)

    def close(self):
        self.sim.close()


def _minibatch_loss_ms(st, torch, reps: int = 20) -> dict:
    """Average duration of one loss-gradient call and one Adam call of the step's update
    loop, each timed alone (CUDA events on the stream, after the timed region)."""
    s = st.simx
    idx = st.perm[0, :st.mb]
    out = {}
    for name, fn in (("loss", lambda: s.ppo_loss_grad(st.policy, st.buf, st.ret, st.adv, idx, st.mb,
                                                      "ppo", CLIP, C_VALUE, C_ENTROPY, st.grad,
                                                      st.stats, st.loss_ws,
                                                      precision=st.precision)),
                     ("adam", lambda: s.adam_step(st.params, st.grad, st.m, st.v, st.t_dev, LR,
                                                  max_grad_norm=MAX_NORM, workspace=st.adam_ws))):
        fn()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            fn()
        e1.record()
        torch.cuda.synchronize()
        out[name] = e0.elapsed_time(e1) / reps
    return out


def _c2_extra(simx, W, torch, reps: int = 5) -> dict:
    """The single-server workload (4096 envs x 512, MMPP, MLP 16-64-64-12, REINFORCE with
    a mean baseline): rollout + returns + baseline + loss gradient over all rows."""
    E, H = 4096, W.HORIZON["c2"]
    dims, hv = W.mlp_dims("c2")
    Ws, bs = W.mlp_weights(dims, 1)
    pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws], [torch.from_numpy(b).cuda() for b in bs], hv)
    sim = simx.Sim(W.c2(E))
    sim.reset(0x5EED0002)
    n = E * H
    buf = simx.alloc_rollout(E, sim.D, H)
    ret = torch.empty((H, E), device="cuda")
    adv = torch.empty((H, E), device="cuda")
    mean = torch.empty(1, device="cuda")
    ws_b = torch.empty(simx.returns_baseline_workspace_size(n), dtype=torch.uint8, device="cuda")
    grad = torch.empty(pol.n_params, device="cuda")
    stats = torch.empty(5, device="cuda")
    ws_l = torch.empty(simx.ppo_loss_grad_workspace_size(pol, n), dtype=torch.uint8, device="cuda")

    def step():
        sim.rollout("sample", H, buf, pol)
        simx.compute_returns_gae(buf["reward"], buf["done"], GAMMA, -1.0, ret)
        simx.returns_baseline(ret, adv, mean, ws_b)
        simx.ppo_loss_grad(pol, buf, ret, adv, None, n, "reinforce", 0.2, 0.0, 0.0, grad, stats,
                           ws_l, precision="tf32")
    for _ in range(3):
        step()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        step()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    sim.close()
    return {"workload": "c2: 4096 envs x 512, MMPP 300/3000 req/s, MLP 16-64-64-12, REINFORCE + "
                        "mean baseline, loss over all rows (tf32)",
            "ms_per_step": ms, "decision_steps_per_s": n / (ms * 1e-3), "steps": reps}


def _c5_extra(simx, W, torch, E: int = 1048576) -> dict:
    """c5 at its largest size: the argmax rollout of 1,048,576 envs x 1024 steps and GAE."""
    H = W.HORIZON["c5"]
    dims, hv = W.mlp_dims("c5")
    Ws, bs = W.policy_weights("c5", dims, 1)
    pol = simx.Policy([torch.from_numpy(w).cuda() for w in Ws], [torch.from_numpy(b).cuda() for b in bs], hv)
    sim = simx.Sim(W.c5(E))
    sim.reset(W.SEED["c5"])
    buf = simx.alloc_rollout(E, sim.D, H, has_value=True)
    sim.rollout("argmax", 8, buf, pol)
    adv = torch.empty((H, E), device="cuda")
    ret = torch.empty((H, E), device="cuda")
    last = torch.zeros(E, device="cuda")
    e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
    e[0].record()
    sim.rollout("argmax", H, buf, pol)
    e[1].record()
    simx.compute_returns_gae(buf["reward"], buf["done"], GAMMA, LAMBDA, ret, adv=adv,
                             val=buf["value"], last_val=last)
    e[2].record()
    torch.cuda.synchronize()
    r_ms, g_ms = e[0].elapsed_time(e[1]), e[1].elapsed_time(e[2])
    st, _ = sim.last_status()
    sim.close()
    del buf, adv, ret
    torch.cuda.empty_cache()
    return {"workload": "c5: %d envs x %d, argmax, MLP 13-128-128-16+V" % (E, H), "status": st,
            "rollout_ms": r_ms, "decision_steps_per_s": E * H / (r_ms * 1e-3),
            "gae_ms": g_ms, "gae_samples_per_s": E * H / (g_ms * 1e-3)}


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

    # Replicas: every rank simulates and trains on its own 65,536 envs (seed offset by
    # rank); no data-path collective, only the timing barrier and max-reduction.
    st = PPOStep(simx, W, torch, replica_seed(rank), a.epochs, a.loss_precision, local)
    E, H, n = st.E, st.H, st.n_rows
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    fp = measure_fp32_peak(simx, torch)

    for _ in range(a.warmup):
        st.run()
    torch.cuda.synchronize()

    cj0 = st.sim.save()[:, 2].astype(np.int64)   # arrival candidates drawn so far
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(a.steps)]
    clocks = Clocks(local) if rank == 0 else None
    l0, r0 = simx.launches(), st.replays
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    t_wall = time.perf_counter()
    for k in range(a.steps):
        flush.zero_()  # evict L2 between steps (outside the timed events)
        st.run(evs[k])
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    t_wall = time.perf_counter() - t_wall
    # launches made from the host plus the library kernels inside every graph replay
    launches = simx.launches() - l0 + (st.replays - r0) * st.graph_launches
    clk = clocks.stop() if clocks else None
    cj1 = st.sim.save()[:, 2].astype(np.int64)
    cand_per_launch = float((cj1 - cj0).sum()) / a.steps
    state_status = st.sim.last_status()

    phase_ms = [[evs[k][i].elapsed_time(evs[k][i + 1]) for i in range(4)] for k in range(a.steps)]
    step_ms = [evs[k][0].elapsed_time(evs[k][4]) for k in range(a.steps)]
    ms = statistics.mean(step_ms)
    ph = [statistics.mean(p[i] for p in phase_ms) for i in range(4)]
    ms = max_over_ranks(ms, dist, "cuda")
    value = job_value(world, n, ms)
    if state_status[0] != 0:
        raise RuntimeError("device status 0x%x after the timed region" % state_status[1])

    # end to end through the public API: the policy's parameters in from pinned host
    # memory, the updated parameters and the last update's statistics back, every step
    e2e = None
    if not a.no_e2e:
        hp = torch.from_numpy(st.host_params.copy()).pin_memory()
        hout = torch.empty_like(hp).pin_memory()
        hs = torch.empty(5, dtype=torch.float32).pin_memory()
        k_e2e = max(3, min(a.steps, 10))
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(k_e2e):
            st.params.copy_(hp, non_blocking=True)
            st.run()
            hout.copy_(st.params, non_blocking=True)
            hs.copy_(st.stats, non_blocking=True)
            torch.cuda.synchronize()
        t_e2e = (time.perf_counter() - t0) / k_e2e
        t_e2e = max_over_ranks(t_e2e, dist, "cuda")
        e2e = {"value": job_value(world, n, t_e2e * 1e3), "unit": UNIT,
               "h2d_bytes_per_step": hp.numel() * 4,
               "d2h_bytes_per_step": hout.numel() * 4 + hs.numel() * 4}

    mb_ms = _minibatch_loss_ms(st, torch)

    # the policy-free batched step (Sec. 5.1 Shortest-Queue router) of the multi-server
    # environment: state read and written every step, HBM-bound
    hbm_step = None if a.no_hbm_step else [hbm_step_measure(simx, W, torch, E=e)
                                            for e in (65536, 1048576)]
    extras = None
    if rank == 0 and not a.no_extras:
        extras = {"c2": _c2_extra(simx, W, torch), "c5_1m": _c5_extra(simx, W, torch)}

    # roofline of the dominant kernel
    peaks, src = _peaks()
    sm_mhz = float(peaks.get("sm_max_mhz", 2070.0))
    fp32_nominal = fp["sms"] * 128 * 2 * sm_mhz * 1e6 / 1e12  # FMA lanes x maximum clock
    fp32_src = ("%d SMs x 128 FP32 lanes x 2 flops x %.0f MHz (unit counts and maximum clock); "
                "the library's FMA probe measures %.1f TFLOP/s" % (fp["sms"], sm_mhz, fp["tflops"]))
    dims = st.dims
    P = sum(dims[l] * dims[l + 1] for l in range(len(dims) - 1))
    hidden = sum(dims[1:-1])
    A = dims[-1] - 1
    flop_rollout = n * (2.0 * P + 20.0 * hidden + 20.0 * A) + 15.0 * cand_per_launch
    flop_mb = st.mb * (6.0 * P - 2.0 * dims[0] * dims[1])
    update_ms = ph[3]
    phases = {"permutation_ms": ph[0], "rollout_ms": ph[1], "bootstrap_gae_ms": ph[2],
              "ppo_update_ms": update_ms, "minibatches_per_step": st.n_mb * st.epochs,
              "loss_grad_call_ms": mb_ms["loss"], "adam_call_ms": mb_ms["adam"]}
    tf32_peak = float(peaks.get("bf16_tflops", 1900.0)) * 0.5
    loss_share = mb_ms["loss"] / max(mb_ms["loss"] + mb_ms["adam"], 1e-9)
    loss_live_ms = update_ms * loss_share / (st.n_mb * st.epochs)
    ach_l = flop_mb / (loss_live_ms * 1e-3) / 1e12
    if a.loss_precision == "tf32":
        roof_loss = {"kernel": "loss gradient (tensor-core tf32 kernels)", "bound": "tensor",
                     "achieved": ach_l, "peak": tf32_peak, "unit": "TFLOP/s", "frac": ach_l / tf32_peak,
                     "traffic": None, "peak_source": "%s bf16_tflops x 0.5 (nominal tf32 / bf16 rate)" % src,
                     "ms_per_call": loss_live_ms}
    else:
        roof_loss = {"kernel": "loss gradient (FP32 SIMT kernels)", "bound": "alu", "achieved": ach_l,
                     "peak": fp32_nominal, "unit": "TFLOP/s", "frac": ach_l / fp32_nominal,
                     "traffic": None, "peak_source": fp32_src, "ms_per_call": loss_live_ms}
    ach_r = flop_rollout / (ph[1] * 1e-3) / 1e12
    roof_rollout = {"kernel": "k_rollout (simulation + fused policy)", "bound": "alu",
                    "achieved": ach_r, "peak": fp32_nominal, "unit": "TFLOP/s",
                    "frac": ach_r / fp32_nominal, "traffic": ROLLOUT_DRAM_BYTES,
                    "traffic_source": ROLLOUT_DRAM_SOURCE, "peak_source": fp32_src,
                    "flop_per_launch": flop_rollout}
    # the dominant single kernel: the loss-gradient call is five kernels (weight images,
    # per-tile forward/backward, weight-gradient products, two reductions), the largest
    # about two thirds of the call (profiles/), so k_rollout leads unless the whole call
    # outweighs it by more than that
    loss_total_ms = update_ms * loss_share
    roof = roof_rollout if ph[1] >= 0.7 * loss_total_ms else roof_loss
    roof_rollout["dominance"] = ("k_rollout %.1f ms per step; the loss-gradient calls %.1f ms per "
                                 "step over five kernels" % (ph[1], loss_total_ms))

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": a.steps,
            "warmup": a.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32+tf32" if a.loss_precision == "tf32" else "f32",
            "data": "synthetic",
            "config": {"workload": WORKLOAD_TEXT, "envs_per_gpu": E, "horizon": H,
                       "ppo_epochs_per_step": st.epochs, "minibatch": st.mb,
                       "l2": "flushed (256 MB write) before every timed step",
                       "parallelism": "replicas" if world > 1 else "single GPU",
                       "loss_precision": "tf32 tensor cores, fp32 accumulation (parity 1e-2)"
                       if a.loss_precision == "tf32" else "fp32 (parity 1e-5)"},
            "phases_ms": phases,
            "roofline": roof,
            "roofline_rollout": roof_rollout,
            "roofline_loss": roof_loss,
            "e2e": e2e,
            "hbm_step": hbm_step,
            "extras": extras,
            "gpu_launches": launches,
            "clocks": clk,
            "wall_s": t_wall,
        }
        if world == 1 and not a.no_cpu_baseline:
            line["cpu_baseline"] = cpu_baseline(a.epochs)
        print(json.dumps(line), flush=True)
    st.close()
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
    if a.grid_rollout:
        run_grid_rollout(a.grid_rollout, a.grid_envs)
        return
    if a.rollout_only:
        from paper_2607_05272_gb300 import workloads as W
        run_rollout_only(a.rollout_only, a.rollout_envs or W.CONFIGS[a.rollout_only]()["n_envs"],
                         a.rollout_steps or W.HORIZON[a.rollout_only])
        return
    if a.hbm_step_only:
        import torch

        from paper_2607_05272_gb300 import build as B
        from paper_2607_05272_gb300 import workloads as W
        B.build()
        from paper_2607_05272_gb300 import simx
        print(json.dumps(hbm_step_measure(simx, W, torch, E=a.hbm_step_only)), flush=True)
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
