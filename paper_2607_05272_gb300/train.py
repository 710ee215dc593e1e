"""On-device policy-gradient training loop (Sec. 4.3: REINFORCE and PPO).

Every numeric step of an iteration runs in the library's kernels:
  rollout_collect (simulators + policy) -> compute_returns_gae -> [returns_baseline]
  -> ppo_loss_grad -> simx_adam_step,
over one flat parameter vector that the policy's layers view, so the optimiser updates
the policy in place and the next rollout uses the new weights.  PyTorch only holds the
device buffers and draws PPO's minibatch permutations (torch.randperm on the device).

REINFORCE uses the discounted returns with a baseline: the learned value row when the
policy has one (advantage G_t - V_t, computed as GAE with lambda = 1, whose telescoping
sum equals it exactly), else the mean return over the batch.  PPO uses GAE(gamma,
lambda) advantages, `epochs` passes of minibatches, and the clipped surrogate.

Command line: ``python -m paper_2607_05272_gb300.train --workload c3s --iters 150``
trains on a workload and reports the trained policy's mean reward per decision beside
the policy-free baselines on the same envs.
"""
from __future__ import annotations

import argparse
import json
import time

import numpy as np

from . import simx
from . import workloads as W


class Trainer:
    def __init__(self, cfg: dict, dims, has_value: bool, acts=None, weights=None, mask=None,
                 algo: str = "reinforce", horizon: int = 256, lr: float = 3e-4,
                 gamma: float = 0.99, lam: float = 0.95, epochs: int = 4, minibatch: int = 8192,
                 clip_eps: float = 0.2, c_value: float = 0.5, c_entropy: float = 0.01,
                 max_grad_norm: float = 0.5, seed: int = 1, precision: str = "fp32",
                 graph: bool = False):
        import torch
        self.torch = torch
        self.cfg, self.algo, self.H = cfg, algo, horizon
        self.gamma, self.lam, self.epochs, self.mb = gamma, lam, epochs, minibatch
        self.clip_eps, self.c_value, self.c_entropy = clip_eps, c_value, c_entropy
        self.lr, self.max_grad_norm, self.precision = lr, max_grad_norm, precision
        self.has_value = bool(has_value)
        Ws, bs = weights if weights is not None else W.mlp_weights(list(dims), seed)
        flat = np.concatenate([np.concatenate([w.ravel(), b.ravel()]) for w, b in zip(Ws, bs)])
        self.params = torch.from_numpy(flat.astype(np.float32)).cuda()
        self.policy = simx.Policy.from_flat(self.params, list(dims), has_value, acts)
        n = self.params.numel()
        self.m = torch.zeros(n, device="cuda")
        self.v = torch.zeros(n, device="cuda")
        self.mask = None if mask is None else torch.from_numpy(np.asarray(mask, np.uint8)).cuda()
        self.grad = torch.empty(n, device="cuda")
        self.stats = torch.empty(5, device="cuda")
        self.adam_ws = torch.empty(simx.adam_workspace_size(n), dtype=torch.uint8, device="cuda")
        self.t = 0                                                      # updates so far (host)
        self.t_dev = torch.zeros(1, dtype=torch.int64, device="cuda")   # Adam's step counter
        E = cfg["n_envs"]
        self.E = E
        self.sim = simx.Sim(cfg)
        self.sim.reset(seed)
        self.buf = simx.alloc_rollout(E, self.sim.D, horizon, has_value=self.has_value)
        self.ret = torch.empty((horizon, E), device="cuda")
        self.adv = torch.empty((horizon, E), device="cuda")
        self.last = torch.zeros(E, device="cuda")  # V of the state after the rollout
        self.obs_next = torch.empty((self.sim.D, E), device="cuda")
        # the bootstrap forward's own repack buffer (captured graphs keep its address)
        self.pf_ws = torch.empty(simx.policy_forward_workspace_size(self.policy),
                                 dtype=torch.uint8, device="cuda")
        self.n_rows = E * horizon
        rows = self.n_rows if algo == "reinforce" else min(minibatch, self.n_rows)
        self.loss_ws = torch.empty(simx.ppo_loss_grad_workspace_size(self.policy, rows),
                                   dtype=torch.uint8, device="cuda")
        self.base_ws = torch.empty(simx.returns_baseline_workspace_size(self.n_rows),
                                   dtype=torch.uint8, device="cuda")
        self.mean = torch.empty(1, device="cuda")
        self.gen = torch.Generator(device="cuda")
        self.gen.manual_seed(seed)
        # PPO minibatch rows of every epoch, drawn before each iteration (outside a graph)
        self.perm = torch.empty((epochs, self.n_rows), dtype=torch.int64, device="cuda")
        self.n_mb = self.n_rows // minibatch if algo == "ppo" else 1
        self.use_graph = graph
        self.graph = None

    def _update(self, idx, n):
        simx.ppo_loss_grad(self.policy, self.buf, self.ret, self.adv, idx, n, self.algo,
                           self.clip_eps, self.c_value if self.has_value else 0.0,
                           self.c_entropy, self.grad, self.stats, self.loss_ws,
                           precision=self.precision)
        simx.adam_step(self.params, self.grad, self.m, self.v, self.t_dev, self.lr,
                       max_grad_norm=self.max_grad_norm, mask=self.mask, workspace=self.adam_ws)

    def iteration(self) -> dict:
        """One rollout of H decisions per env and the policy update(s) on it.  With
        graph=True the first iteration runs eagerly (it sizes the library's internal
        buffers), the second captures the whole iteration in a CUDA graph, and every
        iteration from then on replays it: the same kernels on the same buffers, with
        Adam's step counter advanced on the device."""
        if self.algo == "ppo":
            for e in range(self.epochs):
                self.perm[e] = self.torch.randperm(self.n_rows, device="cuda", generator=self.gen)
        if not self.use_graph or self.t == 0:
            self._body()
        else:
            if self.graph is None:
                self.graph = self.torch.cuda.CUDAGraph()
                # relaxed: the library's host side sets kernel attributes, no stream work
                with self.torch.cuda.graph(self.graph, capture_error_mode="relaxed"):
                    self._body()
            self.graph.replay()
        self.t += self.n_mb * (self.epochs if self.algo == "ppo" else 1)
        st = self.stats.cpu().numpy()
        return {"mean_reward": float(self.buf["reward"].mean().item()), "loss": float(st[0]),
                "entropy": float(st[3]), "updates": self.t}

    def _body(self):
        b = self.buf
        self.sim.rollout("sample", self.H, b, self.policy)
        if self.has_value:  # bootstrap value of each env's current state
            self.sim.observe(self.obs_next)
            simx.policy_forward(self.policy, self.obs_next, self.E, "argmax", 0, 0,
                                value=self.last, workspace=self.pf_ws)
        if self.algo == "reinforce":
            if self.has_value:  # learned baseline: A = G - V (GAE with lambda = 1)
                simx.compute_returns_gae(b["reward"], b["done"], self.gamma, 1.0, self.ret,
                                         adv=self.adv, val=b["value"], last_val=self.last)
            else:               # mean-return baseline
                simx.compute_returns_gae(b["reward"], b["done"], self.gamma, -1.0, self.ret,
                                         last_val=self.last)
                simx.returns_baseline(self.ret, self.adv, self.mean, self.base_ws)
            self._update(None, self.n_rows)
        else:
            simx.compute_returns_gae(b["reward"], b["done"], self.gamma, self.lam, self.ret,
                                     adv=self.adv, val=b["value"], last_val=self.last)
            for e in range(self.epochs):
                for i in range(self.n_mb):
                    self._update(self.perm[e, i * self.mb:(i + 1) * self.mb], self.mb)


def evaluate(cfg: dict, mode: str, horizon: int, seed: int, policy=None, warm: int = 1) -> dict:
    """Mean reward per decision and mean queueing wait per dispatched request (ms) of a
    policy-free baseline (or a given policy) over one rollout of fresh envs, after `warm`
    rollouts that are not counted."""
    sim = simx.Sim(cfg)
    sim.reset(seed)
    buf = simx.alloc_rollout(cfg["n_envs"], sim.D, horizon,
                             has_value=bool(policy is not None and policy.has_value))
    for _ in range(warm):
        sim.rollout(mode, horizon, buf, policy)
    s0 = sim.stats()
    sim.rollout(mode, horizon, buf, policy)
    s1 = sim.stats()
    r = float(buf["reward"].mean().item())
    sim.close()
    n = max(s1["dispatched"] - s0["dispatched"], 1)
    out = {"reward": r, "mean_wait_ms": (s1["sum_wait_us"] - s0["sum_wait_us"]) / n / 1000.0,
           "dropped": s1["dropped"] - s0["dropped"]}
    if cfg["mode"] == W.MODE_ROUTE and cfg["obs_extra"] and cfg["n_types"] == 2:
        # where each request type went: the observation's arriving-type one-hot sits after
        # the 3 features per server and the rate estimate; the action's major is the server
        K = cfg["n_servers"]
        slow = buf["obs"][:, 3 * K + 2, :] > 0.5
        srv = (buf["action"].long() // cfg["n_bsizes"])
        share = {}
        for name, sel in (("fast", ~slow), ("slow", slow)):
            cnt = [int(((srv == k) & sel).sum().item()) for k in range(K)]
            tot = max(sum(cnt), 1)
            share[name] = [c / tot for c in cnt]
        out["route_share"] = share
    return out


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--workload", default="c3s")
    ap.add_argument("--envs", type=int, default=4096)
    ap.add_argument("--horizon", type=int, default=256)
    ap.add_argument("--iters", type=int, default=150)
    ap.add_argument("--algo", default="reinforce", choices=["reinforce", "ppo"])
    ap.add_argument("--lr", type=float, default=1e-3)
    ap.add_argument("--seed", type=int, default=1)
    ap.add_argument("--every", type=int, default=10)
    ap.add_argument("--no-graph", action="store_true", help="launch every kernel from Python")
    a = ap.parse_args(argv)
    import torch
    cfg = W.CONFIGS[a.workload](a.envs)
    dims, hv = W.mlp_dims(a.workload)
    Ws, bs = W.policy_weights(a.workload, dims, a.seed)
    mask = W.param_mask(a.workload, dims)
    tr = Trainer(cfg, dims, hv, W.mlp_acts(a.workload), (Ws, bs), mask, algo=a.algo,
                 horizon=a.horizon, lr=a.lr, seed=a.seed, graph=not a.no_graph)
    t0 = time.perf_counter()
    hist = []
    for i in range(a.iters):
        s = tr.iteration()
        hist.append(s["mean_reward"])
        if (i + 1) % a.every == 0 or i == 0:
            print(json.dumps({"iter": i + 1, **s}), flush=True)
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    ev_seed = a.seed + 1000
    res = {"workload": a.workload, "algo": a.algo, "iters": a.iters, "train_s": wall,
           "decisions_trained": a.iters * a.envs * a.horizon,
           "first_iter_reward": hist[0], "last10_reward": float(np.mean(hist[-10:])),
           "eval": {"trained_sample": evaluate(cfg, "sample", a.horizon, ev_seed, tr.policy),
                    "trained_argmax": evaluate(cfg, "argmax", a.horizon, ev_seed, tr.policy)}}
    modes = ["sq", "rr", "random"] if cfg["mode"] == W.MODE_ROUTE else ["static", "random"]
    for m in modes:
        res["eval"][m] = evaluate(cfg, m, a.horizon, ev_seed)
    print(json.dumps(res), flush=True)
    return res


if __name__ == "__main__":
    main()
