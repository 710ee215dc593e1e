"""Thin ctypes binding of libsimx.so (include/simx.h): argument marshalling only.

Every step of the rollout, returns, baseline and loss computation runs in the CUDA
library; this module turns torch tensors and dicts into the C structs and pointers
the ABI takes, and raises ``SimxError`` for a non-OK status.  There is no CPU
fallback: if the library is missing the first call raises.
"""
from __future__ import annotations

import ctypes as C
import os
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libsimx.so")
_lock = threading.Lock()
_lib = None

OK, EINVAL, ENOMEM, ECUDA, EOVERFLOW, ESTATE = range(6)
POLICY = {"sample": 0, "argmax": 1, "static": 2, "rr": 3, "sq": 4, "random": 5, "external": 6}
ALGO = {"reinforce": 0, "ppo": 1}
TRACE_WIDTH = 4
MAX_LAYERS = 6  # SIMX_MAX_LAYERS
STATE_HEADER_WORDS = 32


class SimxError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__("simx status %d: %s" % (status, msg))
        self.status = status


class Config(C.Structure):
    _fields_ = [
        ("abi_version", C.c_uint32), ("mode", C.c_uint32), ("n_envs", C.c_uint32),
        ("n_servers", C.c_uint32), ("n_types", C.c_uint32), ("queue_cap", C.c_uint32),
        ("episode_len", C.c_uint32), ("arrival_kind", C.c_uint32),
        ("cand_mean_gap_us", C.c_float), ("n_mod_states", C.c_uint32),
        ("accept_thr", C.c_uint32 * 2), ("dwell_mean_us", C.c_float),
        ("epoch_us", C.c_uint32), ("diurnal_len", C.c_uint32),
        ("diurnal_rate", C.c_float * 128), ("burst_sigma", C.c_float),
        ("type0_thr", C.c_uint32), ("alpha_us", C.c_uint32 * 2), ("beta_us", C.c_uint32 * 2),
        ("cost_type", C.c_int32), ("cost_kind", C.c_uint32), ("cost_scale_us", C.c_float),
        ("pareto_inv_alpha", C.c_float), ("w_wait", C.c_float * 2), ("n_bsizes", C.c_uint32),
        ("bsizes", C.c_uint32 * 8), ("static_bi", C.c_uint32), ("obs_extra", C.c_uint32),
        ("obs_dim", C.c_uint32), ("t_window_us", C.c_float), ("rate_scale", C.c_float),
        ("rate_ref", C.c_float), ("busy_norm_us", C.c_float), ("phase_period_us", C.c_uint32),
        ("dwell_kind", C.c_uint32), ("srv_speed16", C.c_uint32 * 8),
        ("action_layout", C.c_uint32),
    ]


class Mlp(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("dims", C.c_int32 * (MAX_LAYERS + 1)),
                ("W", C.c_void_p * MAX_LAYERS), ("b", C.c_void_p * MAX_LAYERS),
                ("has_value", C.c_int32), ("act", C.c_int32 * MAX_LAYERS),
                ("grid", C.c_int32), ("gx", C.c_int32 * MAX_LAYERS)]


ACT = {"tanh": 0, "identity": 1, "gelu": 2}


class Rollout(C.Structure):
    _fields_ = [("ld", C.c_int64), ("obs", C.c_void_p), ("action", C.c_void_p),
                ("logp", C.c_void_p), ("value", C.c_void_p), ("reward", C.c_void_p),
                ("done", C.c_void_p), ("trace", C.c_void_p)]


class LossParams(C.Structure):
    _fields_ = [("algo", C.c_int32), ("clip_eps", C.c_float), ("c_value", C.c_float),
                ("c_entropy", C.c_float), ("precision", C.c_int32)]


PRECISION = {"fp32": 0, "tf32": 1}


class Counters(C.Structure):
    _fields_ = [("arrived", C.c_uint64), ("dropped", C.c_uint64), ("dispatched", C.c_uint64),
                ("batches", C.c_uint64), ("queued", C.c_uint64), ("sum_wait_us", C.c_uint64),
                ("decisions", C.c_uint64), ("envs_flagged", C.c_uint32), ("status_or", C.c_uint32)]


# (name, restype, argtypes) of every exported function, in header order.
P, I32, I64, U32, U64, F, SZ = (C.c_void_p, C.c_int32, C.c_int64, C.c_uint32, C.c_uint64,
                                C.c_float, C.c_size_t)
SIGNATURES = [
    ("simx_obs_dim", U32, [P]),
    ("simx_state_words", U64, [P]),
    ("sim_create", C.c_int, [P, C.c_int, P]),
    ("sim_destroy", None, [P]),
    ("sim_reset", C.c_int, [P, U64, P]),
    ("sim_set_trace", C.c_int, [P, P, P, P, U32]),
    ("simx_adam_workspace_size", SZ, [I64]),
    ("simx_adam_step", C.c_int, [P, P, P, P, P, I64, I64, P, P, P, SZ, P]),
    ("sim_observe", C.c_int, [P, P, I64, P]),
    ("sim_step_batched", C.c_int, [P, P, P, C.c_int, P, I64, P, P, P, P, P]),
    ("rollout_collect", C.c_int, [P, P, C.c_int, I32, P, P]),
    ("simx_launch_shape", C.c_int, [P, P, C.c_int, P]),
    ("policy_forward", C.c_int, [P, P, I64, I64, C.c_int, U64, U32, U32, P, P, P, P, P]),
    ("policy_forward_workspace_size", SZ, [P]),
    ("policy_forward_ws", C.c_int, [P, P, I64, I64, C.c_int, U64, U32, U32, P, P, P, P, P, SZ, P]),
    ("compute_returns_gae", C.c_int, [P, P, P, P, I64, I64, I64, F, F, P, P, P]),
    ("returns_baseline_workspace_size", SZ, [I64]),
    ("returns_baseline", C.c_int, [P, I64, P, P, P, SZ, P]),
    ("ppo_loss_grad_workspace_size", SZ, [P, I64]),
    ("ppo_loss_grad", C.c_int, [P, P, I64, P, P, P, I64, P, P, P, P, SZ, P]),
    ("ppo_loss_grad_noalloc", C.c_int, [P, P, I64, P, P, P, I64, P, P, P, P]),
    ("sim_stats", C.c_int, [P, P]),
    ("sim_save", C.c_int, [P, P, U64]),
    ("sim_load", C.c_int, [P, P, U64]),
    ("simx_last_status", C.c_int, [P, P]),
    ("simx_launches", U64, []),
    ("simx_fma_probe", C.c_int, [I64, P, P, P]),
    ("simx_fma_probe_sink_floats", SZ, []),
    ("simx_strerror", C.c_char_p, [C.c_int]),
    ("simx_last_error", C.c_char_p, []),
]


def lib():
    """Load libsimx.so (built by build.py); raise if it is missing."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError("libsimx.so is not built (%s); run "
                                   "paper_2607_05272_gb300.build.build()" % LIB_PATH)
            L = C.CDLL(LIB_PATH)
            for name, res, args in SIGNATURES:
                fn = getattr(L, name)
                fn.restype = res
                fn.argtypes = args
            _lib = L
    return _lib


def _check(status: int):
    if status != OK:
        raise SimxError(status, lib().simx_last_error().decode())


def make_config(cfg: dict) -> Config:
    c = Config()
    for name, _ in Config._fields_:
        v = cfg[name]
        if isinstance(v, (list, tuple)):
            arr = getattr(c, name)
            for i, x in enumerate(v):
                arr[i] = x
        else:
            setattr(c, name, v)
    return c


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _stream(stream=None):
    if stream is not None:
        return C.c_void_p(stream)
    import torch
    return C.c_void_p(torch.cuda.current_stream().cuda_stream)


class Policy:
    """A simx_mlp over device tensors W_l [out, in] and b_l [out] (fp32, contiguous);
    acts: the activation after each hidden layer ("tanh", "identity" or "gelu"; default
    tanh); grid: for a grid policy (the exact policy forward), the input grid exponent of
    every layer (its weights must lie on the grid that workloads.grid_check checks)."""

    def __init__(self, Ws, bs, has_value: bool, acts=None, grid=None):
        self.Ws = [w.contiguous() for w in Ws]
        self.bs = [b.contiguous() for b in bs]
        self.has_value = bool(has_value)
        m = Mlp()
        m.n_layers = len(self.Ws)
        m.dims[0] = self.Ws[0].shape[1]
        for l, w in enumerate(self.Ws):
            assert w.dtype.is_floating_point and w.is_cuda
            m.dims[l + 1] = w.shape[0]
            m.W[l] = w.data_ptr()
            m.b[l] = self.bs[l].data_ptr()
        m.has_value = int(self.has_value)
        for l, a in enumerate(acts or []):
            m.act[l] = ACT[a] if isinstance(a, str) else int(a)
        if grid is not None:
            m.grid = 1
            for l, e in enumerate(grid):
                m.gx[l] = int(e)
        self.c = m

    flat = None  # the flat parameter vector when built by from_flat

    @classmethod
    def from_flat(cls, flat, dims, has_value: bool, acts=None, grid=None):
        """A policy whose W_l, b_l are views into one flat fp32 device vector in the
        gradient's order (W0, b0, W1, b1, ...): the optimiser updates it in place."""
        Ws, bs, off = [], [], 0
        for k, n in zip(dims[:-1], dims[1:]):
            Ws.append(flat[off:off + n * k].view(n, k))
            off += n * k
            bs.append(flat[off:off + n])
            off += n
        assert off == flat.numel()
        pol = cls(Ws, bs, has_value, acts, grid)
        pol.flat = flat
        return pol

    @property
    def n_actions(self) -> int:
        return self.Ws[-1].shape[0] - (1 if self.has_value else 0)

    @property
    def n_params(self) -> int:
        return sum(w.numel() + b.numel() for w, b in zip(self.Ws, self.bs))


def launches() -> int:
    """Kernels the library has launched so far in this process."""
    return lib().simx_launches()


def obs_dim(cfg: dict) -> int:
    c = make_config(cfg)
    return lib().simx_obs_dim(C.byref(c))


def state_words(cfg: dict) -> int:
    c = make_config(cfg)
    return lib().simx_state_words(C.byref(c))


class Sim:
    """A simulator context (sim_create / sim_destroy)."""

    def __init__(self, cfg: dict, device: int = 0):
        self.cfg = dict(cfg)
        self._c = make_config(cfg)
        h = C.c_void_p()
        _check(lib().sim_create(C.byref(self._c), device, C.byref(h)))
        self._h = h
        self.E = cfg["n_envs"]
        self.D = obs_dim(cfg)
        self.words = state_words(cfg)
        self._trace = None
        if cfg.get("trace") is not None:
            self.set_trace(*cfg["trace"])

    def set_trace(self, gap_us, type=None, cost_us=None):
        """Trace replay input (sim_set_trace): per-request gaps in us, types and costs;
        numpy arrays are copied to the device, device tensors are used as they are
        (int32 / uint8 / int32, values below 2^31).  Takes effect at the next reset."""
        import torch

        def dev(x, dt):
            if x is None:
                return None
            t = x if isinstance(x, torch.Tensor) else torch.from_numpy(np.ascontiguousarray(x).astype(dt))
            return t.contiguous().cuda()
        g = dev(gap_us, np.int32)
        ty = dev(type, np.uint8)
        co = dev(cost_us, np.int32)
        _check(lib().sim_set_trace(self._h, g.data_ptr(), _ptr(ty), _ptr(co), len(g)))
        self._trace = (g, ty, co)

    def close(self):
        if getattr(self, "_h", None):
            lib().sim_destroy(self._h)
            self._h = None

    __del__ = close

    def reset(self, seed: int, stream=None):
        _check(lib().sim_reset(self._h, seed, _stream(stream)))

    def observe(self, obs, stream=None):
        _check(lib().sim_observe(self._h, _ptr(obs), obs.shape[-1], _stream(stream)))

    def step(self, policy_mode: str, policy: Policy = None, actions=None, obs=None, reward=None,
             done=None, action=None, logp=None, stream=None):
        ld = obs.shape[-1] if obs is not None else self.E
        _check(lib().sim_step_batched(
            self._h, _ptr(actions), C.byref(policy.c) if policy else None, POLICY[policy_mode],
            _ptr(obs), ld, _ptr(reward), _ptr(done), _ptr(action), _ptr(logp), _stream(stream)))

    def rollout(self, policy_mode: str, horizon: int, buf: dict, policy: Policy = None,
                stream=None):
        r = Rollout()
        r.ld = buf["reward"].shape[-1]
        for k in ("obs", "action", "logp", "value", "reward", "done", "trace"):
            t = buf.get(k)
            setattr(r, k, None if t is None else t.data_ptr())
        _check(lib().rollout_collect(self._h, C.byref(policy.c) if policy else None,
                                     POLICY[policy_mode], horizon, C.byref(r), _stream(stream)))

    def launch_shape(self, policy_mode: str, policy: Policy = None) -> dict:
        """The launch rollout_collect takes (simx_launch_shape): kernel ("fused" or
        "thread"), lanes per env, threads per block, warp-local policy forward, whether
        a grid policy's forward runs on the tensor cores, and whether the FP32 forward
        stages its weights in shared memory."""
        out = (C.c_int32 * 6)()
        _check(lib().simx_launch_shape(self._h, C.byref(policy.c) if policy else None,
                                       POLICY[policy_mode], out))
        return dict(kernel="thread" if out[0] else "fused", lanes=out[1], threads=out[2],
                    mlp_warp=bool(out[3]), tensor_cores=bool(out[4]), staged=bool(out[5]))

    def stats(self) -> dict:
        c = Counters()
        _check(lib().sim_stats(self._h, C.byref(c)))
        return {name: getattr(c, name) for name, _ in Counters._fields_}

    def last_status(self) -> tuple:
        code = C.c_uint32()
        st = lib().simx_last_status(self._h, C.byref(code))
        return st, code.value

    def save(self):
        import numpy as np
        out = np.zeros(self.E * self.words, np.uint32)
        _check(lib().sim_save(self._h, out.ctypes.data, out.size))
        return out.reshape(self.E, self.words)

    def load(self, words):
        import numpy as np
        w = np.ascontiguousarray(words, dtype=np.uint32).ravel()
        _check(lib().sim_load(self._h, w.ctypes.data, w.size))


def alloc_rollout(E: int, D: int, H: int, has_value: bool = False, trace: bool = False,
                  device="cuda") -> dict:
    """Device buffers for rollout_collect in the ABI's time-major layouts."""
    import torch
    buf = dict(
        obs=torch.empty((H, D, E), dtype=torch.float32, device=device),
        action=torch.empty((H, E), dtype=torch.uint8, device=device),
        logp=torch.empty((H, E), dtype=torch.float32, device=device),
        reward=torch.empty((H, E), dtype=torch.float32, device=device),
        done=torch.empty((H, E), dtype=torch.uint8, device=device),
    )
    if has_value:
        buf["value"] = torch.empty((H, E), dtype=torch.float32, device=device)
    if trace:
        buf["trace"] = torch.empty((H, TRACE_WIDTH, E), dtype=torch.int64, device=device)
    return buf


def policy_forward_workspace_size(policy: Policy) -> int:
    return lib().policy_forward_workspace_size(C.byref(policy.c))


def policy_forward(policy: Policy, obs, n: int, policy_mode: str, seed: int, step: int,
                   env_base: int = 0, logits=None, value=None, action=None, logp=None,
                   stream=None, workspace=None):
    """policy_forward, or policy_forward_ws when a device workspace (uint8 tensor of
    policy_forward_workspace_size bytes) is given: needed for concurrent streams and for
    CUDA-graph capture."""
    if workspace is None:
        _check(lib().policy_forward(C.byref(policy.c), _ptr(obs), obs.shape[-1], n,
                                    POLICY[policy_mode], seed, step, env_base, _ptr(logits),
                                    _ptr(value), _ptr(action), _ptr(logp), _stream(stream)))
        return
    _check(lib().policy_forward_ws(C.byref(policy.c), _ptr(obs), obs.shape[-1], n,
                                   POLICY[policy_mode], seed, step, env_base, _ptr(logits),
                                   _ptr(value), _ptr(action), _ptr(logp), _ptr(workspace),
                                   workspace.numel() * workspace.element_size(), _stream(stream)))


def compute_returns_gae(rew, done, gamma: float, lam: float, ret, adv=None, val=None,
                        last_val=None, stream=None):
    T, E = rew.shape[0], rew.shape[1]
    _check(lib().compute_returns_gae(_ptr(rew), _ptr(val), _ptr(done), _ptr(last_val), T, E,
                                     rew.shape[1], gamma, lam, _ptr(ret), _ptr(adv),
                                     _stream(stream)))


def returns_baseline_workspace_size(n: int) -> int:
    return lib().returns_baseline_workspace_size(n)


def returns_baseline(x, adv_out, mean_out, workspace, stream=None):
    _check(lib().returns_baseline(_ptr(x), x.numel(), _ptr(adv_out), _ptr(mean_out),
                                  _ptr(workspace), workspace.numel() * workspace.element_size(),
                                  _stream(stream)))


def ppo_loss_grad_workspace_size(policy: Policy, n: int) -> int:
    return lib().ppo_loss_grad_workspace_size(C.byref(policy.c), n)


def ppo_loss_grad(policy: Policy, buf: dict, ret, adv, idx, n: int, algo: str, clip_eps: float,
                  c_value: float, c_entropy: float, grad, stats, workspace, stream=None,
                  precision: str = "fp32"):
    r = Rollout()
    r.ld = buf["action"].shape[-1]
    for k in ("obs", "action", "logp", "value", "reward", "done", "trace"):
        t = buf.get(k)
        setattr(r, k, None if t is None else t.data_ptr())
    p = LossParams(ALGO[algo], clip_eps, c_value, c_entropy, PRECISION[precision])
    _check(lib().ppo_loss_grad(C.byref(policy.c), C.byref(r), r.ld, _ptr(ret), _ptr(adv),
                               _ptr(idx), n, C.byref(p), _ptr(grad), _ptr(stats), _ptr(workspace),
                               workspace.numel() * workspace.element_size(), _stream(stream)))


class AdamParams(C.Structure):
    _fields_ = [("lr", C.c_float), ("beta1", C.c_float), ("beta2", C.c_float),
                ("eps", C.c_float), ("max_grad_norm", C.c_float)]


def adam_workspace_size(n: int) -> int:
    return lib().simx_adam_workspace_size(n)


def adam_step(params, grad, m, v, t, lr: float, beta1: float = 0.9, beta2: float = 0.999,
              eps: float = 1e-8, max_grad_norm: float = 0.0, mask=None, workspace=None,
              stream=None):
    """simx_adam_step on flat fp32 device vectors (mask: uint8 or None).  t: the step
    number (int), or an int64 device tensor of one element that the step increments."""
    p = AdamParams(lr, beta1, beta2, eps, max_grad_norm)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    dev = not isinstance(t, int)
    _check(lib().simx_adam_step(_ptr(params), _ptr(grad), _ptr(m), _ptr(v), _ptr(mask),
                                params.numel(), 0 if dev else t, _ptr(t) if dev else None,
                                C.byref(p), _ptr(workspace), ws_bytes, _stream(stream)))


NOALLOC_SCRATCH_BYTES = 64 << 20


def ppo_loss_grad_noalloc(policy: Policy, buf: dict, ret, adv, idx, n: int, algo: str,
                          clip_eps: float, c_value: float, c_entropy: float, grad, stats,
                          stream=None, precision: str = "fp32"):
    """ppo_loss_grad without a caller workspace: the scratch is a buffer inside the
    library, for callers that cannot allocate device memory (see include/simx.h)."""
    r = Rollout()
    r.ld = buf["action"].shape[-1]
    for k in ("obs", "action", "logp", "value", "reward", "done", "trace"):
        t = buf.get(k)
        setattr(r, k, None if t is None else t.data_ptr())
    p = LossParams(ALGO[algo], clip_eps, c_value, c_entropy, PRECISION[precision])
    _check(lib().ppo_loss_grad_noalloc(C.byref(policy.c), C.byref(r), r.ld, _ptr(ret), _ptr(adv),
                                       _ptr(idx), n, C.byref(p), _ptr(grad), _ptr(stats),
                                       _stream(stream)))


def fma_probe_sink_floats() -> int:
    return lib().simx_fma_probe_sink_floats()


def fma_probe(iters: int, sink, stream=None) -> float:
    """Launch the FP32 FMA-rate probe on the stream; returns the FLOPs it performs."""
    fl = C.c_double(0.0)
    _check(lib().simx_fma_probe(iters, _ptr(sink), C.byref(fl), _stream(stream)))
    return fl.value
