"""ctypes binding of the C oracle (test infrastructure only)."""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_HDR = os.path.join(_HERE, "oracle.h")
_SO = os.path.join(_HERE, "_build", "liboracle.so")
MAX_LAYERS = 6  # ORC_MAX_LAYERS
_lock = threading.Lock()
_lib = None

# Compiled exactly as the IEEE-754 reference needs: no contraction, no fast-math.
CFLAGS = ["-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
          "-Wall", "-Wextra"]


def build(force: bool = False) -> str:
    """Compile oracle.c into _build/liboracle.so (gcc) if missing or stale."""
    os.makedirs(os.path.dirname(_SO), exist_ok=True)
    stale = (not os.path.exists(_SO) or
             max(os.path.getmtime(_SRC), os.path.getmtime(_HDR)) > os.path.getmtime(_SO))
    if force or stale:
        tmp = _SO + ".tmp%d" % os.getpid()
        subprocess.check_call(["gcc", *CFLAGS, "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _SO)
    return _SO


class OrcConfig(C.Structure):
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
        ("trace_gap", C.c_void_p), ("trace_type", C.c_void_p), ("trace_cost", C.c_void_p),
        ("trace_len", C.c_uint32),
    ]

_TRACE_FIELDS = ("trace_gap", "trace_type", "trace_cost", "trace_len")


class OrcMlp(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("dims", C.c_int32 * (MAX_LAYERS + 1)),
                ("W", C.c_void_p * MAX_LAYERS), ("b", C.c_void_p * MAX_LAYERS),
                ("has_value", C.c_int32), ("act", C.c_int32 * MAX_LAYERS),
                ("grid", C.c_int32), ("gx", C.c_int32 * MAX_LAYERS)]


class OrcStepOut(C.Structure):
    _fields_ = [("obs", C.c_void_p), ("logits", C.c_void_p), ("action", C.c_int32),
                ("logp", C.c_float), ("value", C.c_float), ("reward", C.c_float),
                ("done", C.c_uint8), ("trace", C.c_int64 * 4)]


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = C.CDLL(build())
            P, U32, U64, F, I32, I64 = C.c_void_p, C.c_uint32, C.c_uint64, C.c_float, C.c_int32, C.c_int64
            L.orc_philox4x32_10.argtypes = [P, P, P]
            for nm in ("orc_detlog", "orc_detexp", "orc_dettanh", "orc_detcos2pi"):
                getattr(L, nm).argtypes = [F]
                getattr(L, nm).restype = F
            L.orc_normal.argtypes = [U32, U32]
            L.orc_normal.restype = F
            L.orc_duration.argtypes = [F]
            L.orc_duration.restype = U32
            L.orc_obs_dim.argtypes = [P]
            L.orc_obs_dim.restype = U32
            L.orc_state_words.argtypes = [P]
            L.orc_state_words.restype = U64
            L.orc_env_new.argtypes = [P, U32, U64]
            L.orc_env_new.restype = P
            L.orc_env_free.argtypes = [P]
            L.orc_env_reset.argtypes = [P]
            L.orc_env_observe.argtypes = [P, P]
            L.orc_env_step.argtypes = [P, P, C.c_int, I32, P]
            L.orc_env_export.argtypes = [P, P]
            L.orc_env_import.argtypes = [P, P]
            L.orc_env_status.argtypes = [P]
            L.orc_env_status.restype = U32
            L.orc_env_little.argtypes = [P, U32, P, P]
            L.orc_env_switch_log.argtypes = [P, P, U32]
            L.orc_env_switch_log_count.argtypes = [P]
            L.orc_env_switch_log_count.restype = U32
            L.orc_policy.argtypes = [P, P, C.c_int, U64, U32, U32, P, P, P, P]
            L.orc_rollout.argtypes = [P, P, U64, C.c_int, P, I64, I32, P, P, P, P, P, P, P, P]
            L.orc_rollout.restype = C.c_int
            L.orc_map.argtypes = [C.c_int, P, P, I64]
            L.orc_philox_n.argtypes = [U32, U32, U32, U64, I64, P]
            L.orc_samplers.argtypes = [P, C.c_int, F, P, I64, P]
            L.orc_gridq_n.argtypes = [P, I64, I32, P]
            _lib = L
    return _lib


def make_config(cfg: dict) -> OrcConfig:
    """cfg: the library's configuration fields, plus for trace replay ``trace`` =
    (gap_us, type or None, cost_us or None) arrays, kept alive by the returned struct."""
    c = OrcConfig()
    tr = cfg.get("trace")
    if tr is not None:
        gap = np.ascontiguousarray(tr[0], dtype=np.uint32)
        typ = None if tr[1] is None else np.ascontiguousarray(tr[1], dtype=np.uint8)
        cst = None if tr[2] is None else np.ascontiguousarray(tr[2], dtype=np.uint32)
        c._keep = (gap, typ, cst)
        c.trace_gap = gap.ctypes.data
        c.trace_type = None if typ is None else typ.ctypes.data
        c.trace_cost = None if cst is None else cst.ctypes.data
        c.trace_len = len(gap)
    for name, _ in OrcConfig._fields_:
        if name in _TRACE_FIELDS:
            continue
        v = cfg[name]
        if isinstance(v, (list, tuple)):
            arr = getattr(c, name)
            for i, x in enumerate(v):
                arr[i] = x
        else:
            setattr(c, name, v)
    return c


class _Mlp:
    """Keeps the numpy weight arrays alive while the C struct points at them."""

    def __init__(self, Ws, bs, has_value, acts=None, grid=None):
        self.Ws = [np.ascontiguousarray(w, dtype=np.float32) for w in Ws]
        self.bs = [np.ascontiguousarray(b, dtype=np.float32) for b in bs]
        m = OrcMlp()
        m.n_layers = len(self.Ws)
        m.dims[0] = self.Ws[0].shape[1]
        for l, w in enumerate(self.Ws):
            m.dims[l + 1] = w.shape[0]
            m.W[l] = w.ctypes.data
            m.b[l] = self.bs[l].ctypes.data
        m.has_value = int(bool(has_value))
        for l, a in enumerate(acts or []):
            m.act[l] = {"tanh": 0, "identity": 1, "gelu": 2}.get(a, a)
        if grid is not None:          # the input grid exponent of every layer
            m.grid = 1
            for l, e in enumerate(grid):
                m.gx[l] = int(e)
        self.c = m


def _mlp(mlp):
    if mlp is None:
        return None, None
    Ws, bs, hv = mlp[:3]
    m = _Mlp(Ws, bs, hv, mlp[3] if len(mlp) > 3 else None, mlp[4] if len(mlp) > 4 else None)
    return m, C.byref(m.c)


def _u32(x: int) -> int:
    return x & 0xFFFFFFFF


def philox(ctr, key) -> np.ndarray:
    c = np.asarray([_u32(v) for v in ctr], dtype=np.uint32)
    k = np.asarray([_u32(v) for v in key], dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib().orc_philox4x32_10(c.ctypes.data, k.ctypes.data, out.ctypes.data)
    return out


def map_fn(fn: str, x) -> np.ndarray:
    """Apply detlog / detexp / dettanh / detcos2pi / detgelu to an fp32 array."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    y = np.empty_like(x)
    code = {"log": 0, "exp": 1, "tanh": 2, "cos2pi": 3, "gelu": 4}[fn]
    lib().orc_map(code, x.ctypes.data, y.ctypes.data, x.size)
    return y


def philox_n(idx0: int, env: int, stream: int, seed: int, n: int) -> np.ndarray:
    """Philox blocks [n][4] for counters (idx0 + i, env, stream, 0)."""
    out = np.empty((n, 4), np.uint32)
    lib().orc_philox_n(_u32(idx0), _u32(env), _u32(stream), seed, n, out.ctypes.data)
    return out


def samplers(cfg: dict, kind: int, words, scale: float = 1.0) -> np.ndarray:
    """The simulator's samplers applied to Philox blocks (see orc_samplers)."""
    c = make_config(cfg)
    w = np.ascontiguousarray(words, dtype=np.uint32)
    out = np.empty(w.shape[0], np.float32)
    lib().orc_samplers(C.byref(c), kind, scale, w.ctypes.data, w.shape[0], out.ctypes.data)
    return out


def gridq(v, e: int) -> np.ndarray:
    """The grid policy's rounding Q(v, e) = clamp(rint(v 2^e), -255, 255) 2^-e (fp32)."""
    v = np.ascontiguousarray(v, dtype=np.float32)
    out = np.empty_like(v)
    lib().orc_gridq_n(v.ctypes.data, v.size, int(e), out.ctypes.data)
    return out


def detlog(x: float) -> float:
    return lib().orc_detlog(x)


def detexp(x: float) -> float:
    return lib().orc_detexp(x)


def dettanh(x: float) -> float:
    return lib().orc_dettanh(x)


def detcos2pi(x: float) -> float:
    return lib().orc_detcos2pi(x)


def normal(w0: int, w1: int) -> float:
    return lib().orc_normal(_u32(w0), _u32(w1))


def duration(x: float) -> int:
    return lib().orc_duration(x)


def obs_dim(cfg: dict) -> int:
    c = make_config(cfg)
    return lib().orc_obs_dim(C.byref(c))


def state_words(cfg: dict) -> int:
    c = make_config(cfg)
    return lib().orc_state_words(C.byref(c))


def policy(mlp, obs, mode: int, seed: int, step: int, env_id: int):
    """One policy evaluation: (logits, value, action, logp)."""
    m, mp = _mlp(mlp)
    obs = np.ascontiguousarray(obs, dtype=np.float32)
    A = m.Ws[-1].shape[0] - (1 if mlp[2] else 0)
    logits = np.zeros(A, dtype=np.float32)
    value = C.c_float()
    action = C.c_int32()
    logp = C.c_float()
    lib().orc_policy(mp, obs.ctypes.data, mode, seed, _u32(step), _u32(env_id), logits.ctypes.data,
                     C.byref(value), C.byref(action), C.byref(logp))
    return logits, value.value, action.value, logp.value


def rollout(cfg: dict, mlp, seed: int, mode: int, env_ids, H: int) -> dict:
    """Reset the given envs and run H steps each; arrays in the library's layouts."""
    c = make_config(cfg)
    m, mp = _mlp(mlp)
    ids = np.ascontiguousarray(env_ids, dtype=np.uint32)
    n = len(ids)
    D = lib().orc_obs_dim(C.byref(c))
    SW = lib().orc_state_words(C.byref(c))
    out = dict(
        obs=np.zeros((H, D, n), np.float32), action=np.zeros((H, n), np.int32),
        logp=np.zeros((H, n), np.float32), value=np.zeros((H, n), np.float32),
        reward=np.zeros((H, n), np.float32), done=np.zeros((H, n), np.uint8),
        trace=np.zeros((H, 4, n), np.int64), state=np.zeros((n, SW), np.uint32),
    )
    rc = lib().orc_rollout(C.byref(c), mp, seed, mode, ids.ctypes.data, n, H,
                           *[out[k].ctypes.data for k in
                             ("obs", "action", "logp", "value", "reward", "done", "trace", "state")])
    if rc != 0:
        raise MemoryError("oracle rollout allocation failed")
    return out


class OracleEnv:
    """One oracle environment, stepped explicitly."""

    def __init__(self, cfg: dict, env_id: int, seed: int):
        self.cfg = cfg
        self._c = make_config(cfg)
        self.D = lib().orc_obs_dim(C.byref(self._c))
        self.SW = lib().orc_state_words(C.byref(self._c))
        self.A = (cfg["n_types"] if cfg["mode"] == 0 else cfg["n_servers"]) * cfg["n_bsizes"]
        self._e = lib().orc_env_new(C.byref(self._c), _u32(env_id), seed)
        if not self._e:
            raise MemoryError("orc_env_new failed")

    def __del__(self):
        e = getattr(self, "_e", None)
        if e:
            lib().orc_env_free(e)
            self._e = None

    def reset(self):
        lib().orc_env_reset(self._e)

    def observe(self) -> np.ndarray:
        o = np.zeros(self.D, np.float32)
        lib().orc_env_observe(self._e, o.ctypes.data)
        return o

    def step(self, mode: int, mlp=None, action: int = 0) -> dict:
        m, mp = _mlp(mlp)
        obs = np.zeros(self.D, np.float32)
        logits = np.zeros(max(self.A, 1), np.float32)
        o = OrcStepOut()
        o.obs = obs.ctypes.data
        o.logits = logits.ctypes.data
        lib().orc_env_step(self._e, mp, mode, int(action), C.byref(o))
        return dict(obs=obs, logits=logits, action=o.action, logp=o.logp, value=o.value,
                    reward=o.reward, done=o.done, trace=list(o.trace))

    def export(self) -> np.ndarray:
        w = np.zeros(self.SW, np.uint32)
        lib().orc_env_export(self._e, w.ctypes.data)
        return w

    def load(self, words) -> None:
        w = np.ascontiguousarray(words, dtype=np.uint32)
        assert w.size == self.SW
        lib().orc_env_import(self._e, w.ctypes.data)

    def status(self) -> int:
        return lib().orc_env_status(self._e)

    def attach_switch_log(self, cap: int) -> None:
        """Record the modulating chain from the next reset on: (time, state) at time 0
        and at every switch processed, up to cap pairs (see switch_log)."""
        self._swlog = np.zeros((cap, 2), np.uint32)
        lib().orc_env_switch_log(self._e, self._swlog.ctypes.data, cap)

    def switch_log(self) -> np.ndarray:
        n = lib().orc_env_switch_log_count(self._e)
        return self._swlog[:n].copy()

    def little(self, t_end: int):
        a = C.c_uint64()
        w = C.c_uint64()
        lib().orc_env_little(self._e, _u32(t_end), C.byref(a), C.byref(w))
        return a.value, w.value
