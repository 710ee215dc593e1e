"""The C-ABI library builds, loads and exports every function include/simx.h declares.

Runs without a GPU: loading libsimx.so makes no CUDA call.  Also checks that the
ctypes structs match the header's field lists, that host-only entry points
(simx_obs_dim, simx_state_words, the workspace-size queries, argument validation)
behave, and that the oracle and the library share no source.
"""
import ctypes as C
import os
import re

import pytest

from paper_2607_05272_gb300 import build as B
from paper_2607_05272_gb300 import simx
from paper_2607_05272_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HDR = os.path.join(ROOT, "include", "simx.h")


@pytest.fixture(scope="module")
def lib():
    B.build()
    return simx.lib()


def _declared():
    src = open(HDR).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[\w\*\s]+?\b(\w+)\s*\(", src, flags=re.M)
    return sorted({n for n in names if n not in ("if", "for", "while", "sizeof")})


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert len(names) >= 18
    for n in names:
        assert hasattr(lib, n), n
    assert {s[0] for s in simx.SIGNATURES} == set(names)


def _struct_fields(name):
    src = open(HDR).read()
    body = re.search(r"typedef struct %s \{(.*?)\} %s;" % (name, name), src, flags=re.S).group(1)
    body = re.sub(r"/\*.*?\*/", "", body, flags=re.S)
    out = []
    for decl in body.split(";"):
        decl = decl.strip()
        if not decl:
            continue
        typ, rest = decl.split(None, 1) if not decl.startswith("const") else (decl.rsplit(None, 1)[0], decl.rsplit(None, 1)[1])
        for v in rest.split(","):
            v = v.strip().lstrip("*").strip()
            out.append(v.split("[")[0].strip().lstrip("*"))
    return out


@pytest.mark.parametrize("name,cls", [("simx_config", simx.Config), ("simx_mlp", simx.Mlp),
                                      ("simx_rollout", simx.Rollout),
                                      ("simx_loss_params", simx.LossParams)])
def test_struct_layouts_match_header(name, cls):
    assert _struct_fields(name) == [f[0] for f in cls._fields_]


STRUCTS = [("simx_config", simx.Config), ("simx_mlp", simx.Mlp), ("simx_rollout", simx.Rollout),
           ("simx_loss_params", simx.LossParams), ("simx_counters", simx.Counters),
           ("simx_adam_params", simx.AdamParams)]


def test_struct_offsets_match_the_c_compiler(tmp_path):
    """Every ctypes struct of the binding has the C compiler's size and field offsets
    (gcc on include/simx.h), so no field drifts between the header and the binding."""
    import shutil
    import subprocess
    if shutil.which("gcc") is None:
        pytest.skip("no gcc")
    lines = ["#include <stdio.h>", "#include <stddef.h>", '#include "simx.h"', "int main(void) {"]
    for name, cls in STRUCTS:
        lines.append('  printf("%s size %%zu\\n", sizeof(%s));' % (name, name))
        for f in cls._fields_:
            lines.append('  printf("%s %s %%zu\\n", offsetof(%s, %s));' % (name, f[0], name, f[0]))
    lines += ["  return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    subprocess.check_call(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), "-o", str(exe),
                           str(src)])
    got = {}
    for ln in subprocess.check_output([str(exe)]).decode().splitlines():
        s_name, field, val = ln.split()
        got[(s_name, field)] = int(val)
    for name, cls in STRUCTS:
        assert got[(name, "size")] == C.sizeof(cls), name
        for f in cls._fields_:
            assert got[(name, f[0])] == getattr(cls, f[0]).offset, (name, f[0])


def test_host_entry_points(lib):
    for name in ("c1", "c2", "c3", "c4", "c5"):
        cfg = W.CONFIGS[name](16)
        assert simx.obs_dim(cfg) == cfg["obs_dim"]
        K, T, cap = cfg["n_servers"], cfg["n_types"], cfg["queue_cap"]
        words = 32 + 2 * K + K * T + K * T * cap + (K * cap if cfg["cost_type"] >= 0 else 0)
        assert simx.state_words(cfg) == words
    assert lib.returns_baseline_workspace_size(1000) >= 8
    assert lib.simx_strerror(1) == b"invalid argument"


def test_invalid_config_rejected_before_any_device_call(lib):
    bad = W.c1(4)
    bad["queue_cap"] = 100  # not a power of two
    h = C.c_void_p()
    st = lib.sim_create(C.byref(simx.make_config(bad)), 0, C.byref(h))
    assert st == simx.EINVAL and not h.value
    assert b"power of two" in lib.simx_last_error()
    bad = W.c3(4)
    bad["obs_dim"] = 12
    st = lib.sim_create(C.byref(simx.make_config(bad)), 0, C.byref(h))
    assert st == simx.EINVAL and b"obs_dim" in lib.simx_last_error()


def test_oracle_shares_no_source_with_the_library():
    lib_files = []
    for d, _, fs in os.walk(os.path.join(ROOT, "paper_2607_05272_gb300")):
        lib_files += [os.path.join(d, f) for f in fs if f.endswith((".py", ".cu", ".cuh", ".h"))]
    for f in lib_files:
        txt = open(f).read()
        assert "import oracle" not in txt and "from oracle" not in txt, f
        assert "oracle.h" not in txt, f
    for f in os.listdir(os.path.join(ROOT, "oracle")):
        if f.endswith((".py", ".c", ".h")):
            txt = open(os.path.join(ROOT, "oracle", f)).read()
            assert "paper_2607_05272_gb300" not in txt, f
            assert "simx.h" not in txt and "csrc" not in txt, f
