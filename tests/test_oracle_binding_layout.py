"""The oracle's ctypes structs have gcc's size and field offsets on oracle/oracle.h (so the
tests hand the oracle the configuration and policy they mean)."""
import ctypes as C
import os
import shutil
import subprocess

import pytest

from oracle import binding as OB

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
STRUCTS = [("orc_config", OB.OrcConfig), ("orc_mlp", OB.OrcMlp), ("orc_step_out", OB.OrcStepOut)]


def test_oracle_struct_offsets_match_the_c_compiler(tmp_path):
    if shutil.which("gcc") is None:
        pytest.skip("no gcc")
    lines = ["#include <stdio.h>", "#include <stddef.h>", '#include "oracle.h"', "int main(void) {"]
    for name, cls in STRUCTS:
        lines.append('  printf("%s size %%zu\\n", sizeof(%s));' % (name, name))
        for f in cls._fields_:
            lines.append('  printf("%s %s %%zu\\n", offsetof(%s, %s));' % (name, f[0], name, f[0]))
    lines += ["  return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    subprocess.check_call(["gcc", "-std=c11", "-I", os.path.join(ROOT, "oracle"), "-o", str(exe),
                           str(src)])
    got = {}
    for ln in subprocess.check_output([str(exe)]).decode().splitlines():
        s_name, field, val = ln.split()
        got[(s_name, field)] = int(val)
    for name, cls in STRUCTS:
        assert got[(name, "size")] == C.sizeof(cls), name
        for f in cls._fields_:
            assert got[(name, f[0])] == getattr(cls, f[0]).offset, (name, f[0])
