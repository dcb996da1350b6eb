"""The C ABI from C: a plain C99 program (tests/c_client/plan_only.c) that
includes only include/topas_attn.h is compiled with gcc, linked against the
library and run on a plan-only context (no GPU, no CUDA call).  It checks
the budget of Eq. 2, lifecycle errors, append, a planned decode step,
eviction and reload, truncation and close, and prints "ok"."""
import os
import shutil
import subprocess

import pytest

from paper_2608_25523_gb300.build import build

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


def test_plain_c_client(tmp_path):
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    lib = build()
    exe = tmp_path / "plan_only"
    libdir = os.path.dirname(lib)
    libname = os.path.basename(lib)
    assert libname.startswith("lib") and libname.endswith(".so")
    cmd = [gcc, "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic",
           "-I", os.path.join(ROOT, "include"), os.path.join(HERE, "c_client", "plan_only.c"),
           "-L", libdir, "-l:" + libname, "-Wl,-rpath," + libdir, "-o", str(exe)]
    subprocess.run(cmd, check=True, capture_output=True, text=True)
    res = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert res.returncode == 0, res.stdout + res.stderr
    assert res.stdout.strip().splitlines()[-1] == "ok", res.stdout
