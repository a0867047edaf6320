"""The C ABI from plain C (examples/kv_roundtrip.c): it compiles against
include/kvxfer.h with gcc on any machine, and on a GPU it round-trips a paged
KV range through pinned host chunks without Python or PyTorch."""
import os
import subprocess

import pytest

from paper_2609_15021_gb300 import _build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CUDA_LIB = "/usr/local/cuda/lib64"


def _compile(out):
    lib = os.path.dirname(_build.build())
    cmd = ["gcc", "-O2", "-std=c11", "-I", os.path.join(ROOT, "include"), "-I", "/usr/local/cuda/include",
           os.path.join(ROOT, "examples", "kv_roundtrip.c"), "-o", out, "-L", lib, "-lkvxfer", "-L", CUDA_LIB,
           "-lcudart", f"-Wl,-rpath,{lib}", f"-Wl,-rpath,{CUDA_LIB}"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    return out


def test_c_example_compiles(tmp_path):
    _compile(str(tmp_path / "kv_roundtrip"))


@pytest.mark.gpu
def test_c_example_runs(tmp_path):
    exe = _compile(str(tmp_path / "kv_roundtrip"))
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "roundtrip ok" in r.stdout
