"""The C ABI from plain C: examples/kv_roundtrip.c (a paged KV range through
pinned host chunks and back) and examples/kv_tier_flow.c (two replicas through
the shared tier: store and commit, prefix lookup, bounded wait, acquire on the
reader's stream, restore, release) compile against include/kvxfer.h with gcc
on any machine, and on a GPU run without Python or PyTorch."""
import os
import subprocess

import pytest

from paper_2609_15021_gb300 import _build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CUDA_LIB = "/usr/local/cuda/lib64"


def _compile(out, source="kv_roundtrip.c"):
    lib = os.path.dirname(_build.build())
    cmd = ["gcc", "-O2", "-std=c11", "-Wall", "-I", os.path.join(ROOT, "include"), "-I", "/usr/local/cuda/include",
           os.path.join(ROOT, "examples", source), "-o", out, "-L", lib, "-lkvxfer", "-L", CUDA_LIB,
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


def test_c_tier_example_compiles(tmp_path):
    _compile(str(tmp_path / "kv_tier_flow"), "kv_tier_flow.c")


@pytest.mark.gpu
def test_c_tier_example_runs(tmp_path):
    exe = _compile(str(tmp_path / "kv_tier_flow"), "kv_tier_flow.c")
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "tier flow ok" in r.stdout
