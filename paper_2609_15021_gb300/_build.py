"""Build libkvxfer.so (the transfer library) and libkvxfer_probe.so (the
measuring probes the tests and the benchmark use) in-tree with nvcc for
sm_103a (no cmake, no torch)."""
from __future__ import annotations

import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "_lib", "libkvxfer.so")
PROBE_LIB = os.path.join(PKG, "_lib", "libkvxfer_probe.so")

SOURCES = ["pack_kernels.cu", "segment_kernels.cu", "tma_kernels.cu", "kvxfer.cu", "no_alloc.cu", "tier.cpp",
           "tier_kernels.cu", "host_alloc.cpp", "host_touch.cpp"]
PROBE_SOURCES = ["probe.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-O2,-Wall,-Wextra", f"-I{INCLUDE}"]


def _nvcc() -> str:
    for cand in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", "nvcc"):
        if cand and (os.path.isabs(cand) and os.path.exists(cand) or cand == "nvcc"):
            return cand
    return "nvcc"


def _inputs(sources) -> list[str]:
    deps = [os.path.join(CSRC, s) for s in sources]
    deps += [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".h", ".cuh"))]
    deps += [os.path.join(INCLUDE, f) for f in os.listdir(INCLUDE) if f.endswith(".h")]
    deps.append(os.path.abspath(__file__))
    return deps


def _fresh(lib, sources) -> bool:
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(d) <= t for d in _inputs(sources))


def up_to_date() -> bool:
    return _fresh(LIB, SOURCES) and _fresh(PROBE_LIB, PROBE_SOURCES)


def build(force: bool = False, verbose: bool = False, ptxas_report: str | None = None) -> str:
    """Compile every CUDA source in parallel and link both shared libraries;
    returns the path of libkvxfer.so."""
    if not force and up_to_date():
        return LIB
    todo = [(lib, srcs) for lib, srcs in ((LIB, SOURCES), (PROBE_LIB, PROBE_SOURCES))
            if force or not _fresh(lib, srcs)]
    os.makedirs(BUILD, exist_ok=True)
    os.makedirs(os.path.dirname(LIB), exist_ok=True)
    nvcc = _nvcc()
    extra = ["-Xptxas", "-v"] if ptxas_report else []

    def compile_one(src: str):
        obj = os.path.join(BUILD, os.path.splitext(src)[0] + ".o")
        cmd = [nvcc, *ARCH, *FLAGS, *extra, "-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        return obj, r.stderr

    all_sources = [s for _, srcs in todo for s in srcs]
    with ThreadPoolExecutor(max_workers=len(all_sources)) as ex:
        results = dict(zip(all_sources, ex.map(compile_one, all_sources)))
    if ptxas_report:
        with open(ptxas_report, "w") as f:
            for _, log in results.values():
                f.write(log)
    for lib, srcs in todo:
        tmp = lib + f".tmp{os.getpid()}"
        cmd = [nvcc, *ARCH, "-shared", "-o", tmp, *[results[s][0] for s in srcs]]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, lib)
        if verbose:
            print(f"built {lib}", file=sys.stderr)
    return LIB


if __name__ == "__main__":
    build(force="--force" in sys.argv, verbose=True,
          ptxas_report=next((a.split("=", 1)[1] for a in sys.argv if a.startswith("--ptxas=")), None))
