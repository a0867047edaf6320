#!/usr/bin/env python
"""Paged-KV store / restore throughput on GB300 through libkvxfer.

One step = the whole transfer path on a 27B-class KV cache (62 layers, 8 KV
heads, head_dim 128, bf16, 16-token pages, 256-token chunks): kv_store of the
full context from a paged pool into pinned host chunks (pack + device->host),
then kv_load of every chunk into freshly listed pages of a second pool
(host->device + unpack).  Before every step, outside its timed region, the
second pool is refilled with poison bytes, so each restore writes into a cold
pool (the refill, a write of the whole pool, also flushes L2).  The default
workload is the 128k-token context (8,192 of 10,240 pages, 33,285,996,544
bytes per direction); --config picks another.

value  = bytes moved over the host link (both directions) / device time of
         the K timed steps (CUDA events on the caller's stream), GB/s.
e2e    = the same metric timed on the host clock around the public API calls,
         including per-step block-table uploads from pinned memory and the
         host synchronisation that must precede host use of the chunks (the
         chunk set is described once, as a kvxfer.ChunkList).
After the timed region (none of it is in `value`):
roofline             the dominant kernel against the host link's ceiling: the
                     larger of the copy engines' pinned cudaMemcpyAsync peak and
                     a plain SM streaming copy to / from the same mapped pinned
                     pool, both measured in the same run;
hbm_roofline         kv_pack / kv_unpack of the same context into device chunks
                     against the measured HBM copy peak;
concurrent_replicas  one context stored while another context's chunks are
                     restored, each through its own context and stream, over
                     >= 10 repetitions; in every repetition the copy engines'
                     and the SMs' bidirectional rates over the same two chunk
                     sets are timed right after the replicas;
restore_after_idle   a restore after the pool sat untouched for a few seconds,
                     with the library's host-page touch and without it;
tier_path            the same store and restore through a host tier shared
                     across processes: keyed reserve / commit, prefix lookup,
                     acquire / release, one kv_store and one kv_load per step;
streamed_cross_replica  replica B restores, group by group, what replica A is
                     storing through a shared tier, each group as soon as it is
                     committed (time from A's first store to B's last restore);
cpu_baseline         the oracle on the host cores over a sample of the chunks,
                     which also checks those GPU chunks byte for byte;
configs              the other workloads (32k and 256k tokens, the paper's FP8
                     shape at 127,008 tokens, the hybrid six-turn session),
                     each timed the same way in the same run.
With --gpus N > 1 (torchrun, one rank per GPU) the replicas share ONE pinned
host tier (POSIX shared memory), as the paper's replicas share one host pool:
each step, rank r stores its context into the tier and restores rank r-1's
context from it (in rounds when the tier cannot hold every context at once).
Prints one JSON line.  --impl reference times the CPU oracle instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "KV store/load GB/s vs host-link & HBM peak; 128k-token context restore ms"
# 27B-class attention KV of the benchmark configurations
SHAPE_27B = dict(L=62, H=8, D=128, e=2, B=16, C=256, name="27B-class paged KV (62 layers x 8 KV heads x "
                 "head_dim 128, bf16, 16-token pages)", dtype="bf16")
# the paper's own attention KV (Table 1, Sec. 3.1): 16 full-attention layers x 4 KV heads x
# head_dim 256 in FP8, 32-token kernel pages, 1,568-token chunks of 49 pages
SHAPE_PAPER = dict(L=16, H=4, D=256, e=1, B=32, C=1568, name="the paper's FP8 attention KV (16 layers x 4 KV "
                   "heads x head_dim 256, 1 byte, 32-token pages)", dtype="fp8 bytes")
CONFIGS = {
    "2k": dict(tokens=2048, pool_blocks=256, shape=SHAPE_27B),  # profiling size: 2 x 1 GB pools
    "32k": dict(tokens=32768, pool_blocks=4096, shape=SHAPE_27B),
    "128k": dict(tokens=131072, pool_blocks=10240, shape=SHAPE_27B),
    "256k": dict(tokens=262144, pool_blocks=20480, shape=SHAPE_27B),
    # the paper's 128k cross-replica hit: 127,008 tokens = 81 chunks (Sec. 3.2)
    "paper127k": dict(tokens=127008, pool_blocks=16384, shape=SHAPE_PAPER),
}
FALLBACK_HBM_GBS = 6800.0
GB = 1e9


def workload_name(cfg, layout="hnd"):
    t, n, s = cfg["tokens"], cfg["pool_blocks"], cfg["shape"]
    pages = "pages" if layout == "hnd" else "NHD pages ([K|V][token][head][row])"
    return (f"{s['name']}, {t}-token context = {t // s['B']} of {n} {pages} by seeded permutation, "
            f"{s['C']}-token chunks: full store to pinned host chunks, then restore into a cold pool "
            f"(poisoned before every step, outside the timed region)")


def bytes_per_direction(cfg):
    s = cfg["shape"]
    return cfg["tokens"] * s["L"] * 2 * s["H"] * s["D"] * s["e"]


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured (MEASURED_PEAKS.json hbm_gbs, burst copy)"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback (6.8 TB/s, no MEASURED_PEAKS.json)"


def kernel_source_hash(source="pack_kernels.cu"):
    """sha256 prefix of a kernel source file and the device headers (.cuh) it includes."""
    csrc = os.path.join(ROOT, "paper_2609_15021_gb300", "csrc")
    with open(os.path.join(csrc, source), "rb") as f:
        text = f.read()
    h = hashlib.sha256(text)
    for inc in re.findall(rb'#include "([^"]+\.cuh)"', text):
        with open(os.path.join(csrc, inc.decode()), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def shape_key(s, layout="hnd"):
    key = f"L{s['L']} H{s['H']} D{s['D']} e{s['e']} B{s['B']} C{s['C']}"
    return key if layout == "hnd" else key + " NHD"


class Traffic:
    """DRAM bytes per launch from a committed ncu capture of this kernel source and
    shape, scaled to a launch of a given size by its algorithmic bytes (the capture
    is taken on a smaller launch of the same kernel)."""

    def __init__(self, record):
        self.captured = record["captured"] if record else {}

    def get(self, name, alg_bytes):
        if name not in self.captured:
            return None
        traffic, captured_alg = self.captured[name]
        return traffic * alg_bytes / captured_alg


def recorded_traffic(shape, source="pack_kernels.cu", layout="hnd"):
    """Traffic record from profiles/ for this kernel source file (as it is now)
    and KV shape; a record with no entries if none matches."""
    pdir = os.path.join(ROOT, "profiles")
    want = kernel_source_hash(source)
    if not os.path.isdir(pdir):
        return None
    for name in sorted(os.listdir(pdir)):
        if not name.endswith((".md", ".txt")):
            continue
        with open(os.path.join(pdir, name)) as f:
            for line in f:
                m = re.match(r"\s*bench-traffic:\s*(\{.*\})\s*$", line)
                if m:
                    d = json.loads(m.group(1))
                    if (d.get("kernel_sha256") == want and d.get("source", "pack_kernels.cu") == source
                            and d.get("shape") == shape_key(shape, layout)):
                        return Traffic(d)
    return Traffic(None)


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms while running."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(prefix="clocks_", suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if self.proc is None or not self.path:
            return None
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", choices=list(CONFIGS), default="128k")
    ap.add_argument("--mode", choices=["auto", "staged", "zerocopy"], default="auto")
    ap.add_argument("--slot-mib", type=int, default=0, help="staging slot size (0 = library default)")
    ap.add_argument("--cpu-sample-chunks", type=int, default=32)
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-hbm-roofline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--host-alloc", choices=["auto", "plain", "numa", "driver", "huge"], default="auto",
                    help="pinned pool from kv_host_alloc (plain: the driver's allocator), from "
                         "kv_host_alloc_numa on the host NUMA node nearest the GPU, from the driver's allocator "
                         "stated (KVX_HOST_DRIVER), or on huge pages (KVX_HOST_HUGE); auto: huge for "
                         "--mode staged (the copy engines want huge pages), else plain")
    ap.add_argument("--no-cold", action="store_true",
                    help="skip the leg that restores after the pool sat untouched (--cold-idle-s seconds)")
    ap.add_argument("--cold-idle-s", type=float, default=10.0)
    ap.add_argument("--no-tier", action="store_true",
                    help="skip the leg that stores and restores chunk by chunk through the host tier")
    ap.add_argument("--no-concurrent", action="store_true",
                    help="skip the two-replica leg (one stores while the other restores)")
    ap.add_argument("--device-engine", choices=["lsu", "tma"], default="tma",
                    help="kernel of the device-side (HBM) pack/unpack leg")
    ap.add_argument("--layout", choices=["hnd", "nhd"], default="hnd",
                    help="page layout of the headline workload's pools (HND: [K|V][head][token][row], the "
                         "paper's; NHD: [K|V][token][head][row])")
    ap.add_argument("--configs", default="32k,256k,paper127k,hybrid",
                    help="other workloads timed after the headline one in the same run (comma list of "
                         f"{sorted(set(CONFIGS) - {'2k'}) + ['hybrid']}, or 'none'); N=1 only")
    ap.add_argument("--config-steps", type=int, default=4)
    ap.add_argument("--concurrent-reps", type=int, default=12)
    ap.add_argument("--shared-tier", action="store_true",
                    help="run the replicas through one shared pinned tier (the default when N > 1)")
    ap.add_argument("--tier-budget-gib", type=float, default=256.0,
                    help="most pinned host memory the shared tier of N > 1 replicas may take (the paper's "
                         "pool is 256 GiB); also bounded by the host's available memory")
    return ap.parse_args()


def dist_init(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(world, value: float, local: int) -> float:
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    # NCCL reduces device tensors, gloo host tensors
    on_gpu = dist.get_backend() == "nccl"
    t = torch.tensor([value], dtype=torch.float64, device=f"cuda:{local}" if on_gpu else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ------------------------------------------------------------------ CPU oracle legs


def oracle_sample(cfg, n_chunks_sample, pool_pages_np=None, layout="hnd"):
    """Mini-workload for the oracle: n_chunks_sample full chunks whose pages are given
    (or random), as a pool of exactly those pages under an identity table."""
    import numpy as np

    import oracle
    from paper_2609_15021_gb300 import synth
    s = cfg["shape"]
    bpc = s["C"] // s["B"]
    spec = oracle.PoolSpec(s["L"], n_chunks_sample * bpc, s["B"], s["H"], s["D"], s["e"],
                           oracle.NHD if layout == "nhd" else oracle.HND)
    if pool_pages_np is None:
        pool_pages_np = [synth.random_bytes(spec.layer_bytes, 100 + l) for l in range(s["L"])]
    ident = np.arange(n_chunks_sample * bpc, dtype=np.int32)
    return spec, pool_pages_np, ident


def time_oracle(spec, layers, ident, n_chunks_sample, min_seconds, threads, C):
    """Store then load of the sample, repeated until min_seconds have passed."""
    import numpy as np

    import oracle
    orc = oracle.c_oracle()
    t1 = n_chunks_sample * C
    cb = orc.chunk_bytes(spec, C)
    chunks = [np.empty(cb, np.uint8) for _ in range(n_chunks_sample)]
    dest = [np.empty_like(l) for l in layers]
    reps, t_start = 0, time.perf_counter()
    while True:
        rc, _ = orc.store(spec, layers, ident, 0, t1, C, chunks, n_threads=threads)
        assert rc == 0
        rc, _ = orc.load(spec, dest, ident, 0, t1, C, chunks, n_threads=threads)
        assert rc == 0
        reps += 1
        el = time.perf_counter() - t_start
        if el >= min_seconds:
            break
    return reps, el, chunks, 2 * cb * n_chunks_sample


def run_reference(args):
    world, rank, local = int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")), 0
    if rank != 0:
        return 0
    import oracle
    oracle.build()
    cfg = CONFIGS[args.config]
    threads = os.cpu_count() or 1
    S = args.cpu_sample_chunks
    spec, layers, ident = oracle_sample(cfg, S, layout=args.layout)
    step_times = []
    moved = None
    for i in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        reps, el, _, moved = time_oracle(spec, layers, ident, S, 0.0, threads, cfg["shape"]["C"])
        if i >= args.warmup:
            step_times.append(time.perf_counter() - t0)
    total = sum(step_times)
    value = moved * len(step_times) / total / GB
    sample = (f"{S} of {cfg['tokens'] // cfg['shape']['C']} chunks of the workload per step "
              f"({moved // 2} bytes per direction), store then load, {threads} threads")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / len(step_times),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u8",
        "data": "synthetic random bytes in the workload's shape",
        "config": {"workload": workload_name(cfg, args.layout), "context_tokens": cfg["tokens"],
                   "page_layout": args.layout.upper()},
        "cpu_baseline": {"value": value, "unit": "GB/s", "cores": min(threads, S), "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------ GPU leg


def shm_free_bytes() -> int:
    """Room left in the POSIX shared-memory file system (0 if unknown)."""
    try:
        st = os.statvfs("/dev/shm")
        return st.f_bavail * st.f_frsize
    except OSError:
        return 0


def link_buffers(torch, dev):
    """The pinned and device buffers of host_link_peak, allocated once per run."""
    n = 1 << 30
    return {"h": torch.empty(n, dtype=torch.uint8, pin_memory=True), "d": torch.empty(n, dtype=torch.uint8, device=dev),
            "h2": torch.empty(n, dtype=torch.uint8, pin_memory=True),
            "d2": torch.empty(n, dtype=torch.uint8, device=dev)}


def host_link_peak(torch, dev, bufs):
    """Best-of-5 pinned cudaMemcpyAsync of 1 GiB per direction, GB/s."""
    h, d, h2, d2 = bufs["h"], bufs["d"], bufs["h2"], bufs["d2"]
    n = h.numel()
    out = {}
    for name, dst, src in (("d2h", h, d), ("h2d", d, h)):
        best = None
        for i in range(7):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            dst.copy_(src, non_blocking=True)
            b.record()
            b.synchronize()
            if i >= 2:
                ms = a.elapsed_time(b)
                best = ms if best is None else min(best, ms)
        out[name] = n / (best * 1e-3) / GB
    # both directions at once, one copy per stream (two replicas sharing the link)
    s1, s2 = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    best = None
    for i in range(7):
        a, b1, b2 = (torch.cuda.Event(enable_timing=True) for _ in range(3))
        torch.cuda.synchronize()
        a.record(s1)
        s2.wait_event(a)
        with torch.cuda.stream(s1):
            h.copy_(d, non_blocking=True)
        with torch.cuda.stream(s2):
            d2.copy_(h2, non_blocking=True)
        b1.record(s1)
        b2.record(s2)
        torch.cuda.synchronize()
        if i >= 2:
            ms = max(a.elapsed_time(b1), a.elapsed_time(b2))
            best = ms if best is None else min(best, ms)
    out["bidir"] = 2 * n / (best * 1e-3) / GB
    return out


def host_mem_available() -> int:
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    return int(line.split()[1]) * 1024
    except OSError:
        pass
    return 0


def cpu_model() -> str:
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    import platform
    return platform.processor() or platform.machine()


def sm_link_peak(torch, probe, dev, host_region, dev_buf, ctas_list=(76, 152, 304)):
    """Best of 5 plain SM streaming copies (kvx_probe_stream_copy) between a device
    buffer and a region of a mapped pinned pool, per direction, GB/s, over a few
    grid sizes (CTAs of 256 threads)."""
    n = min(host_region.numel(), dev_buf.numel()) // 16 * 16
    s = torch.cuda.Stream(device=dev)
    out = {}
    for name, dst, src in (("d2h", host_region, dev_buf), ("h2d", dev_buf, host_region)):
        best, best_ctas = None, None
        for ctas in ctas_list:
            for i in range(7):
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(s)
                probe.kvx_probe_stream_copy(dst, src, n, ctas, stream=s)
                b.record(s)
                b.synchronize()
                if i >= 2 and (best is None or a.elapsed_time(b) < best):
                    best, best_ctas = a.elapsed_time(b), ctas
        out[name] = n / (best * 1e-3) / GB
        out[name + "_ctas"] = best_ctas
    out["bytes"] = n
    return out


def refill(torch, layers, stream, value):
    """Poison a destination pool on `stream` (a write of the whole pool, larger than L2)."""
    with torch.cuda.stream(stream):
        for t in layers:
            t.fill_(value)


def timed_steps(torch, k, ctx, src, dst, ta, tb, T, C, chunks, stream, steps, warmup, refill_fn, world=1):
    """Warm-up then `steps` store + restore steps, each after an untimed refill of the
    destination pool; per-step (store_ms, restore_ms) from CUDA events on `stream`."""
    for _ in range(warmup):
        refill_fn()
        k.kv_store(ctx, src, ta, 0, T, C, chunks, stream=stream)
        k.kv_load(ctx, dst, tb, 0, T, C, chunks, stream=stream)
    stream.synchronize()
    assert k.kv_get_device_error(ctx) == -1
    k.kv_ctx_reset_stats(ctx)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    torch.cuda.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    for i in range(steps):
        refill_fn()
        ev[i][0].record(stream)
        k.kv_store(ctx, src, ta, 0, T, C, chunks, stream=stream)
        ev[i][1].record(stream)
        k.kv_load(ctx, dst, tb, 0, T, C, chunks, stream=stream)
        ev[i][2].record(stream)
    torch.cuda.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    return [e[0].elapsed_time(e[1]) for e in ev], [e[1].elapsed_time(e[2]) for e in ev]


def span(ms):
    return {"median": statistics.median(ms), "min": min(ms), "max": max(ms), "n": len(ms)}


def dominant_kernel(k, stats):
    """Per-direction launches, average duration and bytes of the timed kernel launches."""
    kern = {}
    for d, name in ((0, "pack"), (1, "unpack")):
        nl = stats["timed_launches"][d]
        if nl:
            avg_ms = stats["kernel_ms"][d] / nl
            per_launch = stats["kernel_bytes"][d] / nl
            kern[name] = {"launches": nl, "avg_launch_ms": avg_ms, "bytes_per_launch": per_launch,
                          "total_ms": stats["kernel_ms"][d], "achieved_gbs": per_launch / (avg_ms * 1e-3) / GB}
    return kern


def link_ceiling(link, sm_link, direction):
    """The host link's ceiling for one direction: the larger of the copy engines'
    and the SMs' measured rate, and which one it is."""
    ce, sm = link[direction], (sm_link or {}).get(direction, 0.0)
    return (sm, "sm_stream") if sm > ce else (ce, "copy_engine")


def config_leg(torch, k, synth, name, dev, local, link, sm_link, steps, warmup):
    """Store + restore of another workload, timed the same way as the headline one."""
    cfg = CONFIGS[name]
    s = cfg["shape"]
    L, B, H, D, e, C = s["L"], s["B"], s["H"], s["D"], s["e"], s["C"]
    N, T = cfg["pool_blocks"], cfg["tokens"]
    X = bytes_per_direction(cfg)
    P = 1
    page = 2 * H * B * D * e
    n_chunks = -(-T // C)
    cb = L * 2 * C * H * D * e
    src_layers = [synth.normal_bf16_(torch.empty(N * page, dtype=torch.uint8, device=dev), synth.SEED + l)
                  for l in range(L)]
    dst_layers = [torch.full((N * page,), synth.POISON, dtype=torch.uint8, device=dev) for _ in range(L)]
    src = k.KvPool(src_layers, N, B, H, D, e, k.KVX_LAYOUT_HND, P)
    dst = k.KvPool(dst_layers, N, B, H, D, e, k.KVX_LAYOUT_HND, P)
    ta = torch.from_numpy(synth.permuted_table(N, -(-T // B), seed=1)).to(dev)
    tb = torch.from_numpy(synth.permuted_table(N, -(-T // B), seed=2)).to(dev)
    t_pin = time.perf_counter()
    pool = k.HostBuffer(n_chunks * cb)
    pin_s = time.perf_counter() - t_pin
    chunks = [pool.tensor[i * cb:(i + 1) * cb] for i in range(n_chunks)]
    ctx = k.kv_ctx_create(local, flags=k.KVX_FLAG_TIME_KERNELS)
    stream = torch.cuda.Stream(device=dev)
    torch.cuda.synchronize()  # the pools were written on the default stream; the steps run on `stream`
    try:
        st, ld = timed_steps(torch, k, ctx, src, dst, ta, tb, T, C, chunks, stream, steps, warmup,
                             lambda: refill(torch, dst_layers, stream, synth.POISON))
        kern = dominant_kernel(k, k.kv_ctx_stats(ctx))
        assert k.kv_get_device_error(ctx) == -1
    finally:
        k.kv_ctx_destroy(ctx)
    # the whole pages of the first and the last chunk, restored into the cold pool,
    # equal the source pages (a partial last page holds only the range's tokens)
    same = True
    bpc = C // B
    for c in (0, n_chunks - 1):
        hi = min((c + 1) * bpc, T // B)
        pa, pb = ta[c * bpc:hi].long(), tb[c * bpc:hi].long()
        for l in (0, L - 1):
            same = same and bool(torch.equal(src_layers[l].view(-1, page).index_select(0, pa),
                                             dst_layers[l].view(-1, page).index_select(0, pb)))
    del chunks
    pool.close()
    d2h, d2h_src = link_ceiling(link, sm_link, "d2h")
    h2d, h2d_src = link_ceiling(link, sm_link, "h2d")
    store_gbs = X / (statistics.median(st) * 1e-3) / GB
    restore_gbs = X / (statistics.median(ld) * 1e-3) / GB
    out = {"workload": workload_name(cfg), "tokens": T, "bytes_per_direction": X, "steps": steps,
           "store_ms": span(st), "restore_ms": span(ld),
           "store_gbs": store_gbs, "restore_gbs": restore_gbs,
           "value_gbs": 2 * X * steps / (sum(st) + sum(ld)) / 1e-3 / GB,
           "store_frac": store_gbs / d2h, "restore_frac": restore_gbs / h2d,
           "frac_against": {"d2h": d2h_src, "h2d": h2d_src},
           "kernels": {n_: {"avg_launch_ms": v["avg_launch_ms"], "bytes_per_launch": v["bytes_per_launch"],
                            "link_gbs": v["bytes_per_launch"] / 2 / (v["avg_launch_ms"] * 1e-3) / GB}
                       for n_, v in kern.items()},
           "pinned_host_bytes": n_chunks * cb, "pin_seconds": pin_s,
           "restored_pages_equal_source_on_sample": same}
    del src_layers, dst_layers, src, dst
    torch.cuda.empty_cache()
    return out


def hybrid_leg(torch, k, synth, local):
    """The hybrid six-turn session of two replicas (16 paged attention layers + 48
    recurrent pages of 1,097,728 B): first restore of the 32k-token context with
    its state snapshot, then per turn a restore of the 2,048 tokens the other
    replica added plus the snapshot, and a store of the new tokens plus the new
    snapshot.  Timed with CUDA events on the stream; parity is in the tests."""
    from paper_2609_15021_gb300.hybrid import HybridShape, Replica, SharedTier, load_prefix, store_prefix
    shape = HybridShape()
    first, append, turns, n_blk = 32768, 2048, 6, 4096
    tier = SharedTier(shape, first + (turns - 1) * append, max_snapshots=4)
    reps = [Replica(shape, n_blk, 2, list(map(int, synth.permuted_table(n_blk, n_blk, r + 1)))) for r in range(2)]
    for rep in reps:
        for t in rep.attn_layers + rep.state:
            t.fill_(synth.POISON)
    ctx = k.kv_ctx_create(local)
    stream = torch.cuda.Stream()
    loads, stores = [], []
    try:
        n = 0
        for turn in range(turns):
            rep = reps[turn % 2]
            if turn > 0:
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                lo = rep.tokens
                a.record(stream)
                with torch.cuda.stream(stream):
                    load_prefix(ctx, rep, tier, lo, n, state_slot=0)
                b.record(stream)
                stream.synchronize()
                loads.append((n - lo, a.elapsed_time(b)))
            lo, hi = n, (first if turn == 0 else n + append)
            rep.grow(hi)
            rep.tokens = hi
            torch.cuda.synchronize()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            with torch.cuda.stream(stream):
                store_prefix(ctx, rep, tier, lo, hi, state_slot=0)
            b.record(stream)
            stream.synchronize()
            stores.append((hi - lo, a.elapsed_time(b)))
            n = hi
        assert k.kv_get_device_error(ctx) == -1
    finally:
        k.kv_ctx_destroy(ctx)
        tier.close()
    per_tok = shape.chunk_bytes // shape.chunk_tokens
    first_bytes = loads[0][0] * per_tok + shape.snapshot_bytes
    turn_bytes = append * per_tok + shape.snapshot_bytes
    turn_loads = [ms for tok, ms in loads[1:]]
    turn_stores = [ms for tok, ms in stores[1:]]
    return {"workload": "hybrid six-turn session: 64 layers (16 paged bf16 attention layers x 8 KV heads x "
                        "head_dim 128, 16-token pages; 48 recurrent pages of fp32 16x128x128 state + bf16 "
                        "convolution window, 1,097,728 B each), 32k-token context then +2,048 tokens per turn, "
                        "replicas alternating",
            "first_restore_ms": loads[0][1], "first_restore_bytes": first_bytes,
            "first_restore_gbs": first_bytes / (loads[0][1] * 1e-3) / GB,
            "turn_restore_ms": span(turn_loads), "turn_store_ms": span(turn_stores),
            "turn_bytes_per_direction": turn_bytes,
            "turn_restore_gbs": turn_bytes / (statistics.median(turn_loads) * 1e-3) / GB,
            "turn_store_gbs": turn_bytes / (statistics.median(turn_stores) * 1e-3) / GB}


# ------------------------------------------------------------------ replicas sharing one tier (N > 1)


def ring_plan(world: int, n_chunks: int, chunk_bytes: int, budget_bytes: int) -> dict:
    """How N replicas share one pinned tier: each rank owns `slots_per_rank` slots
    (its whole context if the budget allows) and moves its context in `rounds`
    rounds per step."""
    per_rank = min(n_chunks, budget_bytes // (world * chunk_bytes))
    if per_rank < 1:
        raise RuntimeError(f"a tier of {budget_bytes} bytes holds no chunk of {chunk_bytes} bytes per rank")
    return {"slots_per_rank": int(per_rank), "n_slots": int(per_rank * world), "rounds": -(-n_chunks // per_rank)}


def ring_source(rank: int, world: int) -> int:
    """The rank whose context `rank` restores: rank r stores, rank r+1 restores."""
    return (rank - 1) % world


def context_tokens(rank: int, T: int):
    """Token ids of rank `rank`'s context (its tier keys derive from them)."""
    from paper_2609_15021_gb300 import synth
    return synth.rng(synth.SEED + 7919 * (rank + 1)).integers(0, 150000, size=T).astype("int32")


def step_salt(step: int) -> int:
    """Salt of the tier keys of step `step`.  Every step stores its contexts under
    keys of their own (a new namespace, as for a new request): with the same keys
    every step, a reader would find the previous step's entry still readable,
    pin it and restore it before the writer had stored this step's bytes, and the
    writer's reservation of that key would then fail as busy."""
    return (314159 + 1000003 * step) & (2 ** 64 - 1)


def ring_keys(k, rank: int, world: int, T: int, C: int, step: int):
    """(this rank's keys, the keys of the rank it restores) for one step."""
    own = k.kv_chunk_keys(context_tokens(rank, T), C, salt=step_salt(step))
    src = k.kv_chunk_keys(context_tokens(ring_source(rank, world), T), C, salt=step_salt(step))
    return own, src


def wait_readable(tier, keys, timeout_s: float = 120.0) -> None:
    """Bounded wait, on the host, until every key has a readable entry (the writer's
    GPU has published its commit): kv_tier_wait, which polls with a growing sleep
    and holds the tier's process-shared lock only while it checks."""
    tier.wait(keys, timeout_s)


def ring_round(tier, plan, j, n_chunks, own_keys, src_keys, store_fn, load_fn, settle_fn, barrier_fn, stream):
    """Round j of a step: store this rank's chunks of the round into the tier, restore
    the source rank's chunks of the round from it, settle, and meet the other ranks
    (so that the next round may evict this one's entries)."""
    lo = j * plan["slots_per_rank"]
    hi = min(n_chunks, lo + plan["slots_per_rank"])
    own = own_keys[lo:hi]
    slots = tier.reserve_many(own, as_chunk_list=True)
    store_fn(lo, hi, slots)
    tier.commit_many(own, stream=stream)
    theirs = src_keys[lo:hi]
    wait_readable(tier, theirs)
    slots_r = tier.acquire_many(theirs, stream=stream, as_chunk_list=True)
    load_fn(lo, hi, slots_r)
    tier.release_many(theirs, stream=stream)
    settle_fn()
    tier.poll()
    barrier_fn()


def run_shared(args, world, rank, local):
    """N replicas, one GPU each, sharing one pinned host tier (POSIX shared memory)."""
    import numpy as np
    import torch

    from paper_2609_15021_gb300 import kvxfer as k
    from paper_2609_15021_gb300 import synth

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    cfg = CONFIGS[args.config]
    s = cfg["shape"]
    L, B, H, D, e, C = s["L"], s["B"], s["H"], s["D"], s["e"], s["C"]
    N, T = cfg["pool_blocks"], cfg["tokens"]
    page = 2 * H * B * D * e
    X = bytes_per_direction(cfg)
    n_chunks = -(-T // C)
    cb = L * 2 * C * H * D * e
    src_layers = [synth.normal_bf16_(torch.empty(N * page, dtype=torch.uint8, device=dev),
                                     synth.SEED + 1000 * rank + l) for l in range(L)]
    dst_layers = [torch.full((N * page,), synth.POISON, dtype=torch.uint8, device=dev) for _ in range(L)]
    src = k.KvPool(src_layers, N, B, H, D, e)
    dst = k.KvPool(dst_layers, N, B, H, D, e)
    ta_np = synth.permuted_table(N, T // B, seed=1 + 1000 * rank)
    tb_np = synth.permuted_table(N, T // B, seed=2 + 1000 * rank)
    ta, tb = torch.from_numpy(ta_np).to(dev), torch.from_numpy(tb_np).to(dev)
    ta_host, tb_host = torch.from_numpy(ta_np).pin_memory(), torch.from_numpy(tb_np).pin_memory()
    link = sm_link = None
    if rank == 0:  # this GPU's host-link ceilings, before any rank moves data
        from paper_2609_15021_gb300 import probe
        link_bufs = link_buffers(torch, dev)
        link = host_link_peak(torch, dev, link_bufs)
        sm_link = sm_link_peak(torch, probe, dev, link_bufs["h"], link_bufs["d"])
        del link_bufs
    barrier(world)
    # rank 0 sizes the tier and names it; every rank opens it
    if rank == 0:
        budget = int(min(args.tier_budget_gib * 2 ** 30, host_mem_available() - (32 << 30),
                         shm_free_bytes() - (1 << 30)))
        plan = ring_plan(world, n_chunks, cb, budget)
        name = f"/kvx_ring_{os.getpid()}"
        tier = k.KvTier(cb, plan["n_slots"], shared_name=name, create=True)
        msg = [name, plan]
    else:
        msg = [None, None]
    if world > 1:
        import torch.distributed as dist
        dist.broadcast_object_list(msg, src=0)
    name, plan = msg
    if rank != 0:
        tier = k.KvTier(shared_name=name)
    barrier(world)
    if rank == 0:  # every rank has it open: the memory goes with the last of them, however they end
        try:
            os.unlink("/dev/shm" + name)
        except OSError:
            pass
    step_keys = [ring_keys(k, rank, world, T, C, i) for i in range(args.warmup + args.steps)]
    ctx = k.kv_ctx_create(local, flags=k.KVX_FLAG_TIME_KERNELS)
    stream = torch.cuda.Stream(device=dev)
    torch.cuda.synchronize()  # the pools were written on the default stream; the steps run on `stream`

    def store_fn(lo, hi, slots):
        k.kv_store(ctx, src, ta, lo * C, min(T, hi * C), C, slots, stream=stream)

    def load_fn(lo, hi, slots):
        k.kv_load(ctx, dst, tb, lo * C, min(T, hi * C), C, slots, stream=stream)

    def step(i):
        own_keys, src_keys = step_keys[i]
        for j in range(plan["rounds"]):
            ring_round(tier, plan, j, n_chunks, own_keys, src_keys, store_fn, load_fn, stream.synchronize,
                       lambda: barrier(world), stream)

    for i in range(args.warmup):
        refill(torch, dst_layers, stream, synth.POISON)
        step(i)
    assert k.kv_get_device_error(ctx) == -1
    k.kv_ctx_reset_stats(ctx)
    step_ms, host_s = [], []
    torch.cuda.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    with ClockSampler(local) as clocks:
        for i in range(args.steps):
            refill(torch, dst_layers, stream, synth.POISON)
            stream.synchronize()
            t0 = time.perf_counter()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            with torch.cuda.stream(stream):   # the step's block tables, from pinned host memory
                ta.copy_(ta_host, non_blocking=True)
                tb.copy_(tb_host, non_blocking=True)
            step(args.warmup + i)
            b.record(stream)
            stream.synchronize()
            host_s.append(time.perf_counter() - t0)
            step_ms.append(a.elapsed_time(b))
        torch.cuda.synchronize()
        barrier(world)
        torch.cuda.synchronize()
    clock_info = clocks.summary()
    stats = k.kv_ctx_stats(ctx)
    assert k.kv_get_device_error(ctx) == -1
    # this rank restored rank r-1's context: its restored pages equal the chunk bytes in
    # the tier (checked on sampled chunks after one more step)
    tstats = tier.stats()
    k.kv_ctx_destroy(ctx)
    tier.close()
    total_ms = max_over_ranks(world, sum(step_ms), local)
    total_host = max_over_ranks(world, sum(host_s), local)
    if rank != 0:
        return 0
    value = 2 * X * args.steps * world / (total_ms * 1e-3) / GB
    kern = dominant_kernel(k, stats)
    roofline = None
    if kern:
        dom = max(kern, key=lambda n: kern[n]["total_ms"])
        direction = "d2h" if dom == "pack" else "h2d"
        link_bytes = kern[dom]["bytes_per_launch"] / 2
        achieved = link_bytes / (kern[dom]["avg_launch_ms"] * 1e-3) / GB
        peak, which = link_ceiling(link, sm_link, direction)
        roofline = {"bound": "host_link", "kernel": f"move_kernel<{dom},HND> (zero-copy), rank 0",
                    "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                    "traffic": recorded_traffic(s).get(f"zerocopy_{dom}", link_bytes),
                    "peak_source": f"rank 0's GPU before the timed steps, {direction}: copy engines (pinned "
                                   f"cudaMemcpyAsync of 1 GiB) {link[direction]:.1f} GB/s, SM streaming copy "
                                   f"{sm_link[direction]:.1f} GB/s; used: {which}",
                    "algorithmic_bytes_per_launch": link_bytes}
    line = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u8",
        "data": "synthetic: bf16 ~N(0,1) KV from a fixed seed per rank; seeded random-permutation block tables",
        "config": {"workload": workload_name(cfg), "context_tokens": T, "layers": L, "kv_heads": H, "head_dim": D,
                   "kv_dtype": s["dtype"], "block_tokens": B, "chunk_tokens": C, "pool_blocks": N,
                   "bytes_per_direction_per_rank": X,
                   "l2": f"inputs larger than L2 ({X} bytes per direction); destination pool refilled before "
                         f"every step, outside the timed region",
                   "parallelism": f"replicas x{world} sharing one pinned host tier: rank r stores its context, "
                                  f"rank r+1 restores it",
                   "tier_bytes": plan["n_slots"] * cb, "tier_slots": plan["n_slots"],
                   "rounds_per_step": plan["rounds"]},
        "e2e": {"value": 2 * X * args.steps * world / total_host / GB, "unit": "GB/s",
                "h2d_bytes_per_step": X + ta_np.nbytes + tb_np.nbytes, "d2h_bytes_per_step": X},
        "kernels": kern, "tier": tstats, "gpu_launches": stats["kernel_launches"], "clocks": clock_info,
        "cpu_baseline": None, "roofline": roofline,
        "host_link": {"peak_d2h_gbs": link["d2h"], "peak_h2d_gbs": link["h2d"], "peak_bidir_gbs": link["bidir"],
                      "sm_stream_d2h_gbs": sm_link["d2h"], "sm_stream_h2d_gbs": sm_link["h2d"]},
    }
    print(json.dumps(line), flush=True)
    return 0


def concurrent_leg(torch, k, probe, dev, local, args, mode, ctx, src, dst, ta, tb, T, C, chunks, host_pool,
                   host_pool2, cb, n_chunks, X, link, stream):
    """Two replicas at once: A (ctx, `stream`) stores the context into a second chunk
    set while B (its own context and stream) restores the first chunk set into the
    cold pool; >= 10 repetitions after 2 warm-ups.  Beside it, over the same two
    chunk sets, both directions at once: the copy engines (cudaMemcpyAsync per
    chunk) and the SMs (a plain streaming copy per 4 GiB piece).  The two probes
    run inside every repetition, right after the replicas, so each repetition
    compares the replicas with the link's both-ways rate at that moment (the host
    link's both-ways rate varies from one second to the next on a shared host)."""
    pool2 = host_pool2.info()
    chunks2 = [host_pool2.tensor[i * cb:(i + 1) * cb] for i in range(n_chunks)]
    ctx_b = k.kv_ctx_create(local, store_mode=mode, load_mode=mode, staging_slot_bytes=args.slot_mib << 20,
                            flags=k.KVX_FLAG_TIME_KERNELS)
    s_b = torch.cuda.Stream(device=dev)
    s_c = torch.cuda.Stream(device=dev)
    piece = 4 << 30
    total = n_chunks * cb
    d_a = torch.empty(cb, dtype=torch.uint8, device=dev)
    d_b = torch.empty(cb, dtype=torch.uint8, device=dev)
    dev_a = torch.empty(piece, dtype=torch.uint8, device=dev)
    dev_b = torch.empty(piece, dtype=torch.uint8, device=dev)

    def both_ways(run_d2h, run_h2d):
        """(ms of the D2H side, ms of the H2D side), both started together."""
        a, ea, eb = (torch.cuda.Event(enable_timing=True) for _ in range(3))
        torch.cuda.synchronize()
        a.record(stream)
        s_c.wait_event(a)
        run_d2h(stream)
        ea.record(stream)
        run_h2d(s_c)
        eb.record(s_c)
        torch.cuda.synchronize()
        return a.elapsed_time(ea), a.elapsed_time(eb)

    def ce_d2h(s):   # copy engines: every chunk of both chunk sets, one direction each
        with torch.cuda.stream(s):
            for c in range(n_chunks):
                chunks2[c].copy_(d_a, non_blocking=True)

    def ce_h2d(s):
        with torch.cuda.stream(s):
            for c in range(n_chunks):
                d_b.copy_(chunks[c], non_blocking=True)

    def sm_pass(host, into_host, s):  # SMs: a plain streaming copy, 4 GiB per launch, 76 CTAs a direction
        for off in range(0, total, piece):
            n = min(piece, total - off)
            h = host.tensor[off:off + n]
            if into_host:
                probe.kvx_probe_stream_copy(h, dev_a, n, 76, stream=s)
            else:
                probe.kvx_probe_stream_copy(dev_b, h, n, 76, stream=s)

    st_ms, ld_ms, agg, sm_agg, ce_agg = [], [], [], [], []
    reps = max(10, args.concurrent_reps)
    picks = sorted({0, n_chunks // 3, n_chunks // 2, n_chunks - 1})
    same = False
    with ClockSampler(local) as clocks:
        for i in range(2 + reps):
            if i == 2:
                k.kv_ctx_reset_stats(ctx)
                k.kv_ctx_reset_stats(ctx_b)
            refill(torch, dst.layers, stream, 0xA5)
            a, ea, eb = (torch.cuda.Event(enable_timing=True) for _ in range(3))
            torch.cuda.synchronize()
            a.record(stream)
            s_b.wait_event(a)
            k.kv_store(ctx, src, ta, 0, T, C, chunks2, stream=stream)
            ea.record(stream)
            k.kv_load(ctx_b, dst, tb, 0, T, C, chunks, stream=s_b)
            eb.record(s_b)
            torch.cuda.synchronize()
            if i == 1 + reps:  # A's chunks, before the probes below write over that chunk set
                same = all(torch.equal(chunks2[c], chunks[c]) for c in picks)
            sm = max(both_ways(lambda s: sm_pass(host_pool2, True, s), lambda s: sm_pass(host_pool, False, s)))
            ce = max(both_ways(ce_d2h, ce_h2d))
            if i >= 2:
                st_ms.append(a.elapsed_time(ea))
                ld_ms.append(a.elapsed_time(eb))
                agg.append(2 * X / (max(st_ms[-1], ld_ms[-1]) * 1e-3) / GB)
                sm_agg.append(2 * X / (sm * 1e-3) / GB)
                ce_agg.append(2 * X / (ce * 1e-3) / GB)
    clock_info = clocks.summary()
    sa, sb = k.kv_ctx_stats(ctx), k.kv_ctx_stats(ctx_b)
    assert k.kv_get_device_error(ctx) == -1 and k.kv_get_device_error(ctx_b) == -1
    kernels = {}
    for name, st_, d in (("pack (replica A)", sa, 0), ("unpack (replica B)", sb, 1)):
        if st_["timed_launches"][d]:
            ms = st_["kernel_ms"][d] / st_["timed_launches"][d]
            by = st_["kernel_bytes"][d] / st_["timed_launches"][d] / 2
            kernels[name] = {"avg_launch_ms": ms, "link_bytes_per_launch": by, "link_gbs": by / (ms * 1e-3) / GB,
                             "launches": st_["timed_launches"][d]}
    k.kv_ctx_destroy(ctx_b)
    del d_a, d_b, dev_a, dev_b, chunks2
    host_pool2.close()
    med = statistics.median(agg)
    sm_med, ce_med = statistics.median(sm_agg), statistics.median(ce_agg)
    return {"aggregate_gbs": span(agg), "store_ms": span(st_ms), "restore_ms": span(ld_ms),
            "span_ms": span([max(a_, b_) for a_, b_ in zip(st_ms, ld_ms)]), "reps": len(agg),
            "peak_bidir_gbs": link["bidir"], "frac": med / link["bidir"],
            "peak_bidir_same_size_gbs": ce_med, "frac_same_size": med / ce_med,
            "sm_stream_bidir_same_size_gbs": sm_med, "frac_sm_stream_same_size": med / sm_med,
            "per_rep": {"sm_stream_gbs": span(sm_agg), "copy_engine_gbs": span(ce_agg),
                        "frac_sm_stream": span([r / p for r, p in zip(agg, sm_agg)]),
                        "frac_copy_engine": span([r / p for r, p in zip(agg, ce_agg)])},
            "kernels": kernels, "clocks": clock_info,
            "second_store_equals_first_on_sampled_chunks": same, "second_pool": pool2,
            "what": "replica A kv_store of the context into a second pinned chunk set while replica B kv_load "
                    "of the timed steps' chunks into its (refilled) pool, own context and stream each; "
                    "aggregate = 2 x bytes / the slower of the two, per repetition; peak_bidir = pinned "
                    "cudaMemcpyAsync of 1 GiB each way at once; in every repetition, right after the replicas, "
                    "over the same two chunk sets, both directions at once: cudaMemcpyAsync of every chunk "
                    "(peak_bidir_same_size, median over the repetitions) and a plain SM streaming copy, 76 CTAs "
                    "a direction (sm_stream_bidir_same_size, median); per_rep.frac_* = the replicas' rate over "
                    "the probe's in the same repetition"}


def run_ours(args):
    import numpy as np
    import torch

    world, rank, local = dist_init(args)
    from paper_2609_15021_gb300 import _build
    _build.build()
    if world > 1 or args.shared_tier:
        return run_shared(args, world, rank, local)
    from paper_2609_15021_gb300 import kvxfer as k
    from paper_2609_15021_gb300 import probe
    from paper_2609_15021_gb300 import synth

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    cfg = CONFIGS[args.config]
    s = cfg["shape"]
    L, B, H, D, e, C = s["L"], s["B"], s["H"], s["D"], s["e"], s["C"]
    N, T = cfg["pool_blocks"], cfg["tokens"]
    page = 2 * H * B * D * e
    layer_bytes = N * page
    X = bytes_per_direction(cfg)
    n_chunks = -(-T // C)
    cb = L * 2 * C * H * D * e

    # Every host buffer of the run is pinned up front, before the warm-up: on
    # GB300, pinning or freeing host memory while (or just before) zero-copy
    # kernels ran stalled them for up to a second, and such stalls inside a
    # measured leg would come from this harness, not from the transfer.
    link_bufs = link_buffers(torch, dev)
    link = host_link_peak(torch, dev, link_bufs)

    src_layers = [synth.normal_bf16_(torch.empty(layer_bytes, dtype=torch.uint8, device=dev), synth.SEED + l)
                  for l in range(L)]
    dst_layers = [torch.full((layer_bytes,), synth.POISON, dtype=torch.uint8, device=dev) for _ in range(L)]
    lay = k.KVX_LAYOUT_NHD if args.layout == "nhd" else k.KVX_LAYOUT_HND
    LAY = args.layout.upper()
    src = k.KvPool(src_layers, N, B, H, D, e, lay)
    dst = k.KvPool(dst_layers, N, B, H, D, e, lay)
    ta_np = synth.permuted_table(N, T // B, seed=1)
    tb_np = synth.permuted_table(N, T // B, seed=2)
    ta = torch.from_numpy(ta_np).to(dev)
    tb = torch.from_numpy(tb_np).to(dev)
    avail = host_mem_available()
    t_pin = time.perf_counter()
    # exact-size pinned, mapped pool (no power-of-two rounding)
    host_alloc = args.host_alloc if args.host_alloc != "auto" else "huge" if args.mode == "staged" else "plain"
    host_pool = k.HostBuffer(n_chunks * cb, numa_node=k.KVX_NUMA_NEAREST if host_alloc == "numa" else None,
                             driver=host_alloc == "driver", huge=host_alloc == "huge")
    pin_seconds = time.perf_counter() - t_pin
    chunks = [host_pool.tensor[i * cb:(i + 1) * cb] for i in range(n_chunks)]
    # the pinned memory of the later legs: a second chunk set (two replicas at
    # once) and the e2e leg's pinned block tables.  The shared tier's pool is
    # made once the second chunk set is freed: three 33 GB pools pinned at once
    # left the two-replica leg at half its speed.
    want_conc = not args.no_concurrent and avail > 2 * n_chunks * cb + (32 << 30)
    want_tier = (not args.no_tier and avail > 2 * n_chunks * cb + (32 << 30)
                 and shm_free_bytes() > n_chunks * cb + (1 << 30))
    host_pool2 = k.HostBuffer(n_chunks * cb, huge=host_alloc == "huge") if want_conc else None
    ta_host = torch.from_numpy(ta_np).pin_memory()
    tb_host = torch.from_numpy(tb_np).pin_memory()
    # the SMs' own ceiling on the host link: a plain streaming copy between device
    # memory and the same mapped pinned pool the transfers use
    sm_link = sm_link_peak(torch, probe, dev, host_pool.tensor[: link_bufs["d"].numel()], link_bufs["d"])

    mode = {"auto": k.KVX_MODE_AUTO, "staged": k.KVX_MODE_STAGED, "zerocopy": k.KVX_MODE_ZEROCOPY}[args.mode]
    ctx = k.kv_ctx_create(local, store_mode=mode, load_mode=mode, staging_slot_bytes=args.slot_mib << 20,
                          flags=k.KVX_FLAG_TIME_KERNELS)
    store_mode, load_mode = k.kv_ctx_modes(ctx)
    stream = torch.cuda.Stream(device=dev)
    poison_dst = lambda: refill(torch, dst_layers, stream, synth.POISON)  # noqa: E731
    torch.cuda.synchronize()  # the pools were written on the default stream; the steps run on `stream`

    with ClockSampler(local) as clocks:
        store_ms, restore_ms = timed_steps(torch, k, ctx, src, dst, ta, tb, T, C, chunks, stream, args.steps,
                                           args.warmup, poison_dst)
    clock_info = clocks.summary()
    # the link peak again right after the timed steps: a drop shows traffic from
    # outside this process (the host memory is shared) during the measurement
    link_after = host_link_peak(torch, dev, link_bufs)
    total_ms = sum(store_ms) + sum(restore_ms)
    stats = k.kv_ctx_stats(ctx)
    assert k.kv_get_device_error(ctx) == -1
    value = 2 * X * args.steps / (total_ms * 1e-3) / GB

    # end to end through the public API on the host clock; the refill of the
    # destination pool before each step is outside the timed part
    e2e = None
    if not args.no_e2e:
        e2e_s = 0.0
        chunk_list = k.ChunkList(chunks)  # the chunk set described once, as a serving loop would
        for _ in range(args.steps):
            poison_dst()
            stream.synchronize()
            t0 = time.perf_counter()
            with torch.cuda.stream(stream):
                ta.copy_(ta_host, non_blocking=True)
                tb.copy_(tb_host, non_blocking=True)
            k.kv_store(ctx, src, ta, 0, T, C, chunk_list, stream=stream)
            stream.synchronize()          # the host may use the chunks only after this
            k.kv_load(ctx, dst, tb, 0, T, C, chunk_list, stream=stream)
            stream.synchronize()
            bad = k.kv_get_device_error(ctx)  # device->host read of the step's status word
            e2e_s += time.perf_counter() - t0
            assert bad == -1
        e2e = {"value": 2 * X * args.steps / e2e_s / GB, "unit": "GB/s",
               "h2d_bytes_per_step": X + ta_np.nbytes + tb_np.nbytes, "d2h_bytes_per_step": X + 8}

    # dominant kernel: the direction with more kernel time
    kern = dominant_kernel(k, stats)
    hbm_peak, peak_src = load_peaks()
    traffic = recorded_traffic(s, layout=args.layout)
    roofline = None
    if kern:
        dom = max(kern, key=lambda n: kern[n]["total_ms"])
        zero_copy = (store_mode if dom == "pack" else load_mode) == k.KVX_MODE_ZEROCOPY
        if zero_copy:
            # the kernel moves each byte once over the host link: that link bounds it
            direction = "d2h" if dom == "pack" else "h2d"
            link_bytes = kern[dom]["bytes_per_launch"] / 2
            achieved = link_bytes / (kern[dom]["avg_launch_ms"] * 1e-3) / GB
            peak, which = link_ceiling(link, sm_link, direction)
            roofline = {"bound": "host_link", "kernel": f"move_kernel<{dom},{LAY}> (zero-copy)", "achieved": achieved,
                        "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                        "traffic": traffic.get(f"zerocopy_{dom}", link_bytes),
                        "peak_source": f"the larger of two host-link ceilings measured in this run, {direction}: "
                                       f"copy engines (pinned cudaMemcpyAsync of 1 GiB) {link[direction]:.1f} GB/s, "
                                       f"SM streaming copy over the same mapped pinned pool "
                                       f"({sm_link[direction + '_ctas']} CTAs) {sm_link[direction]:.1f} GB/s; "
                                       f"used: {which}",
                        "copy_engine_peak": link[direction], "sm_stream_peak": sm_link[direction],
                        "frac_of_copy_engine_peak": achieved / link[direction],
                        "frac_of_sm_stream_peak": achieved / sm_link[direction],
                        "algorithmic_bytes_per_launch": link_bytes}
        else:
            roofline = {"bound": "hbm", "kernel": f"tmap_move_kernel<{dom}> (staged: one staging slot per launch)",
                        "achieved": kern[dom]["achieved_gbs"], "peak": hbm_peak, "unit": "GB/s",
                        "frac": kern[dom]["achieved_gbs"] / hbm_peak,
                        "traffic": traffic.get(f"staged_{dom}", kern[dom]["bytes_per_launch"]), "peak_source": peak_src,
                        "algorithmic_bytes_per_launch": kern[dom]["bytes_per_launch"],
                        "note": "in staged mode the copy engines' cudaMemcpyAsync over the host link bound the "
                                "transfer, not this kernel: each launch packs one staging slot in tens of "
                                "microseconds, so launch and tail time weigh on its rate; host_link.store_frac and "
                                "restore_frac give the transfer against the link"}

    # device-side pack / unpack of the same context into device chunks: the
    # HBM-bound form of the kernels (staged mode, kv_pack / kv_unpack)
    hbm_roofline = None
    if not args.no_hbm_roofline:
        dev_slab = torch.empty(n_chunks * cb, dtype=torch.uint8, device=dev)
        dchunks = [dev_slab[i * cb:(i + 1) * cb] for i in range(n_chunks)]

        def device_leg(tma):
            """Per direction: (launches, bytes per launch, ms per launch) of kv_pack / kv_unpack."""
            hctx = k.kv_ctx_create(local, flags=k.KVX_FLAG_TIME_KERNELS | (0 if tma else k.KVX_FLAG_DEVICE_LSU))
            for _ in range(2):
                k.kv_pack(hctx, src, ta, 0, T, C, dchunks, stream=stream)
                k.kv_unpack(hctx, dst, tb, 0, T, C, dchunks, stream=stream)
            stream.synchronize()
            k.kv_ctx_reset_stats(hctx)
            for _ in range(3):
                k.kv_pack(hctx, src, ta, 0, T, C, dchunks, stream=stream)
                k.kv_unpack(hctx, dst, tb, 0, T, C, dchunks, stream=stream)
            stream.synchronize()
            hs = k.kv_ctx_stats(hctx)
            assert k.kv_get_device_error(hctx) == -1
            k.kv_ctx_destroy(hctx)
            return [(hs["timed_launches"][d], hs["kernel_bytes"][d] / hs["timed_launches"][d],
                     hs["kernel_ms"][d] / hs["timed_launches"][d]) for d in (0, 1)]

        tma = args.device_engine == "tma"
        legs = {tma: device_leg(tma), not tma: device_leg(not tma)}  # the chosen engine and the other one
        dev_traffic = recorded_traffic(s, "tma_kernels.cu", args.layout) if tma else traffic
        tma_engine = ("TMA tensor-map boxes (tmap_move_kernel)" if args.layout == "hnd" else
                      "TMA bulk copies, one per side of a unit (tma_move_kernel)")
        hbm_roofline = {"bound": "hbm", "peak": hbm_peak, "unit": "GB/s", "peak_source": peak_src,
                        "engine": tma_engine if tma else "16-byte loads/stores (move_kernel)"}
        for d, name in ((0, "pack"), (1, "unpack")):
            nl, per_launch, ms = legs[tma][d]
            achieved = per_launch / (ms * 1e-3) / GB
            kname = ((f"tmap_move_kernel<{name}>" if args.layout == "hnd" else f"tma_move_kernel<{name},NHD>")
                     if tma else f"move_kernel<{name},{LAY}>")
            hbm_roofline[name] = {"kernel": f"{kname} (device chunks)", "achieved": achieved,
                                  "frac": achieved / hbm_peak, "launches": nl,
                                  "algorithmic_bytes_per_launch": per_launch, "avg_launch_ms": ms,
                                  "traffic": dev_traffic.get(f"device_{name}", per_launch)}
        # this GPU's device-to-device copy rate right now (context for the peak above)
        a = dev_slab[: len(dev_slab) // 2]
        b = dev_slab[len(dev_slab) // 2: 2 * (len(dev_slab) // 2)]
        best = None
        for i in range(6):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            with torch.cuda.stream(stream):
                b.copy_(a)
            e1.record(stream)
            e1.synchronize()
            if i >= 1:
                best = e0.elapsed_time(e1) if best is None else min(best, e0.elapsed_time(e1))
        hbm_roofline["copy_this_run_gbs"] = 2 * a.numel() / (best * 1e-3) / GB
        del a, b
        other = legs[not tma]
        hbm_roofline["other_engine"] = {
            "engine": "16-byte loads/stores (move_kernel)" if tma else tma_engine,
            **{name: {"achieved": other[d][1] / (other[d][2] * 1e-3) / GB,
                      "frac": other[d][1] / (other[d][2] * 1e-3) / GB / hbm_peak, "avg_launch_ms": other[d][2]}
               for d, name in ((0, "pack"), (1, "unpack"))}}
        del dev_slab, dchunks

    store_gbs = X / (statistics.median(store_ms) * 1e-3) / GB
    restore_gbs = X / (statistics.median(restore_ms) * 1e-3) / GB
    d2h_peak, d2h_src = link_ceiling(link, sm_link, "d2h")
    h2d_peak, h2d_src = link_ceiling(link, sm_link, "h2d")
    host_link = {"store_gbs": store_gbs, "restore_gbs": restore_gbs, "peak_d2h_gbs": link["d2h"],
                 "peak_h2d_gbs": link["h2d"], "peak_bidir_gbs": link["bidir"],
                 "sm_stream_d2h_gbs": sm_link["d2h"], "sm_stream_h2d_gbs": sm_link["h2d"],
                 "sm_stream_ctas": {"d2h": sm_link["d2h_ctas"], "h2d": sm_link["h2d_ctas"]},
                 "store_frac": store_gbs / d2h_peak, "restore_frac": restore_gbs / h2d_peak,
                 "frac_against": {"d2h": d2h_src, "h2d": h2d_src},
                 "peak_after_d2h_gbs": link_after["d2h"], "peak_after_h2d_gbs": link_after["h2d"],
                 "peak_source": "copy engines: pinned cudaMemcpyAsync of 1 GiB, best of 5, measured in this run "
                                "before (peak_*) and right after (peak_after_*) the timed steps; SMs: a plain "
                                "16-byte streaming copy kernel (libkvxfer_probe) between 1 GiB of device memory "
                                "and the first 1 GiB of the mapped pinned chunk pool, best of 5 over 76/152/304 "
                                "CTAs"}

    # Two replicas at once, each with its own context and stream: replica A stores
    # the context into a second chunk set while replica B restores the chunks the
    # timed steps wrote.  The host link then carries both directions.
    concurrent = None
    if host_pool2 is not None:
        concurrent = concurrent_leg(torch, k, probe, dev, local, args, mode, ctx, src, dst, ta, tb, T, C, chunks,
                                    host_pool, host_pool2, cb, n_chunks, X, link, stream)

    # The tier path: the same store and restore through a host tier shared across
    # processes (POSIX shared memory, the paper's replicas sharing one pool), as a
    # replica uses it: reserve a slot per chunk key (one call), one kv_store into those slots,
    # commit the keys on the stream (one publication launch per 512); prefix
    # lookup; acquire the keys on the stream, one kv_load from those slots, release
    # the keys on the stream (one event).  The host never waits for the GPU.
    tier_leg = None
    if want_tier:
        shm_name = f"/kvx_bench_{os.getpid()}"
        tier = k.KvTier(cb, n_chunks, shared_name=shm_name, create=True)
        try:  # no other process opens it: unlinked now, the memory goes with this process however it ends
            os.unlink("/dev/shm" + shm_name)
        except OSError:
            pass
        token_ids = synth.rng(synth.SEED).integers(0, 150000, size=T).astype(np.int32)
        keys = k.kv_chunk_keys(token_ids, C, salt=synth.SEED)
        st_ms, ld_ms, host_ms, hits = [], [], [], 0
        for rep in range(2 + 3):
            a, b, c = (torch.cuda.Event(enable_timing=True) for _ in range(3))
            poison_dst()
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            a.record(stream)
            slots = tier.reserve_many(keys, as_chunk_list=True)
            k.kv_store(ctx, src, ta, 0, T, C, slots, stream=stream)
            tier.commit_many(keys, stream=stream)
            b.record(stream)
            hits = tier.prefix_hits(keys)
            slots = tier.acquire_many(keys[:hits], stream=stream, as_chunk_list=True)
            k.kv_load(ctx, dst, tb, 0, T, C, slots, stream=stream)
            tier.release_many(keys[:hits], stream=stream)
            c.record(stream)
            del slots
            t1 = time.perf_counter()
            torch.cuda.synchronize()
            tier.poll()
            if rep >= 2:
                st_ms.append(a.elapsed_time(b))
                ld_ms.append(b.elapsed_time(c))
                host_ms.append((t1 - t0) * 1e3)
        assert k.kv_get_device_error(ctx) == -1
        same = all(torch.equal(tier.acquire(keys[ci], k.KVX_NO_STREAM), chunks[ci])
                   for ci in sorted({0, n_chunks // 2, n_chunks - 1}))
        for ci in sorted({0, n_chunks // 2, n_chunks - 1}):
            tier.release(keys[ci], k.KVX_NO_STREAM)
        tstats = tier.stats()
        tier.close()
        tier_leg = {"store_ms": statistics.median(st_ms), "restore_ms": statistics.median(ld_ms),
                    "store_gbs": X / (statistics.median(st_ms) * 1e-3) / GB,
                    "restore_gbs": X / (statistics.median(ld_ms) * 1e-3) / GB,
                    "host_ms_per_store_and_restore": statistics.median(host_ms),
                    "tier": "shared across processes (POSIX shared memory, base pages, registered pinned "
                            "and mapped)",
                    "prefix_hits": hits, "chunks": n_chunks, "tier_calls_per_step": 5,
                    "transfer_calls_per_direction": 1,
                    "slots_equal_timed_chunks_on_sample": same, "evictions": tstats["evictions"]}

    # The same two replicas, but B restores what A is storing, group by group, as
    # soon as each group is stored: A commits every group of chunks on its stream
    # as it goes, and B's acquire of a group makes B's stream wait for that
    # group's commit.  The time from A's first store to B's last restore is a
    # cross-replica hit that arrives while the context is still being stored.
    streamed = None
    if want_tier:
        shm_name = f"/kvx_stream_{os.getpid()}"
        tier_s = k.KvTier(cb, n_chunks, shared_name=shm_name, create=True)
        try:
            os.unlink("/dev/shm" + shm_name)
        except OSError:
            pass
        token_ids = synth.rng(synth.SEED + 1).integers(0, 150000, size=T).astype(np.int32)
        skeys = k.kv_chunk_keys(token_ids, C, salt=synth.SEED + 1)
        ctx_b = k.kv_ctx_create(local)
        s_b = torch.cuda.Stream(device=dev)
        group = 64
        groups = [(g, min(n_chunks, g + group)) for g in range(0, n_chunks, group)]
        tot_ms, st_ms = [], []
        for rep in range(2 + 3):
            poison_dst()
            torch.cuda.synchronize()
            a, ea, eb = (torch.cuda.Event(enable_timing=True) for _ in range(3))
            a.record(stream)
            s_b.wait_event(a)
            for g0, g1 in groups:
                slots = tier_s.reserve_many(skeys[g0:g1], as_chunk_list=True)
                k.kv_store(ctx, src, ta, g0 * C, min(T, g1 * C), C, slots, stream=stream)
                tier_s.commit_many(skeys[g0:g1], stream=stream)
            ea.record(stream)
            for g0, g1 in groups:
                slots = tier_s.acquire_many(skeys[g0:g1], stream=s_b, as_chunk_list=True)
                k.kv_load(ctx_b, dst, tb, g0 * C, min(T, g1 * C), C, slots, stream=s_b)
                tier_s.release_many(skeys[g0:g1], stream=s_b)
            eb.record(s_b)
            torch.cuda.synchronize()
            tier_s.poll()
            if rep >= 2:
                tot_ms.append(a.elapsed_time(eb))
                st_ms.append(a.elapsed_time(ea))
        assert k.kv_get_device_error(ctx) == -1 and k.kv_get_device_error(ctx_b) == -1
        bpc = C // B
        same = all(bool(torch.equal(src_layers[l].view(-1, page).index_select(0, ta[c * bpc:(c + 1) * bpc].long()),
                                    dst_layers[l].view(-1, page).index_select(0, tb[c * bpc:(c + 1) * bpc].long())))
                   for c in (0, n_chunks // 2, n_chunks - 1) for l in (0, L - 1))
        k.kv_ctx_destroy(ctx_b)
        tier_s.close()
        seq_ms = statistics.median(store_ms) + statistics.median(restore_ms)
        streamed = {"group_chunks": group, "groups": len(groups), "total_ms": span(tot_ms),
                    "store_ms": statistics.median(st_ms),
                    "sequential_ms": seq_ms, "speedup_vs_sequential": seq_ms / statistics.median(tot_ms),
                    "aggregate_gbs": 2 * X / (statistics.median(tot_ms) * 1e-3) / GB,
                    "restored_pages_equal_source_on_sample": same,
                    "what": "replica A stores the context into a shared tier in groups of chunks, committing "
                            "each group on its stream; replica B (own context and stream) acquires each group "
                            "on its stream, which waits for that group's commit, and restores it; total = A's "
                            "first store to B's last restore; sequential = the timed steps' store + restore"}

    # A restore after idle time: the pool untouched for a few seconds, as before
    # the first cross-replica hit after a quiet period.  Once as the library
    # does it by default (its touch threads read one byte per host page first
    # when the context was idle; the transfer waits for them on the stream),
    # once with that off (KVX_FLAG_NO_HOST_TOUCH).  The events bracket the call,
    # so the reads are inside the time; call_ms is the calling thread's time in
    # kv_load.
    cold = None
    if not args.no_cold:
        ctx_nt = k.kv_ctx_create(local, store_mode=mode, load_mode=mode, staging_slot_bytes=args.slot_mib << 20,
                                 flags=k.KVX_FLAG_NO_HOST_TOUCH)
        cold = {"idle_s": args.cold_idle_s}
        for name, c in (("restore_ms_without_host_touch", ctx_nt), ("restore_ms", ctx)):
            poison_dst()
            torch.cuda.synchronize()
            time.sleep(args.cold_idle_s)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            t0 = time.perf_counter()
            k.kv_load(c, dst, tb, 0, T, C, chunks, stream=stream)
            call_ms = (time.perf_counter() - t0) * 1e3
            b.record(stream)
            b.synchronize()
            cold[name] = a.elapsed_time(b)
            cold[name.replace("restore_ms", "call_ms")] = call_ms
        assert k.kv_get_device_error(ctx) == -1 and k.kv_get_device_error(ctx_nt) == -1
        k.kv_ctx_destroy(ctx_nt)
        cold["warm_restore_ms"] = statistics.median(restore_ms)

    cpu = None
    verified = None
    if not args.no_cpu_baseline:
        import oracle
        oracle.build()
        # the chunks of the timed steps' store, written again (the legs above reused the pool)
        k.kv_store(ctx, src, ta, 0, T, C, chunks, stream=stream)
        stream.synchronize()
        S = min(args.cpu_sample_chunks, n_chunks)
        picks = np.linspace(0, n_chunks - 1, S).astype(np.int64)
        bpc = C // B
        pages = np.concatenate([ta_np[c * bpc:(c + 1) * bpc] for c in picks]).astype(np.int64)
        idx = torch.from_numpy(pages).to(dev)
        pool_np = [t.view(-1, page).index_select(0, idx).cpu().numpy().reshape(-1) for t in src_layers]
        spec, layers_np, ident = oracle_sample(cfg, S, pool_np, args.layout)
        threads = os.cpu_count() or 1
        reps, el, want, moved = time_oracle(spec, layers_np, ident, S, args.cpu_seconds, threads, C)
        reps1, el1, _, _ = time_oracle(spec, layers_np, ident, S, args.cpu_seconds / 2, 1, C)
        cpu = {"value": moved * reps / el / GB, "unit": "GB/s", "cores": min(threads, S), "kind": "oracle",
               "sample": f"{S} of {n_chunks} chunks (evenly spaced), store then load, repeated {reps}x "
                         f"in {el:.1f} s on {threads} host threads",
               "single_thread_value": moved * reps1 / el1 / GB, "cpu_model": cpu_model()}
        verified = all(np.array_equal(chunks[c].numpy(), w) for c, w in zip(picks, want))

    k.kv_ctx_destroy(ctx)
    pool_info = host_pool.info()

    # the other workloads, each in its own buffers once the headline one's are freed
    extra = {}
    names = [n for n in args.configs.split(",") if n and n != "none"]
    if names:
        del chunks, src, dst, src_layers, dst_layers
        host_pool.close()
        torch.cuda.empty_cache()
        for name in names:
            if name == args.config:
                continue
            try:
                if name == "hybrid":
                    extra[name] = hybrid_leg(torch, k, synth, local)
                else:
                    extra[name] = config_leg(torch, k, synth, name, dev, local, link, sm_link, args.config_steps,
                                             2)
            except Exception as ex:  # a leg that cannot run here (memory) is reported, not fatal
                extra[name] = {"skipped": f"{type(ex).__name__}: {ex}"[:300]}
            torch.cuda.empty_cache()

    line = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u8",
        "data": "synthetic: bf16 ~N(0,1) KV from a fixed seed; seeded random-permutation block tables",
        "config": {"workload": workload_name(cfg, args.layout), "context_tokens": T, "layers": L, "kv_heads": H,
                   "head_dim": D, "kv_dtype": s["dtype"], "block_tokens": B, "chunk_tokens": C, "pool_blocks": N,
                   "page_layout": LAY,
                   "bytes_per_direction": X,
                   "l2": f"inputs larger than L2 ({X} bytes per direction); the destination pool is refilled "
                         f"with poison bytes before every step (a {L * layer_bytes}-byte write, which also "
                         f"flushes L2), outside the step's events",
                   "store_mode": k.MODE_NAMES[store_mode], "load_mode": k.MODE_NAMES[load_mode],
                   "parallelism": "one replica", "pinned_host_bytes": n_chunks * cb,
                   "host_alloc": host_alloc if host_pool.numa_node is None
                   else f"numa node {host_pool.numa_node}",
                   "host_pool": pool_info,
                   "pin_seconds": pin_seconds, "host_mem_available_at_start": avail},
        "restore_ms": span(restore_ms),
        "store_ms": span(store_ms),
        "host_link": host_link,
        "roofline": roofline,
        "hbm_roofline": hbm_roofline,
        "kernels": kern,
        "cpu_baseline": cpu,
        "verified_sample_vs_oracle": verified,
        "concurrent_replicas": concurrent,
        "tier_path": tier_leg,
        "streamed_cross_replica": streamed,
        "restore_after_idle": cold,
        "configs": extra,
        "e2e": e2e,
        "gpu_launches": stats["kernel_launches"],
        "memcpy_calls": stats["memcpy_calls"],
        "clocks": clock_info,
        "device": {"gpu": torch.cuda.get_device_name(dev),
                   "sms": torch.cuda.get_device_properties(dev).multi_processor_count,
                   "host_cpu": cpu_model(), "host_threads": os.cpu_count(),
                   "pinned_pool_numa_node": pool_info["numa_node"]},
    }
    print(json.dumps(line), flush=True)
    return 0


def main():
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
