"""kv_store_noalloc: the store for callers that cannot allocate device memory.

Such callers (an engine whose pool owns all free GPU memory, or code that must
not let cudaMalloc / cudaFree synchronise the device mid-pipeline) cannot
create a kvx_ctx, because a context allocates a staging ring, streams and
events.  kv_store_noalloc packs into a static device array instead.  These
tests call it through the C ABI and check its chunks byte for byte against
kv_store's on the same inputs, on two calls in a row (the array keeps the
previous call's bytes), plus the size limit and the bad-entry report.  Two
tests run in a fresh process of their own: after the set-up call (an empty
range), calls leave the GPU's free memory and torch's reserved memory exactly
as they were; and a call in a second, driver-API context (where the array has
another address) stores the same bytes as calls in the primary context before
and after it.

This file is collected last so that a stop-at-first-failure run has already
run every other test; it also passes alone in a fresh process.
"""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

import oracle
from gpu_util import POISON, device_pool, first_mismatch, host_layers, kvx, np_of, oracle_store, pinned_chunks
from paper_2609_15021_gb300 import synth

pytestmark = pytest.mark.gpu

# (L, N, B, H, D, e, layout, pages used, C, first chunk, t1 short by)
CALLS = [
    (62, 48, 16, 8, 128, 2, oracle.HND, 40, 256, 0, 3),   # 62 MiB chunks: two batches, one chunk split
    (2, 64, 16, 2, 64, 2, oracle.NHD, 32, 256, 1, 0),     # small chunks, non-zero start
]


def _expected_via_kv_store(orc, pool, table_d, t0, t1, C, spec):
    k = kvx()
    ctx = k.kv_ctx_create(0)
    try:
        host = pinned_chunks(orc, spec, t0, t1, C)
        k.kv_store(ctx, pool, table_d, t0, t1, C, host)
        torch.cuda.synchronize()
    finally:
        k.kv_ctx_destroy(ctx)
    return [np_of(h) for h in host]


def test_noalloc_store_matches_kv_store_twice(orc):
    k = kvx()
    for rnd in range(2):  # the same two calls again: the array now holds older bytes
        for n_call, case in enumerate(CALLS):
            L, N, B, H, D, e, layout, n_used, C, c0, short = case
            spec = oracle.PoolSpec(L, N, B, H, D, e, layout)
            src_np = host_layers(spec, seed=300 + n_call)
            pool = device_pool(spec, src_np)
            table = synth.permuted_table(N, n_used, seed=40 + n_call)
            table_d = torch.from_numpy(table).cuda()
            t0, t1 = c0 * C, n_used * B - short
            want = _expected_via_kv_store(orc, pool, table_d, t0, t1, C, spec)
            extra = 32
            host = pinned_chunks(orc, spec, t0, t1, C, extra=extra)
            stream = torch.cuda.Stream()
            k.kv_store_noalloc(pool, table_d, t0, t1, C, host, stream=stream)
            stream.synchronize()
            for i, (h, w) in enumerate(zip(host, want)):
                got = np_of(h)
                assert first_mismatch(got[:-extra], w) is None, (rnd, n_call, i)
                assert np.all(got[-extra:] == POISON), (rnd, n_call, i)
            ref, _ = oracle_store(orc, spec, src_np, table, t0, t1, C)
            for h, r in zip(host, ref):
                assert first_mismatch(np_of(h)[:-extra], r) is None


def test_noalloc_reports_bad_entries(orc):
    k = kvx()
    spec = oracle.PoolSpec(2, 16, 16, 2, 64, 2, oracle.HND)
    src_np = host_layers(spec, seed=8)
    pool = device_pool(spec, src_np)
    table = synth.permuted_table(16, 12, seed=9)
    table[7] = 99
    table_d = torch.from_numpy(table).cuda()
    err = torch.full((1,), np.iinfo(np.int64).max, dtype=torch.int64, device="cuda")
    host = pinned_chunks(orc, spec, 0, 192, 64)
    k.kv_store_noalloc(pool, table_d, 0, 192, 64, host, dev_first_bad_block=err)
    torch.cuda.synchronize()
    assert int(err.item()) == 7
    want, bad = oracle_store(orc, spec, src_np, table, 0, 192, 64)
    assert bad == 7
    for h, w in zip(host, want):
        assert first_mismatch(np_of(h), w) is None


def test_noalloc_rejects_layers_larger_than_the_array(orc):
    k = kvx()
    # one layer of a 32768-token chunk of 8 heads x 256-byte rows is 128 MiB > 64 MiB
    spec = oracle.PoolSpec(1, 2048, 16, 8, 128, 2, oracle.HND)
    pool = device_pool(spec, fill=1)
    table_d = torch.arange(2048, dtype=torch.int32, device="cuda")
    host = [torch.empty(orc.chunk_bytes(spec, 32768), dtype=torch.uint8).pin_memory()]
    with pytest.raises(k.KvxError) as ex:
        k.kv_store_noalloc(pool, table_d, 0, 32768, 32768, host)
    assert ex.value.status == k.KVX_ERANGE
    assert "static staging array" in str(ex.value)


HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


def _run_fresh(body: str, marker: str):
    """Run one of the bodies below in a new Python process (nothing loaded yet)."""
    code = (f"import sys; sys.path[:0] = [{HERE!r}, {ROOT!r}]; import test_zz_no_alloc as t; t.{body}()")
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=300, cwd=HERE)
    assert r.returncode == 0 and marker in r.stdout, r.stdout[-3000:] + r.stderr[-3000:]


def _allocation_free_body():
    k = kvx()
    orc = oracle.c_oracle()
    # 62 MiB chunks: every call packs two batches and splits one chunk
    spec = oracle.PoolSpec(62, 48, 16, 8, 128, 2, oracle.HND)
    src_np = host_layers(spec, seed=700)
    pool = device_pool(spec, src_np)
    table = synth.permuted_table(48, 40, seed=701)
    table_d = torch.from_numpy(table).cuda()
    t1 = 40 * 16 - 5
    host = pinned_chunks(orc, spec, 0, t1, 256)
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()
    free_before = torch.cuda.mem_get_info()[0]
    k.kv_store_noalloc(pool, table_d, 0, 0, 256, host, stream=stream)  # set-up only: empty range
    torch.cuda.synchronize()
    free0, reserved0 = torch.cuda.mem_get_info()[0], torch.cuda.memory_reserved()
    for _ in range(2):
        k.kv_store_noalloc(pool, table_d, 0, t1, 256, host, stream=stream)
        stream.synchronize()
        free, reserved = torch.cuda.mem_get_info()[0], torch.cuda.memory_reserved()
        assert free == free0, f"free GPU memory moved from {free0} to {free}"
        assert reserved == reserved0
    want, _ = oracle_store(orc, spec, src_np, table, 0, t1, 256)
    for h, w in zip(host, want):
        assert first_mismatch(np_of(h), w) is None
    print(f"NOALLOC_FRESH_OK set-up took {free_before - free0} bytes of GPU memory; later calls none")


def test_noalloc_allocates_nothing_after_the_setup_call():
    _run_fresh("_allocation_free_body", "NOALLOC_FRESH_OK")


def _driver_context_body():
    import ctypes

    k = kvx()
    orc = oracle.c_oracle()
    cu = ctypes.CDLL("libcuda.so.1")
    vp, u64 = ctypes.c_void_p, ctypes.c_uint64

    def ok(rc, what):
        assert rc == 0, f"{what}: CUresult {rc}"

    spec = oracle.PoolSpec(2, 64, 16, 2, 64, 2, oracle.NHD)
    src_np = host_layers(spec, seed=710)
    table = synth.permuted_table(64, 32, seed=711)
    t0, t1, C = 256, 32 * 16 - 7, 256
    want, _ = oracle_store(orc, spec, src_np, table, t0, t1, C)

    def primary_call():
        pool = device_pool(spec, src_np)
        host = pinned_chunks(orc, spec, t0, t1, C)
        k.kv_store_noalloc(pool, torch.from_numpy(table).cuda(), t0, t1, C, host)
        torch.cuda.synchronize()
        return [np_of(h) for h in host]

    first = primary_call()
    # a second context on the same device, current on this thread; its memory
    # comes from the driver API (torch stays in the primary context)
    dev = ctypes.c_int()
    ok(cu.cuDeviceGet(ctypes.byref(dev), 0), "cuDeviceGet")
    ctx2 = vp()
    ok(cu.cuCtxCreate_v4(ctypes.byref(ctx2), None, 0, dev), "cuCtxCreate")
    bufs, pinned = [], []
    try:
        def dalloc(n):
            d = u64()
            ok(cu.cuMemAlloc_v2(ctypes.byref(d), ctypes.c_size_t(n)), "cuMemAlloc")
            bufs.append(d)
            return d.value

        layers = []
        for a in src_np:
            d = dalloc(a.nbytes)
            ok(cu.cuMemcpyHtoD_v2(u64(d), a.ctypes.data_as(vp), ctypes.c_size_t(a.nbytes)), "cuMemcpyHtoD")
            layers.append(d)
        tab = np.ascontiguousarray(table, np.int32)
        td = dalloc(tab.nbytes)
        ok(cu.cuMemcpyHtoD_v2(u64(td), tab.ctypes.data_as(vp), ctypes.c_size_t(tab.nbytes)), "cuMemcpyHtoD")
        sizes = [orc.chunk_bytes(spec, n) for n in oracle.chunk_tokens_of(t0, t1, C)]
        for n in sizes:
            h = vp()
            ok(cu.cuMemHostAlloc(ctypes.byref(h), ctypes.c_size_t(n), 1), "cuMemHostAlloc")  # portable
            ctypes.memset(h, POISON, n)
            pinned.append(h)
        pool2 = k.KvPool(layers, spec.num_blocks, spec.block_tokens, spec.num_heads, spec.head_dim,
                         spec.elem_bytes, spec.layout)
        # stream 0: the legacy default stream of the context current now
        k.kv_store_noalloc(pool2, td, t0, t1, C, [h.value for h in pinned], stream=0, table_len=len(tab))
        ok(cu.cuCtxSynchronize(), "cuCtxSynchronize")
        second = [np.frombuffer(ctypes.string_at(h.value, n), np.uint8).copy() for h, n in zip(pinned, sizes)]
    finally:
        for h in pinned:
            cu.cuMemFreeHost(h)
        for d in bufs:
            cu.cuMemFree_v2(d)
        popped = vp()
        cu.cuCtxPopCurrent_v2(ctypes.byref(popped))
        cu.cuCtxDestroy_v2(ctx2)
    third = primary_call()
    for got in (first, second, third):
        for g, w in zip(got, want):
            assert first_mismatch(g, w) is None
    print("NOALLOC_CONTEXTS_OK")


def test_noalloc_after_a_context_change():
    _run_fresh("_driver_context_body", "NOALLOC_CONTEXTS_OK")
