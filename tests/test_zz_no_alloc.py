"""kv_store_noalloc: the store for callers that cannot allocate device memory.

Such callers (an engine whose pool owns all free GPU memory, or code that must
not let cudaMalloc / cudaFree synchronise the device mid-pipeline) cannot
create a kvx_ctx, because a context allocates a staging ring, streams and
events.  kv_store_noalloc packs into a static device array instead.  These
tests call it through the C ABI and check its chunks byte for byte against
kv_store's on the same inputs, on two calls in a row (the array keeps the
previous call's bytes), plus the size limit and the bad-entry report.

This file is collected last so that a stop-at-first-failure run has already
run every other test; it also passes alone in a fresh process.
"""
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
