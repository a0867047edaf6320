"""Failure handling with host-side fault injection (no GPU fault is produced).

A CUDA call failing in the middle of a transfer must return KVX_ECUDA naming
the call, leave the caller's stream ordered after whatever was enqueued (so a
synchronise returns), and leave the context usable: the next transfer is
bit-exact.  A pinned-pool allocation failure must raise, never fall back to
pageable memory (paper Sec. 3.3).
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import (POISON, device_pool, first_mismatch, host_layers, kvx, np_of, oracle_load, oracle_store,
                      pinned_chunks)
from paper_2609_15021_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def disarm():
    yield
    kvx().kv_fault_inject(None)


# (mode, point, after): the first, or the second, launch of a 3-launch zero-copy store
# failing (zero-copy moves run on the caller's stream: no event); a staged copy failing
# after a few copies; a staged launch failing; the staged pipeline's ordering event failing
CASES = [(2, "launch", 1), (2, "launch", 0), (1, "memcpy", 3), (1, "launch", 2), (1, "event", 0)]


@pytest.mark.parametrize("mode,point,after", CASES)
def test_failure_mid_transfer_then_recovery(orc, mode, point, after):
    k = kvx()
    spec = oracle.PoolSpec(1, 300, 1, 1, 8, 2, oracle.HND)   # 150 two-token chunks: 3 zero-copy launches
    src_np = host_layers(spec, 31)
    src = device_pool(spec, src_np)
    table = synth.permuted_table(300, 300, 9)
    table_d = torch.from_numpy(table).cuda()
    ctx = k.kv_ctx_create(0, store_mode=mode, load_mode=mode, staging_slot_bytes=4096)
    try:
        host = pinned_chunks(orc, spec, 0, 300, 2)
        s = torch.cuda.Stream()
        k.kv_fault_inject(point, after)
        with pytest.raises(k.KvxError) as e:
            k.kv_store(ctx, src, table_d, 0, 300, 2, host, stream=s)
        assert e.value.status == k.KVX_ECUDA
        assert "kvxfer.cu" in str(e.value)
        s.synchronize()                       # the stream was joined to what had been enqueued
        host2 = pinned_chunks(orc, spec, 0, 300, 2)
        k.kv_store(ctx, src, table_d, 0, 300, 2, host2, stream=s)
        s.synchronize()
        want, _ = oracle_store(orc, spec, src_np, table, 0, 300, 2)
        for h, w in zip(host2, want):
            assert first_mismatch(np_of(h), w) is None
        assert k.kv_get_device_error(ctx) == -1
    finally:
        k.kv_ctx_destroy(ctx)


def test_pinned_allocation_failure_raises():
    k = kvx()
    k.kv_fault_inject("host_alloc", 0)
    with pytest.raises(k.KvxError) as e:
        k.HostBuffer(1 << 20)
    assert e.value.status == k.KVX_ENOMEM
    buf = k.HostBuffer(1 << 20)             # the next allocation is made normally
    assert buf.tensor.numel() == 1 << 20
    buf.close()


def test_unknown_fault_point_rejected():
    k = kvx()
    with pytest.raises(k.KvxError) as e:
        k.kv_fault_inject("nowhere", 0)
    assert e.value.status == k.KVX_EINVAL


# (layout, context flags, CTA cap): the tensor-map engine (HND) and the row/flat
# bulk-copy engine (NHD under KVX_FLAG_DEVICE_TMA), each with one unit per CTA
# (a single shared-memory stage) and with a capped grid (a ring of stages, so
# loads for later units are in flight when the first unit's wait runs out)
TMA_CASES = [(oracle.HND, 0, 0), (oracle.HND, 0, 7), (oracle.NHD, 0x4, 0), (oracle.NHD, 0x4, 7)]


@pytest.mark.parametrize("direction", ["pack", "unpack"])
@pytest.mark.parametrize("layout,flags,max_ctas", TMA_CASES)
def test_tma_wait_runs_out_then_recovery(orc, direction, layout, flags, max_ctas):
    """Fault point "tma_wait": the first unit's stage is armed for bytes no copy
    brings, so its bounded wait (2e6 cycles here) runs out with nothing in flight
    for it.  The launch returns, kv_get_device_error reports KVX_ETIMEOUT, that
    unit's bytes are untouched, and the next transfer on the same context is
    bit-exact with the oracle."""
    k = kvx()
    spec = oracle.PoolSpec(2, 64, 16, 8, 128, 2, layout)
    C, T = 256, 32 * 16
    src_np = host_layers(spec, 61)
    table = synth.permuted_table(64, 32, 62)
    table_d = torch.from_numpy(table).cuda()
    want, _ = oracle_store(orc, spec, src_np, table, 0, T, C)
    half = spec.block_tokens * spec.num_heads * spec.head_dim * spec.elem_bytes  # unit 0: layer 0, K, first page
    page_bytes = 2 * half
    ctx = k.kv_ctx_create(0, flags=flags, max_ctas=max_ctas, wait_cycles=2_000_000)
    try:
        s = torch.cuda.Stream()
        if direction == "pack":
            src = device_pool(spec, src_np)
            out = [torch.full((w.size,), POISON, dtype=torch.uint8, device="cuda") for w in want]
            run = lambda: k.kv_pack(ctx, src, table_d, 0, T, C, out, stream=s)
        else:
            chunks = [torch.from_numpy(w).cuda() for w in want]
            dst = device_pool(spec)
            run = lambda: k.kv_unpack(ctx, dst, table_d, 0, T, C, chunks, stream=s)
        torch.cuda.synchronize()  # buffers above were filled on the default stream
        k.kv_fault_inject("tma_wait", 0)
        run()
        s.synchronize()
        with pytest.raises(k.KvxError) as e:
            k.kv_get_device_error(ctx)
        assert e.value.status == k.KVX_ETIMEOUT
        assert k.kv_get_device_error(ctx) == -1      # the query cleared the record
        if direction == "pack":
            got = [np_of(o) for o in out]
            assert np.all(got[0][:half] == POISON)   # the stalled unit was not moved
            if max_ctas == 0:                        # one unit per CTA: every other unit was
                w0 = want[0].copy()
                w0[:half] = POISON
                assert first_mismatch(got[0], w0) is None
                assert first_mismatch(got[1], want[1]) is None
        else:
            layer0 = np_of(dst.layers[0])
            p0 = int(table[0]) * page_bytes
            assert np.all(layer0[p0:p0 + half] == POISON)
            if max_ctas == 0:
                poisoned = [np.full(spec.layer_bytes, POISON, np.uint8) for _ in range(2)]
                want_l, _ = oracle_load(orc, spec, poisoned, table, 0, T, C, want)
                want_l[0][p0:p0 + half] = POISON
                for l in range(2):
                    assert first_mismatch(np_of(dst.layers[l]), want_l[l]) is None
        # the fault point fired once: the next transfer is whole and bit-exact
        run()
        s.synchronize()
        assert k.kv_get_device_error(ctx) == -1
        if direction == "pack":
            for o, w in zip(out, want):
                assert first_mismatch(np_of(o), w) is None
        else:
            poisoned = [np.full(spec.layer_bytes, POISON, np.uint8) for _ in range(2)]
            want_l, _ = oracle_load(orc, spec, poisoned, table, 0, T, C, want)
            for l in range(2):
                assert first_mismatch(np_of(dst.layers[l]), want_l[l]) is None
    finally:
        k.kv_ctx_destroy(ctx)
