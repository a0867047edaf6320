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
from gpu_util import POISON, device_pool, first_mismatch, host_layers, kvx, np_of, oracle_store, pinned_chunks
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
