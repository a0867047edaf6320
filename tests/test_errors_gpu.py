"""Argument errors on the GPU path: each bad call returns its documented status
before anything is enqueued, leaves every buffer as it was, and leaves the
context usable (the next valid call is bit-exact with the oracle).

Covers the checks only a device can make (memory kinds through
cudaPointerGetAttributes, pinned mappings) and the range and alignment rules
through the same entry points: kv_store, kv_load, kv_pack, kv_unpack,
kv_state_store, kv_state_load and kv_store_noalloc.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import POISON, device_pool, first_mismatch, host_layers, kvx, np_of, oracle_store, pinned_chunks
from paper_2609_15021_gb300 import synth

pytestmark = pytest.mark.gpu

SPEC = oracle.PoolSpec(2, 16, 16, 2, 64, 2, oracle.HND)
C, T = 64, 128  # two chunks of 64 tokens


@pytest.fixture(scope="module", params=[1, 2], ids=["staged", "zerocopy"])
def setup(request):
    k = kvx()
    src_np = host_layers(SPEC, 4321)
    src = device_pool(SPEC, src_np)
    dst = device_pool(SPEC)
    table = synth.permuted_table(SPEC.num_blocks, T // SPEC.block_tokens, 5)
    ctx = k.kv_ctx_create(0, store_mode=request.param, load_mode=request.param)
    yield k, ctx, src, src_np, dst, table
    k.kv_ctx_destroy(ctx)


def _untouched(k, ctx, chunks, dst):
    torch.cuda.synchronize()
    for i, c in enumerate(chunks):
        assert bool((c == POISON).all()), f"chunk {i} was written by a rejected call"
    for l, layer in enumerate(dst.layers):
        assert bool((layer == POISON).all()), f"pool layer {l} was written by a rejected call"
    assert k.kv_get_device_error(ctx) == -1


def _rejects(k, status, fn, *args, **kw):
    with pytest.raises(k.KvxError) as e:
        fn(*args, **kw)
    assert e.value.status == status, (e.value.status, status)


def test_memory_kinds_and_layout_rules_rejected_before_any_work(orc, setup):
    k, ctx, src, src_np, dst, table = setup
    tab = torch.from_numpy(table).cuda()
    chunks = pinned_chunks(orc, SPEC, 0, T, C)
    cb = orc.chunk_bytes(SPEC, C)
    pageable = [torch.full((cb,), POISON, dtype=torch.uint8) for _ in range(2)]
    on_device = [torch.full((cb,), POISON, dtype=torch.uint8, device="cuda") for _ in range(2)]
    shifted_buf = torch.full((cb + 16,), POISON, dtype=torch.uint8).pin_memory()
    shifted = [shifted_buf[8:8 + cb], chunks[1]]
    host_table = torch.from_numpy(table).pin_memory()
    host_layer_pool = k.KvPool([torch.full((SPEC.layer_bytes,), POISON, dtype=torch.uint8).pin_memory()
                                for _ in range(SPEC.num_layers)], SPEC.num_blocks, SPEC.block_tokens,
                               SPEC.num_heads, SPEC.head_dim, SPEC.elem_bytes)
    torch.cuda.synchronize()
    for fn, pool in ((k.kv_store, src), (k.kv_load, dst)):
        _rejects(k, k.KVX_ENOTPINNED, fn, ctx, pool, tab, 0, T, C, pageable)        # pageable host chunks
        _rejects(k, k.KVX_ENOTPINNED, fn, ctx, pool, tab, 0, T, C, on_device)       # device memory as host chunks
        _rejects(k, k.KVX_EALIGN, fn, ctx, pool, tab, 0, T, C, shifted)             # chunk not 16-byte aligned
        _rejects(k, k.KVX_EDEVICE, fn, ctx, pool, host_table, 0, T, C, chunks)      # table in host memory
        _rejects(k, k.KVX_EDEVICE, fn, ctx, host_layer_pool, tab, 0, T, C, chunks)  # pool layers in host memory
        _rejects(k, k.KVX_EALIGN, fn, ctx, pool, tab, 16, T, C, chunks)             # tok_begin % C != 0
        _rejects(k, k.KVX_EALIGN, fn, ctx, pool, tab, 0, T, 24, chunks)             # C % B != 0
        _rejects(k, k.KVX_ERANGE, fn, ctx, pool, tab, 0, T + 1, C, chunks + chunks)  # beyond the table
        _rejects(k, k.KVX_ERANGE, fn, ctx, pool, tab, 64, 0, C, chunks)             # tok_end < tok_begin
        _rejects(k, k.KVX_ERANGE, fn, ctx, pool, tab, 0, T, C, chunks[:1])          # too few chunks
    for fn, pool in ((k.kv_pack, src), (k.kv_unpack, dst)):
        _rejects(k, k.KVX_EDEVICE, fn, ctx, pool, tab, 0, T, C, chunks)             # pinned host as device chunks
        _rejects(k, k.KVX_EDEVICE, fn, ctx, pool, tab, 0, T, C, pageable)
    # rows that are not a multiple of 16 bytes (D = 4, bf16: 8-byte rows)
    narrow = k.KvPool([torch.zeros(16 * 2 * 2 * 16 * 8, dtype=torch.uint8, device="cuda")], 16, 16, 2, 4, 2)
    _rejects(k, k.KVX_EALIGN, k.kv_store, ctx, narrow, tab, 0, T, C, chunks)
    _untouched(k, ctx, chunks + on_device + [shifted_buf], dst)
    assert all(bool((p == POISON).all()) for p in pageable)
    # the context still works: a valid store is bit-exact with the oracle
    k.kv_store(ctx, src, tab, 0, T, C, chunks)
    torch.cuda.synchronize()
    want, _ = oracle_store(orc, SPEC, src_np, table, 0, T, C)
    for c, w in zip(chunks, want):
        assert first_mismatch(np_of(c), w) is None
    assert k.kv_get_device_error(ctx) == -1


def test_state_copy_arguments_rejected_before_any_work(setup):
    k, ctx, _, _, _, _ = setup
    L, slots, sb = 3, 2, 4096
    layers = [torch.full((slots * sb,), POISON, dtype=torch.uint8, device="cuda") for _ in range(L)]
    obj = torch.full((L * sb,), POISON, dtype=torch.uint8).pin_memory()
    pageable = torch.full((L * sb,), POISON, dtype=torch.uint8)
    host_layers_ = [torch.full((slots * sb,), POISON, dtype=torch.uint8).pin_memory() for _ in range(L)]
    torch.cuda.synchronize()
    for fn in (k.kv_state_store, k.kv_state_load):
        _rejects(k, k.KVX_ERANGE, fn, ctx, layers, slots, sb, slots, obj)         # slot beyond the pools
        _rejects(k, k.KVX_ERANGE, fn, ctx, layers, slots, sb, -1, obj)
        _rejects(k, k.KVX_EALIGN, fn, ctx, layers, slots, sb - 8, 0, obj)          # slot bytes % 16 != 0
        _rejects(k, k.KVX_ENOTPINNED, fn, ctx, layers, slots, sb, 0, pageable)   # pageable snapshot
        _rejects(k, k.KVX_EDEVICE, fn, ctx, host_layers_, slots, sb, 0, obj)     # state pools in host memory
        _rejects(k, k.KVX_EALIGN, fn, ctx, layers, slots, sb, 0, obj[8:].data_ptr())  # snapshot not aligned
    torch.cuda.synchronize()
    assert all(bool((t == POISON).all()) for t in layers + host_layers_ + [obj, pageable])
    k.kv_state_store(ctx, layers, slots, sb, 1, obj)
    torch.cuda.synchronize()
    assert bool((obj == POISON).all())  # the pools hold poison too: a valid copy of them


def test_allocation_free_store_rejects_bad_memory(orc, setup):
    k, _, src, _, _, table = setup
    tab = torch.from_numpy(table).cuda()
    cb = orc.chunk_bytes(SPEC, C)
    pageable = [torch.full((cb,), POISON, dtype=torch.uint8) for _ in range(2)]
    on_device = [torch.full((cb,), POISON, dtype=torch.uint8, device="cuda") for _ in range(2)]
    torch.cuda.synchronize()
    _rejects(k, k.KVX_ENOTPINNED, k.kv_store_noalloc, src, tab, 0, T, C, pageable)
    _rejects(k, k.KVX_ENOTPINNED, k.kv_store_noalloc, src, tab, 0, T, C, on_device)
    _rejects(k, k.KVX_EDEVICE, k.kv_store_noalloc, src, torch.from_numpy(table).pin_memory(), 0, T, C,
             pinned_chunks(orc, SPEC, 0, T, C))
    torch.cuda.synchronize()
    assert all(bool((c == POISON).all()) for c in pageable + on_device)


def test_modes_pool_info_and_foreign_pointers(orc):
    """KVX_MODE_AUTO resolves to zero-copy both ways (the measured default);
    explicit and mixed modes stay as asked, and the counters show which path
    ran (copies only in staged mode).  kv_host_pool_info knows the start of a
    library pool only; kv_host_free ignores NULL and memory it did not
    allocate."""
    import ctypes
    k = kvx()
    for asked, want in (((0, 0), (2, 2)), ((1, 1), (1, 1)), ((1, 2), (1, 2)), ((2, 1), (2, 1))):
        ctx = k.kv_ctx_create(0, store_mode=asked[0], load_mode=asked[1])
        try:
            assert k.kv_ctx_modes(ctx) == want
            src_np = host_layers(SPEC, 99)
            src, dst = device_pool(SPEC, src_np), device_pool(SPEC)
            tab = torch.from_numpy(synth.permuted_table(SPEC.num_blocks, T // SPEC.block_tokens, 3)).cuda()
            chunks = pinned_chunks(orc, SPEC, 0, T, C)
            torch.cuda.synchronize()
            k.kv_store(ctx, src, tab, 0, T, C, chunks)
            k.kv_load(ctx, dst, tab, 0, T, C, chunks)
            torch.cuda.synchronize()
            st = k.kv_ctx_stats(ctx)
            assert st["kernel_launches"] >= 2
            assert (st["memcpy_calls"] > 0) == (1 in want), (asked, st)
            for l in range(SPEC.num_layers):  # restored through the same table: the pages it names
                idx = tab.long()
                page = SPEC.layer_bytes // SPEC.num_blocks
                assert torch.equal(src.layers[l].view(-1, page)[idx], dst.layers[l].view(-1, page)[idx])
        finally:
            k.kv_ctx_destroy(ctx)
    buf = k.HostBuffer(3 << 20)
    try:
        assert buf.info()["bytes"] == 3 << 20
        with pytest.raises(k.KvxError) as e:
            k.kv_host_pool_info(buf.ptr + 4096)          # inside a pool, not its start
        assert e.value.status == k.KVX_ENOENT
        foreign = torch.full((1 << 20,), 7, dtype=torch.uint8).pin_memory()
        with pytest.raises(k.KvxError) as e:
            k.kv_host_pool_info(foreign.data_ptr())      # pinned, but not the library's
        assert e.value.status == k.KVX_ENOENT
        k._lib.kv_host_free(None)
        k._lib.kv_host_free(ctypes.c_void_p(foreign.data_ptr()))   # ignored: not the library's
        assert int(foreign[-1]) == 7
        d = torch.empty(1 << 20, dtype=torch.uint8, device="cuda")
        d.copy_(foreign, non_blocking=True)                       # still pinned and usable
        torch.cuda.synchronize()
        assert int(d[0]) == 7
    finally:
        buf.close()
