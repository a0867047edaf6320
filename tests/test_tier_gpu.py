"""The shared host tier on the GPU: a replica stores chunks into tier slots on
its stream; another replica, on another stream and with no host
synchronisation in between, restores them -- ordered only by the tier's
commit events (paper Sec. 3.2: every copy waits for the producer on the
current stream).  A producer delayed by ~10^8 SM cycles must not be
overtaken.  Slots still being read by in-flight work must not be evicted.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import POISON, device_pool, first_mismatch, host_layers, kvx, np_of, oracle_load, oracle_store
from paper_2609_15021_gb300 import probe, synth

pytestmark = pytest.mark.gpu

DELAY = 10 ** 8


@pytest.mark.parametrize("commit", ["per_key", "many"])
def test_store_then_restore_across_streams_through_the_tier(orc, commit):
    """commit="many": one kv_store of every chunk into its slot and one
    kv_tier_commit_many, whose entries share one event; the reader takes them
    with one kv_tier_acquire_many, one kv_load and one kv_tier_release_many."""
    k = kvx()
    spec = oracle.PoolSpec(4, 64, 16, 8, 128, 2, oracle.HND)
    C, n_used = 256, 48
    T = n_used * 16
    stale_np = host_layers(spec, 1)
    final_np = host_layers(spec, 2)
    pool_a = device_pool(spec, stale_np)
    final_dev = [torch.from_numpy(a).cuda() for a in final_np]
    pool_b = device_pool(spec)
    ta = synth.permuted_table(64, n_used, 3)
    tb = synth.permuted_table(64, n_used, 4)
    tokens = synth.rng(5).integers(0, 150000, size=T).astype(np.int32)
    keys = k.kv_chunk_keys(tokens, C, salt=314159)
    cb = orc.chunk_bytes(spec, C)
    tier = k.KvTier(cb, 8)
    ctx = k.kv_ctx_create(0)
    s_a, s_b = torch.cuda.Stream(), torch.cuda.Stream()
    try:
        torch.cuda.synchronize()
        # replica A: delayed producer writes the final KV, then each chunk is stored into a slot
        for l in range(spec.num_layers):
            probe.kvx_probe_delayed_copy(pool_a.layers[l], final_dev[l], spec.layer_bytes, DELAY if l == 0 else 0, s_a)
        ta_d = torch.from_numpy(ta).cuda()
        if commit == "many":
            slots = tier.reserve_many(keys)
            k.kv_store(ctx, pool_a, ta_d, 0, T, C, slots, stream=s_a)
            tier.commit_many(keys, stream=s_a)
        else:
            for c, key in enumerate(keys):
                slot = tier.reserve(key)
                k.kv_store(ctx, pool_a, ta_d, c * C, (c + 1) * C, C, [slot], stream=s_a)
                tier.commit(key, stream=s_a)
        # replica B, its own stream, no host synchronisation: ordered by the commit events
        assert tier.prefix_hits(keys) == len(keys)
        tb_d = torch.from_numpy(tb).cuda()
        if commit == "many":
            slots = tier.acquire_many(keys, stream=s_b)
            k.kv_load(ctx, pool_b, tb_d, 0, T, C, slots, stream=s_b)
            tier.release_many(keys, stream=s_b)
        else:
            for c, key in enumerate(keys):
                slot = tier.acquire(key, stream=s_b)
                k.kv_load(ctx, pool_b, tb_d, c * C, (c + 1) * C, C, [slot], stream=s_b)
                tier.release(key, stream=s_b)
        s_b.synchronize()
        s_a.synchronize()
        want, _ = oracle_store(orc, spec, final_np, ta, 0, T, C)
        loaded, _ = oracle_load(orc, spec, [np.full(spec.layer_bytes, POISON, np.uint8)] * spec.num_layers,
                                tb, 0, T, C, want)
        for l in range(spec.num_layers):
            assert first_mismatch(np_of(pool_b.layers[l]), loaded[l]) is None, l
        for c, key in enumerate(keys):
            slot = tier.acquire(key, stream=k.KVX_NO_STREAM)
            assert first_mismatch(np_of(slot), want[c]) is None, c
            tier.release(key, stream=k.KVX_NO_STREAM)
        tier.poll()
        st = tier.stats()
        assert st["pinned"] == 0 and st["entries"] == len(keys)
    finally:
        k.kv_ctx_destroy(ctx)
        tier.close()


def test_slots_in_use_by_the_gpu_are_not_evicted(orc):
    k = kvx()
    spec = oracle.PoolSpec(2, 16, 16, 2, 64, 2, oracle.HND)
    C = 64
    src_np = host_layers(spec, 7)
    src = device_pool(spec, src_np)
    dst = device_pool(spec)
    table = torch.from_numpy(synth.permuted_table(16, 8, 8)).cuda()
    cb = orc.chunk_bytes(spec, C)
    tier = k.KvTier(cb, 2)
    ctx = k.kv_ctx_create(0)
    torch.cuda.synchronize()  # the poisoned pool was filled on the default stream
    s = torch.cuda.Stream()
    busy = torch.empty(1 << 20, dtype=torch.uint8, device="cuda")
    try:
        for key, c in ((101, 0), (102, 1)):
            slot = tier.reserve(key)
            k.kv_store(ctx, src, table, c * C, (c + 1) * C, C, [slot], stream=s)
            tier.commit(key, stream=s)
        s.synchronize()
        # readers enqueue restores behind a long delay and release at once (host side)
        probe.kvx_probe_delayed_copy(busy, busy, busy.numel(), DELAY, s)
        for key, c in ((101, 0), (102, 1)):
            slot = tier.acquire(key, stream=s)
            k.kv_load(ctx, dst, table, c * C, (c + 1) * C, C, [slot], stream=s)
            tier.release(key, stream=s)
        with pytest.raises(k.KvxError) as e:   # both slots are still being read by queued work
            tier.reserve(103)
        assert e.value.status == k.KVX_ENOMEM
        s.synchronize()
        tier.reserve(103)                      # the work finished: the LRU slot may go
        tier.commit(103, stream=k.KVX_NO_STREAM)
        want, _ = oracle_store(orc, spec, src_np, table.cpu().numpy(), 0, 2 * C, C)
        loaded, _ = oracle_load(orc, spec, [np.full(spec.layer_bytes, POISON, np.uint8)] * 2,
                                table.cpu().numpy(), 0, 2 * C, C, want)
        for l in range(2):
            assert first_mismatch(np_of(dst.layers[l]), loaded[l]) is None
    finally:
        k.kv_ctx_destroy(ctx)
        tier.close()
