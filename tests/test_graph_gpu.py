"""kv_store + kv_load captured into a CUDA graph and replayed.

The calls order their side-stream work with an event on the caller's stream
and a join back to it, which stream capture turns into graph edges; the
zero-copy mode allocates nothing per call.  A captured store/restore is
replayed twice with new KV written between the replays and each replay is
checked against the oracle.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import POISON, device_pool, first_mismatch, host_layers, kvx, np_of, oracle_load, oracle_store, pinned_chunks
from paper_2609_15021_gb300 import synth

pytestmark = pytest.mark.gpu


def test_store_restore_replayed_from_a_cuda_graph(orc):
    k = kvx()
    spec = oracle.PoolSpec(4, 64, 16, 8, 128, 2, oracle.HND)
    C, n_used = 256, 40
    T = n_used * 16 - 7
    src = device_pool(spec, host_layers(spec, 1))
    dst = device_pool(spec)
    ta = synth.permuted_table(64, n_used, 2)
    tb = synth.permuted_table(64, n_used, 3)
    ta_d, tb_d = torch.from_numpy(ta).cuda(), torch.from_numpy(tb).cuda()
    host = pinned_chunks(orc, spec, 0, T, C)
    ctx = k.kv_ctx_create(0)
    torch.cuda.synchronize()  # the poisoned pool was filled on the default stream
    try:
        s = torch.cuda.Stream()
        with torch.cuda.stream(s):  # warm up outside the capture
            k.kv_store(ctx, src, ta_d, 0, T, C, host)
            k.kv_load(ctx, dst, tb_d, 0, T, C, host)
        s.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s, capture_error_mode="thread_local"):
            k.kv_store(ctx, src, ta_d, 0, T, C, host)
            k.kv_load(ctx, dst, tb_d, 0, T, C, host)
        for seed in (10, 11):
            new = host_layers(spec, seed)
            for l, a in enumerate(new):
                src.layers[l].copy_(torch.from_numpy(a))
            for t in dst.layers:
                t.fill_(POISON)
            torch.cuda.synchronize()
            g.replay()
            torch.cuda.synchronize()
            want, _ = oracle_store(orc, spec, new, ta, 0, T, C)
            for h, w in zip(host, want):
                assert first_mismatch(np_of(h), w) is None, seed
            loaded, _ = oracle_load(orc, spec, [np.full(spec.layer_bytes, POISON, np.uint8)] * 4, tb, 0, T, C, want)
            for l in range(4):
                assert first_mismatch(np_of(dst.layers[l]), loaded[l]) is None, (seed, l)
        assert k.kv_get_device_error(ctx) == -1
    finally:
        k.kv_ctx_destroy(ctx)


def test_tier_calls_during_a_capture(orc):
    """Tier calls keep host bookkeeping, so one given a capturing stream is
    refused (KVX_EINVAL) and the capture goes on; calls without a stream
    (reserve, lookups) made while the thread captures leave the capture alone.
    The captured store is replayed, then committed outside the capture, and
    its bytes match the oracle."""
    k = kvx()
    spec = oracle.PoolSpec(4, 64, 16, 8, 128, 2, oracle.HND)
    C, n_used = 256, 32
    T = n_used * 16
    layers_np = host_layers(spec, 5)
    src = device_pool(spec, layers_np)
    ta = synth.permuted_table(64, n_used, 6)
    ta_d = torch.from_numpy(ta).cuda()
    keys = [901, 902]
    tier = k.KvTier(orc.chunk_bytes(spec, C), 4, shared_name=f"/kvx_graph_{__import__('os').getpid()}", create=True)
    ctx = k.kv_ctx_create(0)
    try:
        s = torch.cuda.Stream()
        slots = tier.reserve_many(keys)
        with torch.cuda.stream(s):  # warm up outside the capture
            k.kv_store(ctx, src, ta_d, 0, T, C, slots)
        s.synchronize()
        tier.reserve(903)                       # an entry with GPU work pending when the capture starts
        tier.commit(903, stream=s)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):     # the strictest capture mode: global
            k.kv_store(ctx, src, ta_d, 0, T, C, slots)
            for call in (lambda: tier.commit_many(keys, stream=s), lambda: tier.acquire(903, stream=s),
                         lambda: tier.release(903, stream=s)):
                with pytest.raises(k.KvxError) as e:
                    call()
                assert e.value.status == k.KVX_EINVAL
            assert tier.prefix_hits(keys) == 0  # host-side calls go on (with event queries) inside the capture
            tier.reserve(904)
        g.replay()
        tier.commit_many(keys, stream=s)
        s.synchronize()
        assert tier.prefix_hits(keys) == 2
        want, _ = oracle_store(orc, spec, layers_np, ta, 0, T, C)
        for c, key in enumerate(keys):
            got = tier.acquire(key, k.KVX_NO_STREAM)
            assert first_mismatch(np_of(got), want[c]) is None, c
            tier.release(key, k.KVX_NO_STREAM)
        assert k.kv_get_device_error(ctx) == -1
    finally:
        k.kv_ctx_destroy(ctx)
        tier.close()


def test_first_calls_of_a_context_inside_a_capture(orc):
    """A context's first transfer, or its first after more than 1 s, is when the
    library reads the chunks' host pages behind a host function on the stream.
    Made on a capturing stream, that read is skipped: nothing of it enters the
    graph (a replayed host function would wait on a job that no longer exists).
    The capture below is the new context's very first call, and a second one
    follows 1.1 s later; both graphs replay twice bit-exactly."""
    import time
    k = kvx()
    spec = oracle.PoolSpec(4, 64, 16, 8, 128, 2, oracle.HND)
    C, n_used = 256, 40
    T = n_used * 16 - 7
    src = device_pool(spec, host_layers(spec, 21))
    dst = device_pool(spec)
    ta = synth.permuted_table(64, n_used, 22)
    tb = synth.permuted_table(64, n_used, 23)
    ta_d, tb_d = torch.from_numpy(ta).cuda(), torch.from_numpy(tb).cuda()
    host = pinned_chunks(orc, spec, 0, T, C)
    ctx = k.kv_ctx_create(0)
    try:
        s = torch.cuda.Stream()
        torch.cuda.synchronize()
        graphs = []
        for pause in (0.0, 1.1):
            time.sleep(pause)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=s):   # global capture mode
                k.kv_store(ctx, src, ta_d, 0, T, C, host)
                k.kv_load(ctx, dst, tb_d, 0, T, C, host)
            graphs.append(g)
        for i, g in enumerate(graphs * 2):
            new = host_layers(spec, 30 + i)
            for l, a in enumerate(new):
                src.layers[l].copy_(torch.from_numpy(a))
            for t in dst.layers:
                t.fill_(POISON)
            torch.cuda.synchronize()
            g.replay()
            torch.cuda.synchronize()
            want, _ = oracle_store(orc, spec, new, ta, 0, T, C)
            for h, w in zip(host, want):
                assert first_mismatch(np_of(h), w) is None, i
            loaded, _ = oracle_load(orc, spec, [np.full(spec.layer_bytes, POISON, np.uint8)] * 4, tb, 0, T, C, want)
            for l in range(4):
                assert first_mismatch(np_of(dst.layers[l]), loaded[l]) is None, (i, l)
        assert k.kv_get_device_error(ctx) == -1
    finally:
        k.kv_ctx_destroy(ctx)
