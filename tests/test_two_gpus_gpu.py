"""Store on one GPU, restore on another, through one host pool (paper Sec. 2,
Fig. 1: replicas on separate GPUs share one pinned RAM tier).

Two forms, both checked byte for byte against the oracle:
* one process, two contexts: a context on device 0 stores a context into a
  kv_host_alloc pool (page-locked, portable to every device, mapped), a
  context on device 1 restores those chunks into its own pool;
* two processes, one GPU each, sharing a tier in POSIX shared memory: the
  process on device 0 stores and commits on its stream (the GPU publishes the
  commits), the process on device 1 waits until the keys are readable,
  acquires them on its stream and restores them.
Both need two GPUs and are skipped with fewer.
"""
import multiprocessing as mp
import os

import numpy as np
import pytest
import torch

import oracle
from gpu_util import POISON, first_mismatch, host_layers, kvx, np_of, oracle_load, oracle_store
from paper_2609_15021_gb300 import synth

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(torch.cuda.device_count() < 2, reason="needs two GPUs")]

SPEC = oracle.PoolSpec(4, 96, 16, 8, 128, 2, oracle.HND)
C, N_USED = 256, 72
T = N_USED * 16 - 9


def _pool_on(device, layers_np=None):
    k = kvx()
    dev = torch.device("cuda", device)
    if layers_np is None:
        layers = [torch.full((SPEC.layer_bytes,), POISON, dtype=torch.uint8, device=dev) for _ in range(SPEC.num_layers)]
    else:
        layers = [torch.from_numpy(a).to(dev) for a in layers_np]
    return k.KvPool(layers, SPEC.num_blocks, SPEC.block_tokens, SPEC.num_heads, SPEC.head_dim, SPEC.elem_bytes)


def test_store_on_gpu0_restore_on_gpu1_through_one_pinned_pool(orc):
    k = kvx()
    src_np = host_layers(SPEC, 901)
    ta, tb = synth.permuted_table(96, N_USED, 902), synth.permuted_table(96, N_USED, 903)
    sizes = [orc.chunk_bytes(SPEC, n) for n in oracle.chunk_tokens_of(0, T, C)]
    pool = k.HostBuffer(sum(sizes))
    offs = np.cumsum([0] + sizes)
    chunks = [pool.tensor[offs[i]:offs[i + 1]] for i in range(len(sizes))]
    pool.tensor.fill_(POISON)
    ctx0, ctx1 = k.kv_ctx_create(0), k.kv_ctx_create(1)
    try:
        src = _pool_on(0, src_np)
        dst = _pool_on(1)
        s0 = torch.cuda.Stream(device=0)
        s1 = torch.cuda.Stream(device=1)
        k.kv_store(ctx0, src, torch.from_numpy(ta).to("cuda:0"), 0, T, C, chunks, stream=s0)
        s0.synchronize()                    # the store is complete before the other GPU reads the pool
        k.kv_load(ctx1, dst, torch.from_numpy(tb).to("cuda:1"), 0, T, C, chunks, stream=s1)
        s1.synchronize()
        assert k.kv_get_device_error(ctx0) == -1 and k.kv_get_device_error(ctx1) == -1
        want, _ = oracle_store(orc, SPEC, src_np, ta, 0, T, C)
        for c, w in zip(chunks, want):
            assert first_mismatch(np_of(c), w) is None
        want_l, _ = oracle_load(orc, SPEC, [np.full(SPEC.layer_bytes, POISON, np.uint8)] * SPEC.num_layers,
                                tb, 0, T, C, want)
        for l in range(SPEC.num_layers):
            assert first_mismatch(np_of(dst.layers[l]), want_l[l]) is None, l
    finally:
        k.kv_ctx_destroy(ctx0)
        k.kv_ctx_destroy(ctx1)
        del chunks
        pool.close()


def _reader_on_gpu1(name, keys, q):
    """Child process on device 1: wait for the keys, acquire them on its stream,
    restore into its own pool, and send the pool bytes back."""
    try:  # a spawned child gets the parent's sys.path, so this module and its helpers import here
        import torch

        from paper_2609_15021_gb300 import kvxfer as k
        torch.cuda.set_device(1)
        tier = k.KvTier(shared_name=name)
        tier.wait(keys, timeout_s=120)   # until the other GPU has published the commits
        ctx = k.kv_ctx_create(1)
        dst = _pool_on(1)
        s = torch.cuda.Stream(device=1)
        tb = torch.from_numpy(synth.permuted_table(96, N_USED, 903)).to("cuda:1")
        slots = tier.acquire_many(keys, stream=s)
        k.kv_load(ctx, dst, tb, 0, T, C, slots, stream=s)
        tier.release_many(keys, stream=s)
        s.synchronize()
        assert k.kv_get_device_error(ctx) == -1
        q.put([np_of(l) for l in dst.layers])
        k.kv_ctx_destroy(ctx)
        tier.close()
    except BaseException as e:  # reported to the parent, which fails the test
        q.put(repr(e))


def test_store_on_gpu0_restore_on_gpu1_through_a_shared_tier(orc):
    k = kvx()
    name = f"/kvx_2gpu_{os.getpid()}"
    src_np = host_layers(SPEC, 911)
    ta = synth.permuted_table(96, N_USED, 912)
    tb = synth.permuted_table(96, N_USED, 903)
    keys = k.kv_chunk_keys(synth.rng(913).integers(0, 150000, size=T).astype(np.int32), C, salt=5)
    tier = k.KvTier(orc.chunk_bytes(SPEC, C), len(keys), shared_name=name, create=True)
    ctx = k.kv_ctx_create(0)
    mpc = mp.get_context("spawn")
    q = mpc.Queue()
    p = mpc.Process(target=_reader_on_gpu1, args=(name, keys, q))
    p.start()
    try:
        src = _pool_on(0, src_np)
        s = torch.cuda.Stream(device=0)
        slots = tier.reserve_many(keys)
        k.kv_store(ctx, src, torch.from_numpy(ta).to("cuda:0"), 0, T, C, slots, stream=s)
        tier.commit_many(keys, stream=s)     # published by the GPU once the store is done
        got = q.get(timeout=300)
        p.join(timeout=60)
        assert not isinstance(got, str), got
        s.synchronize()
        assert k.kv_get_device_error(ctx) == -1
        want, _ = oracle_store(orc, SPEC, src_np, ta, 0, T, C)
        want_l, _ = oracle_load(orc, SPEC, [np.full(SPEC.layer_bytes, POISON, np.uint8)] * SPEC.num_layers,
                                tb, 0, T, C, want)
        for l in range(SPEC.num_layers):
            assert first_mismatch(got[l], want_l[l]) is None, l
    finally:
        if p.is_alive():
            p.terminate()
        k.kv_ctx_destroy(ctx)
        tier.close()
