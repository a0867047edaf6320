"""Cross-replica restore of a 128k-token context through a shared host tier
(the paper's Fig. 1 at full size: two replicas, each its own process, one
pinned RAM pool between them).

Replica A (a child process) fills its paged KV pool (27B-class shape: 62
layers x 8 KV heads x head_dim 128, bf16, 16-token pages), stores the whole
prefix into the tier with one kv_store and commits every chunk with one
kv_tier_commit_many on its stream, then makes no further tier call.  Replica
B (this process) polls the tier until the GPU has published every commit,
acquires the chunks, restores them with one kv_load into freshly listed pages
of its own pool, and checks sampled pages against its own copy of the same
seeded KV.

Prints the store time in A, when B saw every entry relative to the moment
A's host thread saw its store end (both on the host clock), B's restore time
(the first restore, right after A's store, and the one after it), and how
long B took to open the tier.  Run from the repository root, with the
library built, on a GPU with about 170 GB free and a host with about 80 GB of
free memory and /dev/shm room for 33 GB:
    python examples/cross_replica_128k.py
"""
import multiprocessing as mp
import os
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

L, B, H, D, E, C = 62, 16, 8, 128, 2, 256
N, T = 10240, 131072                    # pool pages, context tokens
PAGE = 2 * H * B * D * E
SEED = 314159


def make_pool(k, synth, fill_seed=None):
    layers = [torch.empty(N * PAGE, dtype=torch.uint8, device="cuda") for _ in range(L)]
    for l, t in enumerate(layers):
        if fill_seed is None:
            t.fill_(synth.POISON)
        else:
            synth.normal_bf16_(t, fill_seed + l)
    return k.KvPool(layers, N, B, H, D, E), layers


def keys_of(k):
    tokens = (np.arange(T, dtype=np.int64) * 7919 % 150001).astype(np.int32)
    return k.kv_chunk_keys(tokens, C, salt=SEED)


def replica_a(name, q, q_in):
    from paper_2609_15021_gb300 import kvxfer as k, synth
    tier = k.KvTier(shared_name=name)
    pool, _ = make_pool(k, synth, SEED)
    table = torch.from_numpy(synth.permuted_table(N, T // B, seed=1)).cuda()
    ctx = k.kv_ctx_create(0)
    s = torch.cuda.Stream()
    keys = keys_of(k)
    torch.cuda.synchronize()
    q.put("ready")
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    slots = tier.reserve_many(keys, as_chunk_list=True)
    a.record(s)
    k.kv_store(ctx, pool, table, 0, T, C, slots, stream=s)
    b.record(s)
    tier.commit_many(keys, stream=s)
    b.synchronize()
    q.put((time.time(), a.elapsed_time(b)))   # host clock at the end of the store, store ms
    q_in.get()                                # until B is done; no tier call meanwhile
    assert k.kv_get_device_error(ctx) == -1
    k.kv_ctx_destroy(ctx)
    tier.close()


def main():
    from paper_2609_15021_gb300 import _build
    _build.build()
    from paper_2609_15021_gb300 import kvxfer as k, synth
    name = f"/kvx_cross_{os.getpid()}"
    cb = L * 2 * C * H * D * E
    n_chunks = T // C
    t_open = time.perf_counter()
    tier = k.KvTier(cb, n_chunks, shared_name=name, create=True)
    open_ms = (time.perf_counter() - t_open) * 1e3
    try:
        mpc = mp.get_context("spawn")
        q_a, q_b = mpc.Queue(), mpc.Queue()
        p = mpc.Process(target=replica_a, args=(name, q_a, q_b))
        p.start()
        dst, dst_layers = make_pool(k, synth)
        src_layers = make_pool(k, synth, SEED)[1]    # B's own copy of A's seeded KV, for the check
        ta = torch.from_numpy(synth.permuted_table(N, T // B, seed=1)).cuda()
        tb = torch.from_numpy(synth.permuted_table(N, T // B, seed=2)).cuda()
        ctx = k.kv_ctx_create(0)
        s = torch.cuda.Stream()
        keys = keys_of(k)
        assert q_a.get(timeout=600) == "ready"
        while tier.prefix_hits(keys) < n_chunks:
            time.sleep(0.0002)
        seen = time.time()
        store_end, store_ms = q_a.get(timeout=600)
        def restore():
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize()
            a.record(s)
            slots = tier.acquire_many(keys, stream=s, as_chunk_list=True)
            k.kv_load(ctx, dst, tb, 0, T, C, slots, stream=s)
            tier.release_many(keys, stream=s)
            b.record(s)
            b.synchronize()
            return a.elapsed_time(b)

        first_ms = restore()     # right after A's store
        restore_ms = restore()   # right after the first restore
        assert k.kv_get_device_error(ctx) == -1
        rng = np.random.default_rng(7)
        for i in rng.choice(T // B, size=64, replace=False):
            pa, pb = int(ta[i]), int(tb[i])
            for l in rng.choice(L, size=4, replace=False):
                got = dst_layers[l][pb * PAGE:(pb + 1) * PAGE]
                want = src_layers[l][pa * PAGE:(pa + 1) * PAGE]
                assert torch.equal(got, want), (i, l)
        x = n_chunks * cb
        print(f"replica A stored {x / 1e9:.1f} GB in {store_ms:.1f} ms ({x / store_ms / 1e6:.1f} GB/s); "
              f"replica B saw all {n_chunks} chunks {(seen - store_end) * 1e3:+.2f} ms from the moment A's host "
              f"saw its store end (negative: B first) and restored them in {first_ms:.1f} ms the first time, "
              f"{restore_ms:.1f} ms ({x / restore_ms / 1e6:.1f} GB/s) the next; "
              f"256 sampled pages bit-exact; B opened the tier in {open_ms:.0f} ms")
        k.kv_ctx_destroy(ctx)
        q_b.put("done")
        p.join(timeout=300)
        assert p.exitcode == 0
    finally:
        tier.close()


if __name__ == "__main__":
    main()
