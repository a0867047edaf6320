"""Two replicas sharing one pinned host tier (the paper's Fig. 1 setting).

Replica A (this process) prefills nothing here: it fills its paged KV pool
with data, stores the prefix chunk by chunk into a shared tier (POSIX shared
memory, registered pinned and mapped in each process), and commits each chunk
on its stream: the GPU publishes each commit into the shared slot table once
the chunk's bytes are written, so other processes see it with no further call
from A.  Replica B (a second process on the same GPU) asks the tier
how much of the prefix it holds, acquires those chunks, restores them into
its own pool through a different block table, and checks the bytes it got
against A's pages, which A hands it through the tier as well.

Run from the repository root, with the library built:
    python examples/two_replicas.py
Prints "replica B restored N chunks, bit-exact" and exits 0 on success.
"""
import multiprocessing as mp
import os
import sys

import numpy as np
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

L, N, B, H, D, E, C = 4, 64, 16, 8, 128, 2, 256   # layers, pages, page tokens, KV heads, head dim, bf16, chunk
TOKENS = 1024                                       # the shared prefix: 4 chunks
PAGE = 2 * H * B * D * E


def chunk_keys(k):
    tokens = (np.arange(TOKENS, dtype=np.int64) * 7919 % 50021).astype(np.int32)  # the prompt's token ids
    return k.kv_chunk_keys(tokens, C, salt=2026)


def replica_b(name, q):
    from paper_2609_15021_gb300 import kvxfer as k
    tier = k.KvTier(shared_name=name)
    keys = chunk_keys(k)
    hits = tier.prefix_hits(keys)
    layers = [torch.full((N * PAGE,), 0xA5, dtype=torch.uint8, device="cuda") for _ in range(L)]
    pool = k.KvPool(layers, N, B, H, D, E)
    table = torch.from_numpy(np.random.default_rng(2).permutation(N)[:TOKENS // B].astype(np.int32)).cuda()
    ctx = k.kv_ctx_create(0)
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()
    slots = tier.acquire_many(keys[:hits], stream=stream)  # acquire, restore, release: all on `stream`
    k.kv_load(ctx, pool, table, 0, hits * C, C, slots, stream=stream)
    tier.release_many(keys[:hits], stream=stream)
    stream.synchronize()
    assert k.kv_get_device_error(ctx) == -1
    got = [t.view(N, PAGE)[table.long()].cpu() for t in layers]
    k.kv_ctx_destroy(ctx)
    tier.close()
    q.put((hits, [g.numpy() for g in got]))


def main():
    from paper_2609_15021_gb300 import _build
    _build.build()
    from paper_2609_15021_gb300 import kvxfer as k
    name = f"/kvx_example_{os.getpid()}"
    cb = L * 2 * C * H * D * E
    tier = k.KvTier(cb, 16, shared_name=name, create=True)
    try:
        # replica A: its pool, a block table, and the store of every chunk
        layers = [torch.randint(0, 256, (N * PAGE,), dtype=torch.uint8, device="cuda") for _ in range(L)]
        pool = k.KvPool(layers, N, B, H, D, E)
        table = torch.from_numpy(np.random.default_rng(1).permutation(N)[:TOKENS // B].astype(np.int32)).cuda()
        ctx = k.kv_ctx_create(0)
        stream = torch.cuda.Stream()
        torch.cuda.synchronize()
        keys = chunk_keys(k)
        slots = tier.reserve_many(keys)              # one slot per chunk key
        k.kv_store(ctx, pool, table, 0, TOKENS, C, slots, stream=stream)
        tier.commit_many(keys, stream=stream)        # readable everywhere once the GPU has passed this point
        stream.synchronize()
        want = [t.view(N, PAGE)[table.long()].cpu().numpy() for t in layers]
        k.kv_ctx_destroy(ctx)

        # replica B in its own process
        mpc = mp.get_context("spawn")
        q = mpc.Queue()
        p = mpc.Process(target=replica_b, args=(name, q))
        p.start()
        hits, got = q.get(timeout=300)
        p.join(timeout=60)
        assert p.exitcode == 0 and hits == len(keys)
        assert all(np.array_equal(a, b) for a, b in zip(got, want)), "restored pages differ"
        print(f"replica B restored {hits} chunks, bit-exact")
    finally:
        tier.close()


if __name__ == "__main__":
    main()
