"""Streamed cross-replica restore of a 128k-token context across two processes
(the paper's Fig. 1: replicas in their own processes share one pinned RAM
pool; here the second replica starts restoring while the first still stores).

Replica A (a child process) stores its context (27B-class shape: 62 layers x
8 KV heads x head_dim 128, bf16, 16-token pages) into a shared tier in groups
of 64 chunks, committing each group on its stream: the GPU publishes a
group's entries in the tier as soon as its bytes are stored.  Replica B (this
process) waits for each group with kv_tier_wait, acquires it on its own
stream, restores it into freshly listed pages of its own pool, and releases
it; so B can restore group g while A stores group g+1.  With each replica on
its own GPU (the paper's setting), the two overlap.  With both processes on
one GPU, as here without MPS, the GPU time-slices the two processes' contexts,
so their kernels do not run at the same time and the streamed restore ends
about when a store followed by a restore would; what the run shows then is
that every group is published, found and restored intact.  (Two replicas in
one process, on two streams of one context, do overlap: bench.py's
streamed_cross_replica leg.)

Prints A's store time, when B's last restore ended relative to the start of
A's store (host clocks of the two processes), the same for a store followed
by a restore, and checks sampled pages against B's own copy of the seeded KV.
Run from the repository root with the library built, on a GPU with about 170
GB free and a host with /dev/shm room for 33 GB:
    python examples/streamed_cross_replica.py
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
SEED = 271828
GROUP = 64                              # chunks per commit


def make_pool(k, synth, fill_seed=None):
    layers = [torch.empty(N * PAGE, dtype=torch.uint8, device="cuda") for _ in range(L)]
    for l, t in enumerate(layers):
        if fill_seed is None:
            t.fill_(synth.POISON)
        else:
            synth.normal_bf16_(t, fill_seed + l)
    return k.KvPool(layers, N, B, H, D, E), layers


def keys_of(k, salt):
    tokens = (np.arange(T, dtype=np.int64) * 104729 % 150001).astype(np.int32)
    return k.kv_chunk_keys(tokens, C, salt=salt)


def groups():
    n = T // C
    return [(g, min(n, g + GROUP)) for g in range(0, n, GROUP)]


def replica_a(name, q, q_in):
    from paper_2609_15021_gb300 import kvxfer as k, synth
    tier = k.KvTier(shared_name=name)
    pool, _ = make_pool(k, synth, SEED)
    table = torch.from_numpy(synth.permuted_table(N, T // B, seed=1)).cuda()
    ctx = k.kv_ctx_create(0)
    s = torch.cuda.Stream()
    torch.cuda.synchronize()
    q.put("ready")
    for salt, grouped in q_in.get():          # the runs B asks for: (key salt, commit per group?)
        keys = keys_of(k, salt)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        t0 = time.time()
        a.record(s)
        for g0, g1 in (groups() if grouped else [(0, T // C)]):
            slots = tier.reserve_many(keys[g0:g1], as_chunk_list=True)
            k.kv_store(ctx, pool, table, g0 * C, g1 * C, C, slots, stream=s)
            tier.commit_many(keys[g0:g1], stream=s)
        b.record(s)
        b.synchronize()
        q.put((t0, a.elapsed_time(b)))
        assert q_in.get() == "next"
    assert k.kv_get_device_error(ctx) == -1
    k.kv_ctx_destroy(ctx)
    tier.close()


def main():
    from paper_2609_15021_gb300 import _build
    _build.build()
    from paper_2609_15021_gb300 import kvxfer as k, synth
    name = f"/kvx_stream_{os.getpid()}"
    cb = L * 2 * C * H * D * E
    n_chunks = T // C
    tier = k.KvTier(cb, n_chunks, shared_name=name, create=True)   # each run's keys evict the last run's
    runs = [(SEED, True), (SEED + 1, False), (SEED + 2, True)]   # streamed, whole store first, streamed
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
        assert q_a.get(timeout=600) == "ready"
        q_b.put(runs)
        results = []
        for salt, grouped in runs:
            keys = keys_of(k, salt)
            for t in dst_layers:
                t.fill_(synth.POISON)
            torch.cuda.synchronize()
            for g0, g1 in (groups() if grouped else [(0, n_chunks)]):
                tier.wait(keys[g0:g1], timeout_s=120)     # until A's GPU has published the group
                slots = tier.acquire_many(keys[g0:g1], stream=s, as_chunk_list=True)
                k.kv_load(ctx, dst, tb, g0 * C, g1 * C, C, slots, stream=s)
                tier.release_many(keys[g0:g1], stream=s)
            s.synchronize()
            end = time.time()
            t0, store_ms = q_a.get(timeout=600)
            results.append(((end - t0) * 1e3, store_ms))
            tier.poll()
            q_b.put("next")
            rng = np.random.default_rng(salt)
            for i in rng.choice(T // B, size=64, replace=False):
                pa, pb = int(ta[i]), int(tb[i])
                for l in rng.choice(L, size=4, replace=False):
                    got = dst_layers[l][pb * PAGE:(pb + 1) * PAGE]
                    want = src_layers[l][pa * PAGE:(pa + 1) * PAGE]
                    assert torch.equal(got, want), (salt, i, l)
        assert k.kv_get_device_error(ctx) == -1
        (s1, st1), (w, stw), (s2, st2) = results
        x = n_chunks * cb
        print(f"streamed: B's last restore ended {s1:.1f} / {s2:.1f} ms after A began storing "
              f"({2 * x / min(s1, s2) / 1e6:.1f} GB/s both ways; A's store took {st1:.1f} / {st2:.1f} ms); "
              f"whole store then restore: {w:.1f} ms (store {stw:.1f} ms); 256 sampled pages bit-exact per run")
        k.kv_ctx_destroy(ctx)
        p.join(timeout=300)
        assert p.exitcode == 0
    finally:
        tier.close()


if __name__ == "__main__":
    main()
