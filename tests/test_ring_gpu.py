"""Replicas sharing one pinned tier in a ring, on the GPU (the data path of
bench.py --gpus N, paper Sec. 2 / Fig. 1).

Two processes (gloo ranks for the barriers) both use the one GPU of this
run: each keeps its own paged pool, rank 0 creates a tier in POSIX shared
memory and hands its name to rank 1, and every step each rank stores its own
context into the tier (kv_store, commit on its stream: the GPU publishes the
commits) and restores the other rank's context from it (host wait until the
keys are readable, acquire on its stream, kv_load, release).  The tier holds
half a context per rank, so each step runs in two rounds whose entries the
next round evicts.  Every step stores new bytes under keys of its own; each
rank checks its restored pages against the oracle's restore of the other
rank's chunks of that step.  No kernel waits on another process:
only the host polls the tier.
"""
import multiprocessing
import os
import sys

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    try:
        import torch
        import torch.distributed as dist

        import bench
        import oracle
        from gpu_util import POISON, first_mismatch, host_layers, device_pool, np_of, oracle_load, oracle_store
        from paper_2609_15021_gb300 import kvxfer as k
        from paper_2609_15021_gb300 import synth

        dist.init_process_group("gloo")
        orc = oracle.c_oracle()
        spec = oracle.PoolSpec(4, 96, 16, 8, 128, 2, oracle.HND)
        C, n_used = 256, 72
        T = n_used * 16 - 9                      # 5 chunks, the last one short
        n_chunks = -(-T // C)
        cb = orc.chunk_bytes(spec, C)

        def src_np_of(r, step):     # every step's context bytes differ: a stale restore would show
            return host_layers(spec, 5000 + 17 * r + 101 * step)

        def ta_of(r):
            return synth.permuted_table(96, n_used, 6000 + r)

        tb = synth.permuted_table(96, n_used, 7000 + rank)
        src = device_pool(spec, src_np_of(rank, 0))
        dst = device_pool(spec)
        ta_d, tb_d = torch.from_numpy(ta_of(rank)).cuda(), torch.from_numpy(tb).cuda()
        if rank == 0:
            plan = bench.ring_plan(world, n_chunks, cb, 3 * world * cb)   # 3 slots per rank: 2 rounds
            name = f"/kvx_ring_gpu_{os.getpid()}"
            tier = k.KvTier(cb, plan["n_slots"], shared_name=name, create=True)
            msg = [name, plan]
        else:
            msg = [None, None]
        dist.broadcast_object_list(msg, src=0)
        name, plan = msg
        if rank != 0:
            tier = k.KvTier(shared_name=name)
        dist.barrier()
        if rank == 0:
            os.unlink("/dev/shm" + name)
        ctx = k.kv_ctx_create(0)
        torch.cuda.synchronize()  # pools made on the default stream before the side stream uses them
        stream = torch.cuda.Stream()

        def store_fn(lo, hi, slots):
            k.kv_store(ctx, src, ta_d, lo * C, min(T, hi * C), C, slots, stream=stream)

        def load_fn(lo, hi, slots):
            k.kv_load(ctx, dst, tb_d, lo * C, min(T, hi * C), C, slots, stream=stream)

        ok = []
        for step in range(3):
            for l, a in zip(src.layers, src_np_of(rank, step)):
                l.copy_(torch.from_numpy(a))
            for l in dst.layers:
                l.fill_(POISON)
            torch.cuda.synchronize()
            own_keys, src_keys = bench.ring_keys(k, rank, world, T, C, step)
            for j in range(plan["rounds"]):
                bench.ring_round(tier, plan, j, n_chunks, own_keys, src_keys, store_fn, load_fn, stream.synchronize,
                                 dist.barrier, stream)
            assert k.kv_get_device_error(ctx) == -1
            s_rank = bench.ring_source(rank, world)
            chunks, _ = oracle_store(orc, spec, src_np_of(s_rank, step), ta_of(s_rank), 0, T, C)
            want, _ = oracle_load(orc, spec, [np.full(spec.layer_bytes, POISON, np.uint8)] * spec.num_layers,
                                  tb, 0, T, C, chunks)
            ok.append(all(first_mismatch(np_of(dst.layers[l]), want[l]) is None for l in range(spec.num_layers)))
        st = tier.stats()
        out[rank] = (ok, plan["rounds"], st["evictions"], st["pinned"])
        dist.barrier()
        k.kv_ctx_destroy(ctx)
        tier.close()
        dist.destroy_process_group()
    except BaseException as e:  # reported to the parent
        out[rank] = repr(e)
        raise


def test_two_replicas_share_one_tier_in_a_ring():
    sys.path[:0] = [os.path.dirname(os.path.abspath(__file__)), ROOT]
    port = 32500 + os.getpid() % 1000
    mpc = multiprocessing.get_context("spawn")
    with mpc.Manager() as m:
        out = m.dict()
        procs = [mpc.Process(target=_rank, args=(r, 2, port, out)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(timeout=600)
        res = dict(out)
    assert set(res) == {0, 1}, res
    for rank, r in res.items():
        assert not isinstance(r, str), f"rank {rank}: {r}"
        ok, rounds, evictions, pinned = r
        assert ok == [True, True, True], f"rank {rank} restored bytes differ from the oracle: {ok}"
        assert rounds == 2 and evictions > 0 and pinned == 0
