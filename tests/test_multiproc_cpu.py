"""The N > 1 plumbing of bench.py on CPU (gloo, world size 2).

Replicas share no GPU data path (paper Sec. 2: each replica owns one GPU);
state moves only through one host pool that all of them map.  bench.py runs
N > 1 replicas over one shared tier: each step, rank r stores its context
into the tier and rank r+1 restores it, in rounds when the tier cannot hold
every context at once.  Here the ranks are CPU processes: the tier is the
same shared-memory tier without page-locking (KVX_TIER_NO_PIN), and host
byte copies into and out of its slots stand in for kv_store / kv_load, so the
rank pairing, the tier name handed from rank 0 to the others, the rounds and
their evictions are checked without a GPU.  Timing across ranks is a barrier
and the maximum of the ranks' elapsed times.  The reference arm under
torchrun runs on rank 0 alone and prints exactly one line.
"""
import json
import multiprocessing
import os
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    dist.init_process_group("gloo")
    bench.barrier(world)
    got = bench.max_over_ranks(world, float(10 * (rank + 1)), rank)
    out[rank] = got
    dist.destroy_process_group()


def test_max_over_ranks_gloo():
    port = 29500 + os.getpid() % 1000
    with multiprocessing.get_context("spawn").Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(2, port, out), nprocs=2, join=True)
        assert dict(out) == {0: 20.0, 1: 20.0}


def test_reference_arm_under_torchrun_prints_once():
    port = 30500 + os.getpid() % 1000
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "1", "--cpu-sample-chunks", "2"]
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"


def test_ring_plan_fits_eight_replicas_in_one_pool():
    sys.path.insert(0, ROOT)
    import bench
    cb = 65_011_712                       # a 256-token chunk of the 27B-class shape
    budget = 168 << 30                    # what a 199 GiB host leaves after 32 GiB of headroom
    for world in (1, 2, 4, 8):
        plan = bench.ring_plan(world, 512, cb, budget)
        assert plan["n_slots"] == plan["slots_per_rank"] * world
        assert plan["n_slots"] * cb <= budget                    # one pool for all ranks
        assert plan["rounds"] * plan["slots_per_rank"] >= 512    # every chunk moves each step
        assert (plan["rounds"] - 1) * plan["slots_per_rank"] < 512
    assert bench.ring_plan(2, 512, cb, budget)["rounds"] == 1   # 2 x 33 GB fit whole
    assert bench.ring_plan(8, 512, cb, budget)["rounds"] == 2
    assert [bench.ring_source(r, 4) for r in range(4)] == [3, 0, 1, 2]
    with pytest.raises(RuntimeError):
        bench.ring_plan(8, 512, cb, cb)


def _chunk_bytes(rank, c, n, step):
    import numpy as np
    return ((np.arange(n, dtype=np.int64) * 7 + 131 * c + 977 * rank + 61 * step) % 251).astype(np.uint8)


def _ring_worker(rank, world, port, out, slots_per_rank):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import ctypes

    import numpy as np
    import torch.distributed as dist

    import bench
    from paper_2609_15021_gb300 import kvxfer as k
    dist.init_process_group("gloo")
    cb, T, C = 256, 5 * 64 - 10, 64      # 5 chunks per context, the last one short
    n_chunks = -(-T // C)
    if rank == 0:
        plan = bench.ring_plan(world, n_chunks, cb, world * slots_per_rank * cb)
        name = f"/kvx_ring_test_{os.getpid()}"
        tier = k.KvTier(cb, plan["n_slots"], shared_name=name, create=True, pin=False)
        msg = [name, plan]
    else:
        msg = [None, None]
    dist.broadcast_object_list(msg, src=0)
    name, plan = msg
    if rank != 0:
        tier = k.KvTier(shared_name=name, pin=False)
    dist.barrier()
    if rank == 0:
        os.unlink("/dev/shm" + name)
    got = {}
    step = 0

    def view(addr):                   # the ring hands the slots over as addresses (a ChunkList)
        return np.ctypeslib.as_array((ctypes.c_uint8 * cb).from_address(addr))

    def store_fn(lo, hi, slots):      # this rank's chunks into its slots (kv_store's part)
        assert len(slots) == hi - lo
        for i, c in enumerate(range(lo, hi)):
            view(slots[i])[:] = _chunk_bytes(rank, c, cb, step)

    def load_fn(lo, hi, slots):       # the source rank's chunks out of the tier (kv_load's part)
        assert len(slots) == hi - lo
        for i, c in enumerate(range(lo, hi)):
            got[c] = view(slots[i]).copy()

    ok = True
    for step in range(3):             # each step's bytes differ: a stale read would show
        got.clear()
        own_keys, src_keys = bench.ring_keys(k, rank, world, T, C, step)
        for j in range(plan["rounds"]):
            bench.ring_round(tier, plan, j, n_chunks, own_keys, src_keys, store_fn, load_fn, lambda: None,
                             dist.barrier, k.KVX_NO_STREAM)
        src_rank = bench.ring_source(rank, world)
        ok = ok and sorted(got) == list(range(n_chunks))
        ok = ok and all(np.array_equal(got[c], _chunk_bytes(src_rank, c, cb, step)) for c in got)
    st = tier.stats()
    out[rank] = (ok, plan["rounds"], st["evictions"], st["pinned"], st["slots"])
    dist.barrier()
    tier.close()
    dist.destroy_process_group()


@pytest.mark.parametrize("world,slots_per_rank,rounds", [(2, 2, 3), (2, 5, 1), (3, 2, 3)])
def test_replicas_share_one_tier_in_a_ring_gloo(world, slots_per_rank, rounds):
    """Two slots per rank: three rounds a step, each evicting the last.  Five:
    whole contexts, so the previous step's entries are still in the tier when
    the next step starts; each step's own keys keep a reader from taking them
    for this step's (their bytes differ, and the test would see them).  Three
    ranks: each restores the one before it, not the one after."""
    port = 31500 + os.getpid() % 1000 + 10 * world + slots_per_rank
    with multiprocessing.get_context("spawn").Manager() as m:
        out = m.dict()
        mp.spawn(_ring_worker, args=(world, port, out, slots_per_rank), nprocs=world, join=True)
        res = dict(out)
    assert set(res) == set(range(world))
    for rank, (ok, got_rounds, evictions, pinned, slots) in res.items():
        assert ok, f"rank {rank} did not restore its source rank's chunks"
        assert got_rounds == rounds and slots == world * slots_per_rank
        assert evictions > 0 and pinned == 0
