"""A host tier shared by two processes (paper Fig. 1: each replica is its own
process; both use one pinned RAM pool).

CPU test: the bookkeeping only (KVX_TIER_NO_PIN): entries written and
committed by one process are found, read and pinned by the other; LRU and
pinning hold across processes.

GPU test: process A stores chunks of a pool into the shared pool on its
stream, behind a producer delayed by ~2*10^9 GPU cycles, and commits them on
that stream.  Process B must not see them while A's GPU work is pending,
must see them once the GPU has published the commits although A makes no
further call, and then restores them into its own pool on the same GPU and
checks every byte against the oracle (so the publication came after the
bytes).  The processes synchronise on the host only (no kernel waits on
another process).
"""
import multiprocessing as mp
import os
import sys

import numpy as np
import pytest

from paper_2609_15021_gb300 import probe

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _name(tag):
    return f"/kvx_{tag}_{os.getpid()}"


def _child_cpu(name, q_in, q_out):
    sys.path.insert(0, ROOT)
    from paper_2609_15021_gb300 import kvxfer as k
    NO = -1
    t = k.KvTier(shared_name=name, pin=False)
    assert q_in.get() == "written"
    assert t.prefix_hits([1, 2, 3]) == 2
    s = t.acquire(1, NO)
    q_out.put(int(s[0]))                 # the byte the other process wrote
    s2 = t.reserve(7)                    # write an entry of our own
    s2.fill_(77)
    t.commit(7, NO)
    q_out.put("pinned 1, wrote 7")
    assert q_in.get() == "check"
    q_out.put(t.prefix_hits([1, 7]))
    t.release(1, NO)
    q_out.put("released")
    assert q_in.get() == "bye"
    t.close()


def test_shared_tier_bookkeeping_across_processes():
    sys.path.insert(0, ROOT)
    from paper_2609_15021_gb300 import _build
    _build.build()
    from paper_2609_15021_gb300 import kvxfer as k
    NO = -1
    name = _name("cpu")
    t = k.KvTier(64, 3, shared_name=name, create=True, pin=False)
    ctx = mp.get_context("spawn")
    q_in, q_out = ctx.Queue(), ctx.Queue()
    p = ctx.Process(target=_child_cpu, args=(name, q_in, q_out))
    p.start()
    try:
        for key in (1, 2):
            s = t.reserve(key)
            s.fill_(10 + key)
            t.commit(key, NO)
        q_in.put("written")
        assert q_out.get(timeout=60) == 11
        assert q_out.get(timeout=60) == "pinned 1, wrote 7"
        assert t.prefix_hits([7]) == 1
        assert int(t.acquire(7, NO)[3]) == 77
        t.release(7, NO)
        # 3 slots: 1 (pinned by the child), 2, 7; a new key may evict 2 or 7, never 1
        t.reserve(8)
        t.commit(8, NO)
        t.reserve(9)
        t.commit(9, NO)
        q_in.put("check")
        assert q_out.get(timeout=60) == 1      # child still sees 1; 7 was evicted (least recent)
        assert q_out.get(timeout=60) == "released"
        st = t.stats()
        assert st["entries"] == 3 and st["evictions"] == 2
        assert t.prefix_hits([1]) == 1
        q_in.put("bye")
        p.join(timeout=60)
        assert p.exitcode == 0
    finally:
        if p.is_alive():
            p.kill()
        t.close()


def _child_dies(name, q_out):
    """Pins an entry, reserves another, then the process ends without releasing
    or committing either (a replica that crashed)."""
    sys.path.insert(0, ROOT)
    from paper_2609_15021_gb300 import kvxfer as k
    NO = -1
    t = k.KvTier(shared_name=name, pin=False)
    t.acquire(1, NO)
    t.reserve(5).fill_(55)
    q_out.put("holding")
    q_out.close()
    q_out.join_thread()             # the message is out before the process ends
    os._exit(0)                     # no release, no commit, no close


def test_dead_process_pins_and_writes_are_reclaimed():
    """Failure detection on the host: a process that dies holding a pin and a
    half-written entry does not keep either slot forever."""
    sys.path.insert(0, ROOT)
    from paper_2609_15021_gb300 import _build
    _build.build()
    from paper_2609_15021_gb300 import kvxfer as k
    NO = -1
    name = _name("dead")
    t = k.KvTier(64, 2, shared_name=name, create=True, pin=False)
    try:
        t.reserve(1).fill_(11)
        t.commit(1, NO)
        ctx = mp.get_context("spawn")
        q_out = ctx.Queue()
        p = ctx.Process(target=_child_dies, args=(name, q_out))
        p.start()
        assert q_out.get(timeout=60) == "holding"
        p.join(timeout=60)
        assert p.exitcode == 0
        st = t.stats()
        assert st["entries"] == 2 and st["pinned"] == 2      # 1 pinned by the dead reader, 5 reserved
        assert t.prefix_hits([5]) == 0                       # never committed: not visible
        # both slots are held: a reservation reclaims what the dead process left, then succeeds
        s = t.reserve(6)
        s.fill_(66)
        t.commit(6, NO)
        assert t.prefix_hits([1]) == 1 and int(t.acquire(1, NO)[0]) == 11   # the committed entry survives
        t.release(1, NO)
        assert t.prefix_hits([5]) == 0 and t.prefix_hits([6]) == 1
        st = t.stats()
        assert st["pinned"] == 0 and st["entries"] == 2
        assert t.reclaim() == 0                              # nothing left to reclaim
    finally:
        t.close()


def _child_dies_mid_reserve(name, after_calls):
    sys.path.insert(0, ROOT)
    from paper_2609_15021_gb300 import kvxfer as k
    t = k.KvTier(shared_name=name, pin=False)
    k.kv_fault_inject("tier_exit", after_calls)
    for key in (30, 31):
        t.reserve(key)                 # the armed reservation ends the process inside the lock
    os._exit(0)                        # not reached when the hook fires


@pytest.mark.parametrize("after_calls", [0, 1])
def test_process_dying_mid_reserve_leaves_no_wrong_entry(after_calls):
    """Failure detection on the host: a replica that dies inside kv_tier_reserve,
    holding the table lock, right after it has evicted an entry and indexed
    its new key, leaves neither that key readable (the slot still holds the
    evicted bytes) nor a lock that blocks the others.  The next call here takes
    the lock over (the mutex is robust), rebuilds the key index, and the dead
    process's slot is reclaimed."""
    sys.path.insert(0, ROOT)
    from paper_2609_15021_gb300 import _build
    _build.build()
    from paper_2609_15021_gb300 import kvxfer as k
    NO = -1
    name = _name(f"midres{after_calls}")
    t = k.KvTier(64, 3, shared_name=name, create=True, pin=False)
    try:
        for key, fill in ((1, 11), (2, 22), (3, 33)):      # a full tier: the child must evict
            t.reserve(key).fill_(fill)
            t.commit(key, NO)
        ctx = mp.get_context("spawn")
        p = ctx.Process(target=_child_dies_mid_reserve, args=(name, after_calls))
        p.start()
        p.join(timeout=120)
        assert p.exitcode == 3                              # the hook's exit, inside the lock
        died_at = 30 + after_calls
        assert t.prefix_hits([died_at]) == 0                # never readable under the new key
        with pytest.raises(k.KvxError) as e:
            t.acquire(died_at, NO)
        assert e.value.status == k.KVX_ENOENT
        survivors = [key for key in (1, 2, 3) if t.prefix_hits([key]) == 1]
        assert len(survivors) == 2 - after_calls           # one eviction per reservation the child made
        for key in survivors:                               # what survives reads its own bytes
            assert int(t.acquire(key, NO)[0]) == key * 11
            t.release(key, NO)
        assert t.reclaim() == 1 + after_calls               # the dead writer's reservation(s)
        s = t.reserve(died_at)                              # the key is usable again
        s.fill_(44)
        t.commit(died_at, NO)
        assert int(t.acquire(died_at, NO)[0]) == 44
        t.release(died_at, NO)
        st = t.stats()
        assert st["pinned"] == 0 and st["entries"] == len(survivors) + 1
    finally:
        t.close()


def test_reclaim_leaves_live_processes_alone():
    sys.path.insert(0, ROOT)
    from paper_2609_15021_gb300 import _build
    _build.build()
    from paper_2609_15021_gb300 import kvxfer as k
    NO = -1
    name = _name("live")
    t = k.KvTier(64, 2, shared_name=name, create=True, pin=False)
    try:
        t.reserve(1)
        t.commit(1, NO)
        t.acquire(1, NO)
        t.reserve(2)                                         # this process is alive: nothing reclaimed
        assert t.reclaim() == 0
        assert t.stats()["pinned"] == 2
        with pytest.raises(k.KvxError) as e:
            t.reserve(3)
        assert e.value.status == k.KVX_ENOMEM
        t.release(1, NO)
        with pytest.raises(k.KvxError) as e:
            t.release(1, NO)                                 # no pin left to drop
        assert e.value.status == k.KVX_EINVAL
        t.release(2, NO)                                     # give the reservation up
        assert t.stats()["entries"] == 1
    finally:
        t.close()


def _child_gpu(name, q_in, q_out):
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import torch

    import oracle
    from gpu_util import POISON, device_pool, first_mismatch, host_layers, np_of, oracle_load, oracle_store
    from paper_2609_15021_gb300 import kvxfer as k
    from paper_2609_15021_gb300 import synth
    spec = oracle.PoolSpec(4, 64, 16, 8, 128, 2, oracle.HND)
    C, n_used = 256, 32
    import time
    t = k.KvTier(shared_name=name)
    final_np = host_layers(spec, 2)
    ta = synth.permuted_table(64, n_used, 3)
    tb = synth.permuted_table(64, n_used, 4)
    dst = device_pool(spec)
    ctx = k.kv_ctx_create(0)
    s = torch.cuda.Stream()
    tb_d = torch.from_numpy(tb).cuda()
    torch.cuda.synchronize()
    q_out.put("ready")                             # every slow set-up step is done
    keys = q_in.get()
    q_out.put(t.prefix_hits(keys))                 # A's GPU work is still delayed: nothing visible
    t0, hits = time.monotonic(), 0
    while hits < len(keys) and time.monotonic() - t0 < 120:
        hits = t.prefix_hits(keys)                 # A makes no call meanwhile: the GPU publishes
        time.sleep(0.001)
    q_out.put(hits)
    for c, key in enumerate(keys):
        slot = t.acquire(key, stream=s)
        k.kv_load(ctx, dst, tb_d, c * C, (c + 1) * C, C, [slot], stream=s)
        t.release(key, stream=s)
    s.synchronize()
    orc = oracle.c_oracle()
    want, _ = oracle_store(orc, spec, final_np, ta, 0, n_used * 16, C)
    loaded, _ = oracle_load(orc, spec, [np.full(spec.layer_bytes, POISON, np.uint8)] * 4, tb, 0, n_used * 16, C, want)
    ok = all(first_mismatch(np_of(dst.layers[l]), loaded[l]) is None for l in range(4))
    k.kv_ctx_destroy(ctx)
    t.close()
    q_out.put(ok)


@pytest.mark.gpu
@pytest.mark.parametrize("commit", ["per_key", "many"])
def test_shared_tier_store_in_one_process_restore_in_another(commit):
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import torch

    import oracle
    from gpu_util import device_pool, host_layers
    from paper_2609_15021_gb300 import kvxfer as k
    from paper_2609_15021_gb300 import synth
    spec = oracle.PoolSpec(4, 64, 16, 8, 128, 2, oracle.HND)
    C, n_used = 256, 32
    T = n_used * 16
    orc = oracle.c_oracle()
    name = _name(f"gpu{commit}")
    tier = k.KvTier(orc.chunk_bytes(spec, C), 4, shared_name=name, create=True)
    ctx_mp = mp.get_context("spawn")
    q_in, q_out = ctx_mp.Queue(), ctx_mp.Queue()
    p = ctx_mp.Process(target=_child_gpu, args=(name, q_in, q_out))
    p.start()
    ctx = k.kv_ctx_create(0)
    try:
        stale_np, final_np = host_layers(spec, 1), host_layers(spec, 2)
        pool = device_pool(spec, stale_np)
        final_dev = [torch.from_numpy(a).cuda() for a in final_np]
        ta_d = torch.from_numpy(synth.permuted_table(64, n_used, 3)).cuda()
        keys = k.kv_chunk_keys(synth.rng(11).integers(0, 150000, size=T).astype(np.int32), C, salt=1)
        s = torch.cuda.Stream()
        torch.cuda.synchronize()
        assert q_out.get(timeout=300) == "ready"  # the other process waits for the keys from here on
        for l in range(4):   # the producer finishes writing the KV ~2*10^9 cycles (~1 s) later
            probe.kvx_probe_delayed_copy(pool.layers[l], final_dev[l], spec.layer_bytes, 2 * 10 ** 9 if l == 0 else 0, s)
        if commit == "many":                    # one store, one publication launch for both chunks
            slots = tier.reserve_many(keys)
            k.kv_store(ctx, pool, ta_d, 0, T, C, slots, stream=s)
            tier.commit_many(keys, stream=s)
        else:
            for c, key in enumerate(keys):
                slot = tier.reserve(key)
                k.kv_store(ctx, pool, ta_d, c * C, (c + 1) * C, C, [slot], stream=s)
                tier.commit(key, stream=s)
        q_in.put(keys)
        assert q_out.get(timeout=120) == 0      # still in flight on our stream: invisible elsewhere
        # no tier call and no synchronisation here until the other process has seen every entry
        assert q_out.get(timeout=180) == len(keys)
        assert q_out.get(timeout=300) is True   # the other process restored every byte
        s.synchronize()
        tier.poll()
        p.join(timeout=120)
        assert p.exitcode == 0
    finally:
        if p.is_alive():
            p.kill()
        k.kv_ctx_destroy(ctx)
        tier.close()


def _child_commits_then_dies(name, q_out):
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import torch

    import oracle
    from gpu_util import device_pool, host_layers
    from paper_2609_15021_gb300 import kvxfer as k
    from paper_2609_15021_gb300 import synth
    spec = oracle.PoolSpec(4, 64, 16, 8, 128, 2, oracle.HND)
    C, n_used = 256, 32
    t = k.KvTier(shared_name=name)
    pool = device_pool(spec, host_layers(spec, 21))
    ta_d = torch.from_numpy(synth.permuted_table(64, n_used, 22)).cuda()
    ctx = k.kv_ctx_create(0)
    s = torch.cuda.Stream()
    t.reserve(503)                   # a reservation left unfinished
    scratch = torch.empty(4096, dtype=torch.uint8, device="cuda")
    torch.cuda.synchronize()
    probe.kvx_probe_delayed_fill(scratch, 4096, 0, 4 * 10 ** 8, s)   # the stores start ~0.2 s from now
    for c, key in enumerate([501, 502]):
        slot = t.reserve(key)
        k.kv_store(ctx, pool, ta_d, c * C, (c + 1) * C, C, [slot], stream=s)
        t.commit(key, stream=s)      # every tier call of this process comes before the GPU work ends
    s.synchronize()                  # the GPU has published both commits; no tier call after this
    q_out.put("done")
    q_out.close()
    q_out.join_thread()
    os._exit(0)


@pytest.mark.gpu
def test_published_entries_of_a_dead_writer_stay_readable():
    """Failure detection: a replica that committed chunks on its stream and died
    after its GPU work finished, with no tier call in between, leaves those
    entries complete and readable (the GPU published them); reclaim frees only
    the reservation it never finished.  The bytes restored in this process
    match the oracle."""
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import torch

    import oracle
    from gpu_util import POISON, device_pool, first_mismatch, host_layers, np_of, oracle_load, oracle_store
    from paper_2609_15021_gb300 import kvxfer as k
    from paper_2609_15021_gb300 import synth
    spec = oracle.PoolSpec(4, 64, 16, 8, 128, 2, oracle.HND)
    C, n_used = 256, 32
    orc = oracle.c_oracle()
    name = _name("pubdead")
    tier = k.KvTier(orc.chunk_bytes(spec, C), 4, shared_name=name, create=True)
    try:
        ctx_mp = mp.get_context("spawn")
        q_out = ctx_mp.Queue()
        p = ctx_mp.Process(target=_child_commits_then_dies, args=(name, q_out))
        p.start()
        assert q_out.get(timeout=300) == "done"
        p.join(timeout=120)
        assert p.exitcode == 0
        assert tier.prefix_hits([501, 502]) == 2
        assert tier.reclaim() == 1                           # the unfinished reservation only
        assert tier.prefix_hits([501, 502, 503]) == 2
        dst = device_pool(spec)
        tb = synth.permuted_table(64, n_used, 23)
        tb_d = torch.from_numpy(tb).cuda()
        ctx = k.kv_ctx_create(0)
        torch.cuda.synchronize()  # the poisoned pool was filled on the default stream
        s = torch.cuda.Stream()
        try:
            for c, key in enumerate([501, 502]):
                slot = tier.acquire(key, stream=s)
                k.kv_load(ctx, dst, tb_d, c * C, (c + 1) * C, C, [slot], stream=s)
                tier.release(key, stream=s)
            s.synchronize()
            assert k.kv_get_device_error(ctx) == -1
        finally:
            k.kv_ctx_destroy(ctx)
        ta = synth.permuted_table(64, n_used, 22)
        want, _ = oracle_store(orc, spec, host_layers(spec, 21), ta, 0, n_used * 16, C)
        loaded, _ = oracle_load(orc, spec, [np.full(spec.layer_bytes, POISON, np.uint8)] * 4, tb, 0,
                                n_used * 16, C, want)
        for l in range(4):
            assert first_mismatch(np_of(dst.layers[l]), loaded[l]) is None, f"layer {l}"
    finally:
        tier.close()


def _late_writer(name, keys, delay_s, q):
    sys.path.insert(0, ROOT)
    import time
    from paper_2609_15021_gb300 import kvxfer as k
    t = k.KvTier(shared_name=name, pin=False)
    q.put("open")
    time.sleep(delay_s)
    for key in keys:
        t.reserve(key).fill_(key % 251)
        t.commit(key, -1)
    q.put("committed")
    t.close()


def test_tier_wait_across_processes():
    """kv_tier_wait returns at once for readable keys, runs out (KVX_ETIMEOUT,
    the readable prefix reported) when one is missing, and returns soon after
    another process commits the keys it waits for, well inside its limit."""
    import time
    sys.path.insert(0, ROOT)
    from paper_2609_15021_gb300 import kvxfer as k
    name = _name("wait")
    t = k.KvTier(64, 8, shared_name=name, create=True, pin=False)
    try:
        for key in (1, 2):
            t.reserve(key)
            t.commit(key, -1)
        assert t.wait([1, 2], timeout_s=0.0) == 2
        t0 = time.perf_counter()
        with pytest.raises(k.KvxError) as e:
            t.wait([1, 2, 3], timeout_s=0.05)
        waited = time.perf_counter() - t0
        assert e.value.status == k.KVX_ETIMEOUT and e.value.hits == 2
        assert 0.04 < waited < 2.0
        lib = k._lib
        keys = (__import__("ctypes").c_uint64 * 1)(1)
        assert lib.kv_tier_wait(t.handle, keys, 1, -1, None) == k.KVX_EINVAL
        assert lib.kv_tier_wait(t.handle, keys, -1, 0, None) == k.KVX_EINVAL
        ctx = mp.get_context("spawn")
        q = ctx.Queue()
        p = ctx.Process(target=_late_writer, args=(name, [11, 12, 13], 0.3, q))
        p.start()
        assert q.get(timeout=60) == "open"
        t0 = time.perf_counter()
        assert t.wait([11, 12, 13], timeout_s=30.0) == 3
        waited = time.perf_counter() - t0
        assert q.get(timeout=60) == "committed"
        p.join(timeout=60)
        assert 0.25 < waited < 10.0
        assert int(t.acquire(12, -1)[0]) == 12
        t.release(12, -1)
    finally:
        t.close()


def _stress_worker(name, seed, n_ops, n_keys, q_out, start=None):
    """Random reserve / write / commit (or abandon), acquire / check / hold /
    release on one shared tier.  Every writer of a key writes the same bytes
    (the key repeated), so a slot this process holds pinned must always read
    back as its key: any other bytes mean the slot went to another key, or to
    a writer, while it was pinned.  Puts (bytes mismatches, counts) on q_out;
    a call that had to succeed and did not is reported there too."""
    import collections
    import ctypes
    import random
    import traceback
    sys.path.insert(0, ROOT)
    from paper_2609_15021_gb300 import kvxfer as k
    lib = k._lib
    t = k.KvTier(shared_name=name, pin=False)
    nb = t.slot_bytes
    no = ctypes.c_void_p(k.KVX_NO_STREAM & (2**64 - 1))
    pattern = {key: key.to_bytes(8, "little") * (nb // 8) for key in range(1, n_keys + 1)}
    rnd = random.Random(seed)
    held, counts = [], collections.Counter()

    def check(key, ptr):
        if ctypes.string_at(ptr, nb) != pattern[key]:
            counts["bad bytes"] += 1

    def must(status, what):
        if status != k.KVX_OK:
            raise RuntimeError(f"{what} returned {status}")

    if start is not None:
        start.wait(timeout=120)  # every process begins at once
    try:
        for _ in range(n_ops):
            key = rnd.randint(1, n_keys)
            r = rnd.random()
            out = ctypes.c_void_p()
            if r < 0.4:
                st = lib.kv_tier_reserve(t.handle, key, ctypes.byref(out))
                if st == k.KVX_OK:
                    ctypes.memmove(out.value, pattern[key], nb)
                    if rnd.random() < 0.1:
                        must(lib.kv_tier_release(t.handle, key, no), "release of a reservation")
                        counts["abandoned"] += 1
                    else:
                        must(lib.kv_tier_commit(t.handle, key, no), "commit")
                        counts["committed"] += 1
                elif st in (k.KVX_EBUSY, k.KVX_ENOMEM):
                    counts[f"reserve {st}"] += 1
                else:
                    must(st, "reserve")
            elif r < 0.85:
                st = lib.kv_tier_acquire(t.handle, key, no, ctypes.byref(out))
                if st == k.KVX_OK:
                    check(key, out.value)
                    counts["acquired"] += 1
                    if rnd.random() < 0.3 and len(held) < 3:
                        held.append((key, out.value))
                    else:
                        must(lib.kv_tier_release(t.handle, key, no), "release")
                elif st in (k.KVX_ENOENT, k.KVX_EBUSY):
                    counts[f"acquire {st}"] += 1
                else:
                    must(st, "acquire")
            elif held:
                key, ptr = held.pop(rnd.randrange(len(held)))
                check(key, ptr)
                must(lib.kv_tier_release(t.handle, key, no), "release of a held pin")
        for key, ptr in held:
            check(key, ptr)
            must(lib.kv_tier_release(t.handle, key, no), "release of a held pin")
    except Exception:
        counts["failed"] += 1
        counts[traceback.format_exc().strip().splitlines()[-1]] += 1
    t.close()
    q_out.put(dict(counts))


def test_processes_racing_on_one_tier_never_share_a_pinned_slot():
    """Three processes make thousands of random tier calls on 8 slots shared by
    24 keys (constant eviction).  No pinned slot ever changes under its holder,
    every committed entry reads back as its key, and nothing stays pinned."""
    sys.path.insert(0, ROOT)
    from paper_2609_15021_gb300 import _build
    _build.build()
    from paper_2609_15021_gb300 import kvxfer as k
    n_keys, n_ops = 24, 20000
    name = _name("stress")
    t = k.KvTier(4096, 8, shared_name=name, create=True, pin=False)
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    start = ctx.Barrier(4)
    procs = [ctx.Process(target=_stress_worker, args=(name, seed, n_ops, n_keys, q, start)) for seed in (11, 12, 13)]
    for p in procs:
        p.start()
    try:
        start.wait(timeout=120)
        results = [q.get(timeout=300) for _ in procs]
        for p in procs:
            p.join(timeout=60)
            assert p.exitcode == 0
        for counts in results:
            assert "failed" not in counts and "bad bytes" not in counts, counts
            assert counts.get("committed", 0) > 1000 and counts.get("acquired", 0) > 1000, counts
        st = t.stats()
        assert st["pinned"] == 0 and st["entries"] <= 8 and st["evictions"] > 0, st
        import ctypes
        no = ctypes.c_void_p(k.KVX_NO_STREAM & (2**64 - 1))
        for key in range(1, n_keys + 1):
            out = ctypes.c_void_p()
            if k._lib.kv_tier_acquire(t.handle, key, no, ctypes.byref(out)) == k.KVX_OK:
                assert ctypes.string_at(out.value, 4096) == key.to_bytes(8, "little") * 512
                assert k._lib.kv_tier_release(t.handle, key, no) == k.KVX_OK
    finally:
        for p in procs:
            if p.is_alive():
                p.kill()
        t.close()


def _pin_holder(name, q_in, q_out):
    """Acquires key 1 of a shared tier, reports, and releases it when told."""
    import ctypes
    sys.path.insert(0, ROOT)
    from paper_2609_15021_gb300 import kvxfer as k
    t = k.KvTier(shared_name=name, pin=False)
    no = ctypes.c_void_p(k.KVX_NO_STREAM & (2**64 - 1))
    out = ctypes.c_void_p()
    q_out.put(k._lib.kv_tier_acquire(t.handle, 1, no, ctypes.byref(out)))
    assert q_in.get(timeout=120) == "release"
    q_out.put(k._lib.kv_tier_release(t.handle, 1, no))
    t.close()


def test_at_most_eight_processes_pin_one_entry():
    """Eight processes hold pins on one entry; a ninth gets KVX_EBUSY, and gets
    its pin once one of the eight has released (pins are kept per process, so
    a process's second pin on the entry costs no extra holder)."""
    import ctypes
    sys.path.insert(0, ROOT)
    from paper_2609_15021_gb300 import _build
    _build.build()
    from paper_2609_15021_gb300 import kvxfer as k
    name = _name("holders")
    t = k.KvTier(64, 2, shared_name=name, create=True, pin=False)
    no = ctypes.c_void_p(k.KVX_NO_STREAM & (2**64 - 1))
    out = ctypes.c_void_p()
    assert k._lib.kv_tier_reserve(t.handle, 1, ctypes.byref(out)) == k.KVX_OK
    assert k._lib.kv_tier_commit(t.handle, 1, no) == k.KVX_OK
    ctx = mp.get_context("spawn")
    q_out = ctx.Queue()
    holders = [(ctx.Process(target=_pin_holder, args=(name, q_in, q_out)), q_in)
               for q_in in (ctx.Queue() for _ in range(8))]
    try:
        for p, _ in holders:
            p.start()
        assert [q_out.get(timeout=120) for _ in holders] == [k.KVX_OK] * 8
        assert t.stats()["pinned"] == 1
        assert k._lib.kv_tier_acquire(t.handle, 1, no, ctypes.byref(out)) == k.KVX_EBUSY  # a ninth process
        assert k._lib.kv_tier_reserve(t.handle, 1, ctypes.byref(out)) == k.KVX_EBUSY      # pinned: no rewrite
        p0, q0 = holders[0]
        q0.put("release")
        assert q_out.get(timeout=120) == k.KVX_OK
        p0.join(timeout=60)
        assert k._lib.kv_tier_acquire(t.handle, 1, no, ctypes.byref(out)) == k.KVX_OK
        assert k._lib.kv_tier_acquire(t.handle, 1, no, ctypes.byref(out)) == k.KVX_OK  # same process, same holder
        for _ in range(2):
            assert k._lib.kv_tier_release(t.handle, 1, no) == k.KVX_OK
        for p, q_in in holders[1:]:
            q_in.put("release")
        assert [q_out.get(timeout=120) for _ in holders[1:]] == [k.KVX_OK] * 7
        for p, _ in holders:
            p.join(timeout=60)
            assert p.exitcode == 0
        assert t.stats()["pinned"] == 0
    finally:
        for p, _ in holders:
            if p.is_alive():
                p.kill()
        t.close()
