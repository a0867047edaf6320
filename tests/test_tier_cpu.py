"""The shared host tier's bookkeeping on CPU: chunk keys, LRU eviction, pinning.

Runs over caller-owned host memory with KVX_NO_STREAM (no CUDA call is made).
"""
import numpy as np
import pytest

from paper_2609_15021_gb300 import _build


@pytest.fixture(scope="module")
def k():
    _build.build()
    from paper_2609_15021_gb300 import kvxfer
    return kvxfer


NO = -1  # KVX_NO_STREAM


def test_chunk_keys_chain_over_the_prefix(k):
    toks = np.arange(1000, dtype=np.int32) * 7 % 5003
    keys = k.kv_chunk_keys(toks, 256, salt=1)
    assert len(keys) == 4 and len(set(keys)) == 4
    assert keys == k.kv_chunk_keys(toks, 256, salt=1)                 # deterministic
    assert all(a != b for a, b in zip(keys, k.kv_chunk_keys(toks, 256, salt=2)))  # salt = namespace
    t2 = toks.copy()
    t2[600] += 1                                                      # a token of chunk 2
    k2 = k.kv_chunk_keys(t2, 256, salt=1)
    assert k2[:2] == keys[:2] and all(a != b for a, b in zip(k2[2:], keys[2:]))
    t3 = toks.copy()
    t3[0] += 1                                                        # the first token: every key
    assert all(a != b for a, b in zip(k.kv_chunk_keys(t3, 256, salt=1), keys))
    assert k.kv_chunk_keys(toks[:999], 256, salt=1)[:3] == keys[:3]
    assert k.kv_chunk_keys(toks[:999], 256, salt=1)[3] != keys[3]     # a shorter last chunk differs
    # the same chunk tokens after a different prefix get a different key
    a = np.concatenate([np.full(256, 5, np.int32), np.full(256, 9, np.int32)])
    b = np.concatenate([np.full(256, 6, np.int32), np.full(256, 9, np.int32)])
    assert k.kv_chunk_keys(a, 256)[1] != k.kv_chunk_keys(b, 256)[1]


def _tier(k, slots, slot_bytes=64):
    buf = np.zeros(slots * slot_bytes + 16, np.uint8)
    off = (-buf.ctypes.data) % 16
    return k.KvTier(slot_bytes, slots, base=buf.ctypes.data + off), buf


def test_lru_eviction_and_prefix_hits(k):
    tier, buf = _tier(k, 3)
    for key in (11, 12, 13):
        s = tier.reserve(key)
        s.fill_(key)
        tier.commit(key, NO)
    assert tier.prefix_hits([11, 12, 13, 14]) == 3
    s = tier.acquire(11, NO)                 # 11 becomes most recently used
    assert int(s[0]) == 11
    tier.release(11, NO)
    tier.reserve(14).fill_(14)                # evicts the least recently used: 12
    tier.commit(14, NO)
    assert tier.prefix_hits([11, 12, 13]) == 1
    assert tier.prefix_hits([11, 13, 14]) == 3
    with pytest.raises(k.KvxError) as e:
        tier.acquire(12, NO)
    assert e.value.status == k.KVX_ENOENT
    st = tier.stats()
    assert st["entries"] == 3 and st["evictions"] == 1 and st["hits"] == 1 and st["misses"] == 1
    assert int(tier.acquire(14, NO)[5]) == 14
    tier.release(14, NO)
    tier.close()


def test_pinned_entries_are_never_evicted(k):
    tier, buf = _tier(k, 2)
    for key in (1, 2):
        tier.reserve(key)
        tier.commit(key, NO)
    tier.acquire(1, NO)                       # pinned by a reader
    tier.reserve(3)                           # evicts 2, not the pinned 1
    assert tier.prefix_hits([1]) == 1
    with pytest.raises(k.KvxError) as e:      # 1 is read, 3 is being written: nothing to evict
        tier.reserve(4)
    assert e.value.status == k.KVX_ENOMEM
    with pytest.raises(k.KvxError) as e:      # a pinned key cannot be rewritten
        tier.reserve(1)
    assert e.value.status == k.KVX_EBUSY
    assert tier.prefix_hits([3]) == 0         # reserved but not committed: not readable
    tier.commit(3, NO)
    tier.release(1, NO)
    tier.reserve(4)                           # now the least recently used (1) goes
    tier.commit(4, NO)
    assert tier.prefix_hits([1]) == 0 and tier.prefix_hits([3, 4]) == 2
    with pytest.raises(k.KvxError) as e:      # releasing more than acquired
        tier.release(4, NO)
    assert e.value.status == k.KVX_EINVAL
    tier.close()


def test_bad_tier_arguments(k):
    with pytest.raises(k.KvxError):
        k.KvTier(17, 4, base=16 * 1000)       # slot size not a multiple of 16
    with pytest.raises(k.KvxError):
        k.KvTier(64, 0, base=16 * 1000)


def test_abandoned_reservation_frees_its_key(k):
    """A writer that releases its reservation without committing gives the slot back:
    the key can be reserved again, and once the slot holds another key the abandoned
    key is not found (no stale mapping to the reused slot)."""
    tier, buf = _tier(k, 1)
    s = tier.reserve(21)
    s.fill_(21)
    tier.release(21, NO)                      # give up before committing
    assert tier.stats()["entries"] == 0
    assert tier.prefix_hits([21]) == 0
    s = tier.reserve(21)                      # the same key again
    tier.release(21, NO)
    s = tier.reserve(22)                      # the only slot now holds 22
    s.fill_(22)
    tier.commit(22, NO)
    with pytest.raises(k.KvxError) as e:
        tier.acquire(21, NO)
    assert e.value.status == k.KVX_ENOENT
    assert int(tier.acquire(22, NO)[0]) == 22
    tier.release(22, NO)


class _Model:
    """The tier's documented rules for one process with KVX_NO_STREAM: a reserve takes
    the key's own READY unpinned slot, else the first FREE slot, else the least
    recently used READY unpinned slot; commit makes READY; acquire pins a READY
    entry; release unpins, and frees a reservation given up."""

    def __init__(self, n):
        self.slots = [{"key": None, "state": "FREE", "pins": 0, "tick": 0} for _ in range(n)]
        self.clock = 0
        self.hits = self.misses = self.evictions = 0

    def find(self, key):
        for i, s in enumerate(self.slots):
            if s["state"] != "FREE" and s["key"] == key:
                return i
        return None

    def reserve(self, key):
        i = self.find(key)
        if i is not None:
            s = self.slots[i]
            if s["pins"] > 0 or s["state"] != "READY":
                return "EBUSY", None
        else:
            free = [j for j, s in enumerate(self.slots) if s["state"] == "FREE"]
            if free:
                i = free[0]
            else:
                cand = [j for j, s in enumerate(self.slots) if s["state"] == "READY" and s["pins"] == 0]
                if not cand:
                    return "ENOMEM", None
                i = min(cand, key=lambda j: self.slots[j]["tick"])
                self.evictions += 1
        self.clock += 1
        self.slots[i] = {"key": key, "state": "WRITING", "pins": 1, "tick": self.clock}
        return "OK", i

    def commit(self, key):
        i = self.find(key)
        if i is None:
            return "ENOENT"
        s = self.slots[i]
        if s["state"] != "WRITING":
            return "EINVAL"
        s["state"], s["pins"] = "READY", s["pins"] - 1
        self.clock += 1
        s["tick"] = self.clock
        return "OK"

    def reserve_many(self, keys):
        for j, key in enumerate(keys):        # in order, up to the first failure
            st, _ = self.reserve(key)
            if st != "OK":
                return st, j
        return "OK", len(keys)

    def commit_many(self, keys):
        idx = []
        for key in keys:                      # every key is checked before any is committed
            i = self.find(key)
            if i is None:
                return "ENOENT"
            if self.slots[i]["state"] != "WRITING" or i in idx:
                return "EINVAL"
            idx.append(i)
        for i in idx:
            s = self.slots[i]
            s["state"], s["pins"] = "READY", s["pins"] - 1
            self.clock += 1
            s["tick"] = self.clock
        return "OK"

    def acquire(self, key):
        i = self.find(key)
        if i is None or self.slots[i]["state"] != "READY":
            self.misses += 1
            return "ENOENT"
        s = self.slots[i]
        s["pins"] += 1
        self.clock += 1
        s["tick"] = self.clock
        self.hits += 1
        return "OK"

    def release(self, key):
        i = self.find(key)
        if i is None:
            return "ENOENT"
        s = self.slots[i]
        if s["pins"] < 1:
            return "EINVAL"
        s["pins"] -= 1
        if s["state"] == "WRITING" and s["pins"] == 0:
            s["state"] = "FREE"
        return "OK"

    def acquire_many(self, keys):
        for key in keys:                      # all or nothing
            i = self.find(key)
            if i is None or self.slots[i]["state"] != "READY":
                self.misses += 1
                return "ENOENT"
        for key in keys:
            assert self.acquire(key) == "OK"
        return "OK"

    def release_many(self, keys):
        asked = {}
        for key in keys:
            i = self.find(key)
            if i is None:
                return "ENOENT"
            asked[i] = asked.get(i, 0) + 1
            if self.slots[i]["pins"] < asked[i]:
                return "EINVAL"
        for key in keys:
            assert self.release(key) == "OK"
        return "OK"

    def prefix_hits(self, keys):
        h = 0
        for key in keys:
            i = self.find(key)
            if i is None or self.slots[i]["state"] != "READY":
                break
            h += 1
        return h


@pytest.mark.parametrize("seed,n_slots,n_keys", [(1, 5, 12), (2, 1, 3), (3, 16, 40), (4, 64, 70)])
def test_tier_follows_its_rules_under_random_operations(k, seed, n_slots, n_keys):
    """Thousands of random operations against a model of the documented rules:
    statuses, hits / misses / evictions, prefix hits, and the bytes in every slot
    handed out (each key's slot holds that key's pattern)."""
    tier, buf = _tier(k, n_slots)
    model = _Model(n_slots)
    rng = np.random.default_rng(seed)
    status = {k.KVX_EBUSY: "EBUSY", k.KVX_ENOMEM: "ENOMEM", k.KVX_ENOENT: "ENOENT", k.KVX_EINVAL: "EINVAL"}

    def call(fn, *a):
        try:
            return "OK", fn(*a)
        except k.KvxError as e:
            return status[e.status], None

    for step in range(4000):
        key = int(rng.integers(1, n_keys + 1)) * 1000003
        op = rng.choice(["reserve", "reserve_many", "commit", "commit_many", "acquire", "acquire_many", "release",
                         "release_many", "prefix"], p=[0.22, 0.08, 0.17, 0.08, 0.14, 0.06, 0.14, 0.06, 0.05])
        if op == "reserve":
            got, view = call(tier.reserve, key)
            want, _ = model.reserve(key)
            if got == "OK":
                view.fill_(key % 251)
        elif op == "commit":
            got, _ = call(tier.commit, key, NO)
            want = model.commit(key)
        elif op == "reserve_many":
            keys = [int(x) * 1000003 for x in rng.integers(1, n_keys + 1, size=int(rng.integers(0, 4)))]
            try:
                views, got = tier.reserve_many(keys), "OK"
            except k.KvxError as e:
                views, got = e.reserved, status[e.status]
            want, n_done = model.reserve_many(keys)
            assert len(views) == n_done, (step, keys)
            for kk, view in zip(keys, views):
                view.fill_(kk % 251)
        elif op == "commit_many":
            keys = [int(x) * 1000003 for x in rng.integers(1, n_keys + 1, size=int(rng.integers(0, 4)))]
            got, _ = call(tier.commit_many, keys, NO)
            want = model.commit_many(keys)
        elif op in ("acquire_many", "release_many"):
            keys = [int(x) * 1000003 for x in rng.integers(1, n_keys + 1, size=int(rng.integers(0, 4)))]
            got, views = call(getattr(tier, op), keys, NO)
            want = getattr(model, op)(keys)
            if op == "acquire_many" and got == "OK":
                for kk, view in zip(keys, views):
                    assert int(view[0]) == kk % 251 and int(view[-1]) == kk % 251, step
        elif op == "acquire":
            got, view = call(tier.acquire, key, NO)
            want = model.acquire(key)
            if got == "OK":
                assert int(view[0]) == key % 251 and int(view[-1]) == key % 251, step
        elif op == "release":
            got, _ = call(tier.release, key, NO)
            want = model.release(key)
        else:
            keys = [int(x) * 1000003 for x in rng.integers(1, n_keys + 1, size=4)]
            got, want = tier.prefix_hits(keys), model.prefix_hits(keys)
        assert got == want, (step, op, key, got, want)
    st = tier.stats()
    assert (st["hits"], st["misses"], st["evictions"]) == (model.hits, model.misses, model.evictions)
    assert st["entries"] == sum(s["state"] != "FREE" for s in model.slots)
    assert st["pinned"] == sum(s["pins"] > 0 for s in model.slots)


def test_absurd_counts_return_enomem_not_a_crash(k):
    """A batch call given a count no host could hold fails with KVX_ENOMEM (the
    library's allocation fails inside the call); no C++ exception ends the
    process, and the tier stays usable."""
    import ctypes
    tier, _ = _tier(k, 2)
    key = (ctypes.c_uint64 * 1)(7)
    slots = (ctypes.c_void_p * 1)()
    n = ctypes.c_int64()
    huge = 1 << 50
    assert k._lib.kv_tier_commit_many(tier.handle, key, huge, NO) == k.KVX_ENOMEM
    assert k._lib.kv_tier_acquire_many(tier.handle, key, huge, NO, slots) == k.KVX_ENOMEM
    assert k._lib.kv_tier_release_many(tier.handle, key, huge, NO) == k.KVX_ENOMEM
    tier.reserve(7).fill_(7)
    tier.commit(7, NO)
    assert tier.prefix_hits([7]) == 1


def test_batch_slots_as_a_chunk_list(k):
    """reserve_many / acquire_many with as_chunk_list hand back the slots'
    addresses (the same ones the tensor form views) with the slot size as each
    chunk's size, so the transfer calls' size check still applies."""
    import torch
    t, buf = _tier(k, 4, 1024)
    cl = t.reserve_many([5, 6, 7], as_chunk_list=True)
    assert isinstance(cl, k.ChunkList) and len(cl) == 3
    assert list(cl._sizes) == [1024] * 3 and len({cl[i] for i in range(3)}) == 3
    t.commit_many([5, 6, 7], stream=NO)
    views = t.acquire_many([5, 6, 7], stream=NO)
    acl = t.acquire_many([6, 7], stream=NO, as_chunk_list=True)
    assert [acl[i] for i in range(2)] == [v.data_ptr() for v in views[1:]] == [cl[1], cl[2]]
    t.release_many([5, 6, 7, 6, 7], stream=NO)
    # a 1024-byte slot holds 16 tokens of a pool with 64 bytes per token, not 17
    pool = k.KvPool([torch.empty(8 * 2 * 2 * 16 * 16, dtype=torch.uint8)], 8, 16, 2, 8, 2)
    table = torch.zeros(8, dtype=torch.int32)
    k._check_transfer_tensors(pool, table, 0, 48, 16, cl)
    with pytest.raises(ValueError, match="chunk 0 holds 1024 bytes, needs 2048"):
        k._check_transfer_tensors(pool, table, 0, 64, 32, cl)
    t.close()
