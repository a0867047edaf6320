"""Bit-exact parity of the CUDA path with the CPU oracle, through the C ABI.

Sizes are small enough for the oracle to finish in well under a second each,
yet span several warp units, several kernel launches (more chunks than one
launch carries), staging batches that split a chunk by layers, ragged last
pages and short last chunks, a non-zero start, both page layouts, the fast
(power-of-two row) and generic row paths, and both transfer modes.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import (POISON, device_chunks, device_pool, first_mismatch, host_layers, kvx, np_of,
                      oracle_load, oracle_store, pinned_chunks, spec_of)
from paper_2609_15021_gb300 import synth

pytestmark = pytest.mark.gpu

HND, NHD = oracle.HND, oracle.NHD

# name: (L, N, B, H, D, e, layout, n_used, C, first_chunk, t1 short by)
CASES = {
    "tiny_cfg_hnd": (2, 64, 16, 2, 64, 2, HND, 32, 256, 0, 0),
    "tiny_cfg_nhd": (2, 64, 16, 2, 64, 2, NHD, 32, 256, 0, 0),
    "ragged_tail_offset_start": (3, 40, 16, 4, 64, 2, HND, 37, 64, 1, 5),
    "ragged_tail_nhd": (3, 40, 16, 4, 64, 2, NHD, 37, 64, 2, 9),
    "rows_48B_generic": (2, 20, 4, 3, 24, 2, HND, 17, 8, 0, 3),
    "rows_1KiB_generic": (2, 12, 8, 2, 256, 4, HND, 10, 16, 0, 1),
    # rows of 2 KiB (the widest a tensor map describes: 256 eight-byte elements) and of
    # 4 KiB (beyond it: the TMA engine falls back to row copies, the default to loads/stores)
    "rows_2KiB_esz8": (2, 16, 4, 1, 512, 4, HND, 12, 8, 0, 1),
    "rows_4KiB_no_tensor_map": (1, 10, 2, 1, 1024, 4, HND, 8, 4, 0, 1),
    "rows_16B_16_heads": (1, 30, 2, 16, 16, 1, HND, 25, 4, 2, 1),
    "fp8_1568_token_chunks": (4, 120, 32, 4, 256, 1, HND, 103, 1568, 0, 7),
    "many_chunks_three_launches": (1, 300, 1, 1, 8, 2, HND, 300, 2, 0, 1),
    "one_token": (2, 8, 16, 8, 128, 2, HND, 1, 256, 0, 15),
    "27b_shape_two_chunks": (62, 48, 16, 8, 128, 2, HND, 40, 256, 0, 3),
    # logical blocks of packed pages (Sec. 3.1): 49 pages of 32 tokens per 1,568-token block;
    # n_used counts logical blocks, N pages
    "paper_logical_blocks_49": (4, 49 * 6, 32, 4, 256, 1, HND, 5, 1568, 1, 100, 49),
    "logical_blocks_4_nhd_ragged": (3, 4 * 20, 16, 2, 64, 2, NHD, 17, 96, 2, 7, 4),
    # the most layers a pool description holds (KVX_MAX_LAYERS)
    "max_layers_128": (128, 24, 16, 2, 64, 2, HND, 20, 64, 1, 5),
    "max_layers_128_nhd_logical": (128, 2 * 12, 16, 2, 64, 2, NHD, 10, 64, 1, 5, 2),
}

MODES = {"staged": 1, "zerocopy": 2}


def _unpack(case):
    """(L, N, B, H, D, e, layout, n_used, C, c0, short, pages per logical block)"""
    return tuple(case) + (1,) * (12 - len(case))


def _range(case):
    L, N, B, H, D, e, layout, n_used, C, c0, short, ppb = _unpack(case)
    return c0 * C, n_used * ppb * B - short


@pytest.fixture(scope="module")
def ctxs():
    k = kvx()
    made = {}

    def get(mode, slot_bytes=0, flags=0, max_ctas=0):
        key = (mode, slot_bytes, flags, max_ctas)
        if key not in made:
            made[key] = k.kv_ctx_create(0, store_mode=mode, load_mode=mode, staging_slot_bytes=slot_bytes,
                                        flags=flags, max_ctas=max_ctas)
        return made[key]

    yield get
    for c in made.values():
        k.kv_ctx_destroy(c)


def _run_case(orc, ctx, case, stream):
    k = kvx()
    L, N, B, H, D, e, layout, n_used, C, c0, short, ppb = _unpack(case)
    spec = oracle.PoolSpec(L, N, B, H, D, e, layout, ppb)
    t0, t1 = _range(case)
    src_np = host_layers(spec, seed=hash(case) % 100000)
    src = device_pool(spec, src_np)
    ta = synth.permuted_table(N // ppb, n_used, seed=11)
    tb = synth.permuted_table(N // ppb, n_used, seed=12)
    ta_d = torch.from_numpy(ta).cuda()
    tb_d = torch.from_numpy(tb).cuda()
    extra = 48
    host = pinned_chunks(orc, spec, t0, t1, C, extra=extra)
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        k.kv_store(ctx, src, ta_d, t0, t1, C, host)
    stream.synchronize()
    want, _ = oracle_store(orc, spec, src_np, ta, t0, t1, C)
    assert len(want) == len(host)
    for i, (h, w) in enumerate(zip(host, want)):
        got = np_of(h)
        assert first_mismatch(got[:-extra], w) is None, (i, first_mismatch(got[:-extra], w))
        assert np.all(got[-extra:] == POISON), f"chunk {i}: bytes written past its end"
    # load into a poisoned pool through another table
    dst = device_pool(spec)
    with torch.cuda.stream(stream):
        k.kv_load(ctx, dst, tb_d, t0, t1, C, host)
    stream.synchronize()
    poisoned = [np.full(spec.layer_bytes, POISON, np.uint8) for _ in range(L)]
    want_l, _ = oracle_load(orc, spec, poisoned, tb, t0, t1, C, want)
    for l in range(L):
        assert first_mismatch(np_of(dst.layers[l]), want_l[l]) is None, (l, first_mismatch(np_of(dst.layers[l]), want_l[l]))
    assert k.kv_get_device_error(ctx) == -1


@pytest.mark.parametrize("mode", list(MODES))
@pytest.mark.parametrize("name", list(CASES))
def test_store_load_parity(orc, ctxs, name, mode):
    stream = torch.cuda.Stream()  # a non-blocking pool stream, as in the paper's setting
    _run_case(orc, ctxs(MODES[mode]), CASES[name], stream)


@pytest.mark.parametrize("name", list(CASES))
def test_store_load_parity_staged_tma(orc, ctxs, name):
    """Staged mode with the TMA bulk-copy kernel packing into / unpacking from the ring."""
    _run_case(orc, ctxs(1, 0, kvx().KVX_FLAG_DEVICE_TMA), CASES[name], torch.cuda.Stream())


@pytest.mark.parametrize("name", ["ragged_tail_offset_start", "27b_shape_two_chunks", "fp8_1568_token_chunks"])
def test_staged_one_layer_per_slot(orc, ctxs, name):
    """Staging slots that hold exactly one layer of a full chunk: every chunk is split
    into per-layer pieces, and the ring of slots is reused many times per call."""
    case = CASES[name]
    L, N, B, H, D, e, layout, n_used, C, c0, short = case
    slot = 2 * C * H * D * e
    _run_case(orc, ctxs(1, slot), case, torch.cuda.Stream())


# Engines of the device-side launches: by default one warp (LSU) or CTA (TMA)
# per unit; "_capped" grids of 7 CTAs make every warp or CTA stride over many
# units (the TMA kernel then runs its ring of shared-memory stages).
ENGINES = {"lsu": ("KVX_FLAG_DEVICE_LSU", 0), "default": (None, 0), "tma": ("KVX_FLAG_DEVICE_TMA", 0),
           "lsu_capped": ("KVX_FLAG_DEVICE_LSU", 7), "default_capped": (None, 7),
           "tma_capped": ("KVX_FLAG_DEVICE_TMA", 7)}


@pytest.mark.parametrize("engine", list(ENGINES))
@pytest.mark.parametrize("name", ["tiny_cfg_hnd", "ragged_tail_nhd", "rows_48B_generic", "many_chunks_three_launches",
                                  "27b_shape_two_chunks", "paper_logical_blocks_49", "logical_blocks_4_nhd_ragged",
                                  "rows_16B_16_heads", "one_token", "rows_1KiB_generic", "rows_2KiB_esz8",
                                  "rows_4KiB_no_tensor_map", "fp8_1568_token_chunks"])
def test_device_pack_unpack_parity(orc, ctxs, name, engine):
    k = kvx()
    case = CASES[name]
    L, N, B, H, D, e, layout, n_used, C, c0, short, ppb = _unpack(case)
    spec = oracle.PoolSpec(L, N, B, H, D, e, layout, ppb)
    t0, t1 = _range(case)
    src_np = host_layers(spec, seed=77)
    src = device_pool(spec, src_np)
    ta = synth.permuted_table(N // ppb, n_used, seed=21)
    tb = synth.permuted_table(N // ppb, n_used, seed=22)
    extra = 32
    dev = device_chunks(orc, spec, t0, t1, C, extra=extra)
    flag, max_ctas = ENGINES[engine]
    ctx = ctxs(1, 0, getattr(k, flag) if flag else 0, max_ctas)
    k.kv_pack(ctx, src, torch.from_numpy(ta).cuda(), t0, t1, C, dev)
    torch.cuda.synchronize()
    assert k.kv_get_device_error(ctx) == -1   # no bad entry, no expired wait (KVX_ETIMEOUT raises)
    want, _ = oracle_store(orc, spec, src_np, ta, t0, t1, C)
    for i, (d, w) in enumerate(zip(dev, want)):
        got = np_of(d)
        assert first_mismatch(got[:-extra], w) is None, i
        assert np.all(got[-extra:] == POISON)
    dst = device_pool(spec)
    k.kv_unpack(ctx, dst, torch.from_numpy(tb).cuda(), t0, t1, C, dev)
    torch.cuda.synchronize()
    want_l, _ = oracle_load(orc, spec, [np.full(spec.layer_bytes, POISON, np.uint8) for _ in range(L)],
                            tb, t0, t1, C, want)
    for l in range(L):
        assert first_mismatch(np_of(dst.layers[l]), want_l[l]) is None, l
    assert k.kv_get_device_error(ctx) == -1


def test_tma_out_of_range_pages(orc, ctxs):
    """The TMA engine applies the same bad-entry rule (zeros on pack, skip on unpack)."""
    k = kvx()
    spec = oracle.PoolSpec(2, 16, 16, 2, 64, 2, HND)
    src_np = host_layers(spec, seed=15)
    src = device_pool(spec, src_np)
    table = synth.permuted_table(16, 12, seed=13)
    table[3] = 16
    table[10] = -1
    C, t0, t1 = 64, 0, 12 * 16
    dev = device_chunks(orc, spec, t0, t1, C)
    ctx = ctxs(1, 0, k.KVX_FLAG_DEVICE_TMA)
    k.kv_pack(ctx, src, torch.from_numpy(table).cuda(), t0, t1, C, dev)
    torch.cuda.synchronize()
    assert k.kv_get_device_error(ctx) == 3
    want, bad = oracle_store(orc, spec, src_np, table, t0, t1, C)
    assert bad == 3
    for d, w in zip(dev, want):
        assert first_mismatch(np_of(d), w) is None
    dst = device_pool(spec)
    k.kv_unpack(ctx, dst, torch.from_numpy(table).cuda(), t0, t1, C, dev)
    torch.cuda.synchronize()
    assert k.kv_get_device_error(ctx) == 3
    want_l, _ = oracle_load(orc, spec, [np.full(spec.layer_bytes, POISON, np.uint8) for _ in range(2)],
                            table, t0, t1, C, want)
    for l in range(2):
        assert first_mismatch(np_of(dst.layers[l]), want_l[l]) is None


@pytest.mark.parametrize("mode", list(MODES))
def test_out_of_range_pages_reported(orc, ctxs, mode):
    """Entries outside [0, num_blocks) skip their page and report the lowest bad logical block;
    every other byte still matches the oracle (which applies the same rule)."""
    k = kvx()
    spec = oracle.PoolSpec(2, 16, 16, 2, 64, 2, HND)
    src_np = host_layers(spec, seed=5)
    src = device_pool(spec, src_np)
    table = synth.permuted_table(16, 12, seed=3)
    table[5] = 16      # one past the last page
    table[9] = -3
    C, t0, t1 = 64, 0, 12 * 16
    host = pinned_chunks(orc, spec, t0, t1, C)
    ctx = ctxs(MODES[mode])
    k.kv_store(ctx, src, torch.from_numpy(table).cuda(), t0, t1, C, host)
    torch.cuda.synchronize()
    assert k.kv_get_device_error(ctx) == 5
    assert k.kv_get_device_error(ctx) == -1  # cleared by the query
    want, bad = oracle_store(orc, spec, src_np, table, t0, t1, C)
    assert bad == 5
    for h, w in zip(host, want):
        assert first_mismatch(np_of(h), w) is None


@pytest.mark.parametrize("mode", list(MODES))
def test_empty_range_is_a_no_op(orc, ctxs, mode):
    k = kvx()
    spec = oracle.PoolSpec(1, 4, 16, 1, 64, 2, HND)
    src = device_pool(spec, host_layers(spec, 1))
    host = [torch.full((4096,), POISON, dtype=torch.uint8).pin_memory()]
    table = torch.arange(4, dtype=torch.int32, device="cuda")
    ctx = ctxs(MODES[mode])
    k.kv_store(ctx, src, table, 32, 32, 32, host)
    k.kv_load(ctx, src, table, 32, 32, 32, [])
    torch.cuda.synchronize()
    assert np.all(np_of(host[0]) == POISON)


def test_back_to_back_calls_reuse_slots(orc, ctxs):
    """store A -> load B -> store B with no host synchronisation in between, through
    one-layer staging slots: slot reuse across calls must respect every event edge."""
    k = kvx()
    spec = oracle.PoolSpec(4, 64, 16, 4, 64, 2, HND)
    C, n_used = 128, 60
    t0, t1 = 0, n_used * 16 - 3
    src_np = host_layers(spec, 99)
    src = device_pool(spec, src_np)
    ta = torch.from_numpy(synth.permuted_table(64, n_used, 1)).cuda()
    tb = torch.from_numpy(synth.permuted_table(64, n_used, 2)).cuda()
    ctx = ctxs(1, 2 * C * 4 * 64 * 2)
    h1 = pinned_chunks(orc, spec, t0, t1, C)
    h2 = pinned_chunks(orc, spec, t0, t1, C)
    dst = device_pool(spec)
    torch.cuda.synchronize()  # the poisoned pool was filled on the default stream
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        for _ in range(3):
            k.kv_store(ctx, src, ta, t0, t1, C, h1)
            k.kv_load(ctx, dst, tb, t0, t1, C, h1)
            k.kv_store(ctx, dst, tb, t0, t1, C, h2)
    s.synchronize()
    want, _ = oracle_store(orc, spec, src_np, ta.cpu().numpy(), t0, t1, C)
    for a, b, w in zip(h1, h2, want):
        assert first_mismatch(np_of(a), w) is None
        assert first_mismatch(np_of(b), w) is None


@pytest.mark.parametrize("which", ["legacy_default", "per_thread", "torch_default"])
def test_special_streams(orc, ctxs, which):
    k = kvx()
    spec = oracle.PoolSpec(2, 32, 16, 2, 64, 2, HND)
    src_np = host_layers(spec, 3)
    src = device_pool(spec, src_np)
    table = synth.permuted_table(32, 20, 4)
    host = pinned_chunks(orc, spec, 0, 320, 64)
    stream = {"legacy_default": 0, "per_thread": 2, "torch_default": torch.cuda.default_stream().cuda_stream}[which]
    k.kv_store(ctxs(1), src, torch.from_numpy(table).cuda(), 0, 320, 64, host, stream=stream)
    torch.cuda.synchronize()
    want, _ = oracle_store(orc, spec, src_np, table, 0, 320, 64)
    for h, w in zip(host, want):
        assert first_mismatch(np_of(h), w) is None


@pytest.mark.parametrize("mode", list(MODES))
@pytest.mark.parametrize("L,slots,sb", [(5, 4, 16 * 128 * 128 * 4 // 64), (3, 4, 81968), (120, 4, 16016),
                                         (1, 4, 16), (48, 4, 1097728)])
def test_state_snapshot_parity(orc, ctxs, mode, L, slots, sb):
    """Recurrent-state snapshots: slot 3 of L layers out to host, then into slot 1.
    Slot sizes that are not multiples of the copy unit make units cross layer
    ends; 120 layers take two launches; 48 x 1,097,728 B is the hybrid model's."""
    k = kvx()
    layers_np = [synth.splitmix64_bytes(slots * sb, 900 + l) for l in range(L)]
    layers = [torch.from_numpy(a).cuda() for a in layers_np]
    obj = torch.full((L * sb,), POISON, dtype=torch.uint8).pin_memory()
    ctx = ctxs(MODES[mode])
    k.kv_state_store(ctx, layers, slots, sb, 3, obj)
    torch.cuda.synchronize()
    want = np.full(L * sb, POISON, np.uint8)
    assert orc.state_copy(layers_np, sb, 3, want, True) == 0
    assert first_mismatch(np_of(obj), want) is None
    dst_np = [np.full(slots * sb, POISON, np.uint8) for _ in range(L)]
    dst = [torch.from_numpy(a).cuda() for a in dst_np]
    k.kv_state_load(ctx, dst, slots, sb, 1, obj)
    torch.cuda.synchronize()
    assert orc.state_copy(dst_np, sb, 1, want, False) == 0
    for a, b in zip(dst, dst_np):
        assert first_mismatch(np_of(a), b) is None


def test_two_contexts_at_once_and_one_context_from_two_threads(orc):
    """Replica A stores while replica B restores other chunks (two contexts, two
    streams, overlapping on the GPU); then one context serves two host threads at
    once.  Every result must match the oracle."""
    import threading
    k = kvx()
    L, N, B, H, D, e, C = 3, 64, 16, 4, 64, 2, 128
    spec = oracle.PoolSpec(L, N, B, H, D, e, HND)
    T = 40 * B - 3
    src_np, other_np = host_layers(spec, 501), host_layers(spec, 502)
    ta, tb = synth.permuted_table(N, 40, 31), synth.permuted_table(N, 40, 32)
    want_a, _ = oracle_store(orc, spec, src_np, ta, 0, T, C)
    want_b, _ = oracle_store(orc, spec, other_np, ta, 0, T, C)
    restored_b, _ = oracle_load(orc, spec, [np.full(spec.layer_bytes, POISON, np.uint8)] * L, tb, 0, T, C, want_b)
    ta_d, tb_d = torch.from_numpy(ta).cuda(), torch.from_numpy(tb).cuda()

    # two contexts at once
    src = device_pool(spec, src_np)
    dst_b = device_pool(spec)
    out_a = pinned_chunks(orc, spec, 0, T, C)
    in_b = [torch.from_numpy(w).pin_memory() for w in want_b]
    ca, cb_ = k.kv_ctx_create(0), k.kv_ctx_create(0)
    try:
        sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
        torch.cuda.synchronize()
        k.kv_store(ca, src, ta_d, 0, T, C, out_a, stream=sa)
        k.kv_load(cb_, dst_b, tb_d, 0, T, C, in_b, stream=sb)
        torch.cuda.synchronize()
        assert k.kv_get_device_error(ca) == -1 and k.kv_get_device_error(cb_) == -1
    finally:
        k.kv_ctx_destroy(ca)
        k.kv_ctx_destroy(cb_)
    for got, w in zip(out_a, want_a):
        assert first_mismatch(np_of(got)[:w.size], w) is None
    for l in range(L):
        assert first_mismatch(np_of(dst_b.layers[l]), restored_b[l]) is None

    # one context, two host threads, each with its own stream and buffers
    ctx = k.kv_ctx_create(0)
    pools = [device_pool(spec, src_np), device_pool(spec, other_np)]
    outs = [pinned_chunks(orc, spec, 0, T, C) for _ in range(2)]
    errors = []

    def worker(i):
        try:
            s = torch.cuda.Stream()
            for _ in range(5):
                k.kv_store(ctx, pools[i], ta_d, 0, T, C, outs[i], stream=s)
            s.synchronize()
        except Exception as ex:  # reported below
            errors.append(ex)

    try:
        torch.cuda.synchronize()
        threads = [threading.Thread(target=worker, args=(i,)) for i in range(2)]
        for t in threads:
            t.start()
        for t in threads:
            t.join(timeout=120)
        assert not errors, errors
        assert k.kv_get_device_error(ctx) == -1
    finally:
        k.kv_ctx_destroy(ctx)
    for got, w in zip(outs[0], want_a):
        assert first_mismatch(np_of(got)[:w.size], w) is None
    for got, w in zip(outs[1], want_b):
        assert first_mismatch(np_of(got)[:w.size], w) is None


@pytest.mark.parametrize("touch", [True, False])
def test_calls_after_idle_time(orc, touch):
    """A context idle for more than 1 s reads one byte per host page of its
    chunks before a transfer (unless KVX_FLAG_NO_HOST_TOUCH): the store and the
    restore that follow idle gaps, across several host buffers and a short last
    chunk, still match the oracle byte for byte."""
    import time
    k = kvx()
    spec = oracle.PoolSpec(4, 96, 16, 8, 128, 2, oracle.HND)
    C, n_used = 256, 72
    T = n_used * 16 - 9
    src_np = host_layers(spec, 31)
    src, dst = device_pool(spec, src_np), device_pool(spec)
    ta, tb = synth.permuted_table(96, n_used, 32), synth.permuted_table(96, n_used, 33)
    ta_d, tb_d = torch.from_numpy(ta).cuda(), torch.from_numpy(tb).cuda()
    host = pinned_chunks(orc, spec, 0, T, C)
    ctx = k.kv_ctx_create(0, flags=0 if touch else k.KVX_FLAG_NO_HOST_TOUCH)
    torch.cuda.synchronize()  # the poisoned pool was filled on the default stream
    try:
        s = torch.cuda.Stream()
        time.sleep(1.1)
        k.kv_store(ctx, src, ta_d, 0, T, C, host, stream=s)
        s.synchronize()
        time.sleep(1.1)
        k.kv_load(ctx, dst, tb_d, 0, T, C, host, stream=s)
        s.synchronize()
        assert k.kv_get_device_error(ctx) == -1
    finally:
        k.kv_ctx_destroy(ctx)
    want, _ = oracle_store(orc, spec, src_np, ta, 0, T, C)
    for c, w in enumerate(want):
        assert first_mismatch(np_of(host[c]), w) is None, c
    loaded, _ = oracle_load(orc, spec, [np.full(spec.layer_bytes, POISON, np.uint8)] * 4, tb, 0, T, C, want)
    for l in range(4):
        assert first_mismatch(np_of(dst.layers[l]), loaded[l]) is None, l


@pytest.mark.parametrize("mode", list(MODES))
def test_tok_end_limit_with_logical_blocks(orc, ctxs, mode):
    """The range rule of kvxfer.h: tok_end <= table_len * P * B with P pages per
    logical block.  Exactly at the limit a store, a restore and the allocation-free
    store move every token bit-exactly; one token beyond it each returns KVX_ERANGE
    and leaves the chunks and the pool untouched."""
    k = kvx()
    P, B, C, n_log = 4, 16, 128, 17
    spec = oracle.PoolSpec(2, P * 20, B, 2, 64, 2, HND, P)
    src_np = host_layers(spec, seed=515)
    src = device_pool(spec, src_np)
    ta = synth.permuted_table(20, n_log, seed=516)
    tb = synth.permuted_table(20, n_log, seed=517)
    ta_d, tb_d = torch.from_numpy(ta).cuda(), torch.from_numpy(tb).cuda()
    limit = n_log * P * B
    ctx = ctxs(MODES[mode])
    # one token beyond: rejected before anything is enqueued
    full = oracle.chunk_tokens_of(0, limit + 1, C)
    host = [torch.full((orc.chunk_bytes(spec, n),), POISON, dtype=torch.uint8).pin_memory() for n in full]
    dst = device_pool(spec)
    for call in (lambda: k.kv_store(ctx, src, ta_d, 0, limit + 1, C, host),
                 lambda: k.kv_load(ctx, dst, tb_d, 0, limit + 1, C, host),
                 lambda: k.kv_store_noalloc(src, ta_d, 0, limit + 1, C, host)):
        with pytest.raises(k.KvxError) as ex:
            call()
        assert ex.value.status == k.KVX_ERANGE
    torch.cuda.synchronize()
    assert all(np.all(np_of(h) == POISON) for h in host)
    assert all(np.all(np_of(l) == POISON) for l in dst.layers)
    # exactly at the limit
    want, _ = oracle_store(orc, spec, src_np, ta, 0, limit, C)
    for store in (lambda h: k.kv_store(ctx, src, ta_d, 0, limit, C, h),
                  lambda h: k.kv_store_noalloc(src, ta_d, 0, limit, C, h)):
        got = pinned_chunks(orc, spec, 0, limit, C)
        store(got)
        torch.cuda.synchronize()
        for g, w in zip(got, want):
            assert first_mismatch(np_of(g), w) is None
    k.kv_load(ctx, dst, tb_d, 0, limit, C, got)
    torch.cuda.synchronize()
    poisoned = [np.full(spec.layer_bytes, POISON, np.uint8) for _ in range(2)]
    want_l, _ = oracle_load(orc, spec, poisoned, tb, 0, limit, C, want)
    for l in range(2):
        assert first_mismatch(np_of(dst.layers[l]), want_l[l]) is None
    assert k.kv_get_device_error(ctx) == -1


@pytest.mark.parametrize("mode", list(MODES))
def test_chunk_lists_move_what_lists_move(orc, ctxs, mode):
    """kv_store / kv_load / kv_pack / kv_unpack / kv_store_noalloc given a
    ChunkList, or a slice of one for a range that starts at a later chunk,
    move the same bytes the oracle gives for the whole range."""
    k = kvx()
    spec = oracle.PoolSpec(3, 64, 16, 4, 64, 2, HND)
    C, n_used, c0 = 64, 50, 3
    T, t0 = n_used * 16 - 5, c0 * C
    src_np = host_layers(spec, 808)
    src, dst, dst2 = device_pool(spec, src_np), device_pool(spec), device_pool(spec)
    ta, tb = synth.permuted_table(64, n_used, 81), synth.permuted_table(64, n_used, 82)
    ta_d, tb_d = torch.from_numpy(ta).cuda(), torch.from_numpy(tb).cuda()
    host = k.ChunkList(pinned_chunks(orc, spec, 0, T, C))
    host2 = k.ChunkList(pinned_chunks(orc, spec, 0, T, C))
    devc = k.ChunkList(device_chunks(orc, spec, 0, T, C))
    ctx = ctxs(MODES[mode])
    torch.cuda.synchronize()
    k.kv_store(ctx, src, ta_d, 0, t0, C, host[:c0])
    k.kv_store(ctx, src, ta_d, t0, T, C, host[c0:])
    k.kv_pack(ctx, src, ta_d, 0, T, C, devc)
    k.kv_store_noalloc(src, ta_d, 0, T, C, host2)
    torch.cuda.synchronize()
    want, _ = oracle_store(orc, spec, src_np, ta, 0, T, C)
    for i, w in enumerate(want):
        for name, cl in (("store", host), ("pack", devc), ("noalloc", host2)):
            assert first_mismatch(np_of(cl[i]), w) is None, (name, i)
    k.kv_load(ctx, dst, tb_d, t0, T, C, host[c0:])
    k.kv_load(ctx, dst, tb_d, 0, t0, C, host[:c0])
    k.kv_unpack(ctx, dst2, tb_d, 0, T, C, devc)
    torch.cuda.synchronize()
    want_l, _ = oracle_load(orc, spec, [np.full(spec.layer_bytes, POISON, np.uint8)] * spec.num_layers,
                            tb, 0, T, C, want)
    for l in range(spec.num_layers):
        assert first_mismatch(np_of(dst.layers[l]), want_l[l]) is None, ("load", l)
        assert first_mismatch(np_of(dst2.layers[l]), want_l[l]) is None, ("unpack", l)
    assert k.kv_get_device_error(ctx) == -1
