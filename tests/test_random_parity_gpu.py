"""Seeded random sweep: the CUDA path against the oracle on many random shapes.

Each case draws a layout, page size, head count, row size (16-byte multiples
only, as the C ABI requires), element size, logical-block packing, pool and
table size, chunk size, start chunk and ragged end, then runs store and load
in one transfer mode (or device pack/unpack) and compares every byte.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import (POISON, device_chunks, device_pool, first_mismatch, host_layers, kvx, np_of, oracle_load,
                      oracle_store, pinned_chunks)
from paper_2609_15021_gb300 import synth

pytestmark = pytest.mark.gpu

N_CASES = 24


def draw(seed):
    r = synth.rng(seed)
    layout = int(r.integers(0, 2))
    B = int(r.choice([1, 2, 4, 8, 16, 32]))
    H = int(r.integers(1, 9))
    e = int(r.choice([1, 2, 4]))
    D = int(r.choice([16, 32, 64, 128, 256])) // e * 1 if e == 1 else int(r.choice([8, 16, 24, 64, 128]))
    D = max(D, 16 // e)
    if (D * e) % 16:
        D = (D * e + 15) // 16 * 16 // e
    P = int(r.choice([1, 1, 1, 2, 3]))
    L = int(r.integers(1, 5))
    n_logical = int(r.integers(2, 24))
    N = n_logical * P
    used = int(r.integers(1, n_logical + 1))
    C = B * P * int(r.integers(1, 4)) if r.random() < 0.5 else B * int(r.integers(1, 6))
    total = used * P * B
    n_chunks = -(-total // C)
    c0 = int(r.integers(0, n_chunks))
    t0 = c0 * C
    t1 = int(r.integers(t0 + 1, total + 1)) if t0 < total else total
    return oracle.PoolSpec(L, N, B, H, D, e, layout, P), used, C, t0, t1


@pytest.fixture(scope="module")
def ctxs():
    k = kvx()
    made = {m: k.kv_ctx_create(0, store_mode=m, load_mode=m) for m in (1, 2)}
    yield made
    for c in made.values():
        k.kv_ctx_destroy(c)


@pytest.mark.parametrize("seed", range(N_CASES))
def test_random_case(orc, ctxs, seed):
    k = kvx()
    spec, used, C, t0, t1 = draw(1000 + seed)
    P = spec.pages_per_block
    src_np = host_layers(spec, 5000 + seed)
    src = device_pool(spec, src_np)
    ta = synth.permuted_table(spec.num_blocks // P, used, 7 + seed)
    tb = synth.permuted_table(spec.num_blocks // P, used, 8 + seed)
    want, _ = oracle_store(orc, spec, src_np, ta, t0, t1, C)
    want_l, _ = oracle_load(orc, spec, [np.full(spec.layer_bytes, POISON, np.uint8)] * spec.num_layers,
                            tb, t0, t1, C, want)
    which = ("staged", "zerocopy", "device")[seed % 3]
    if which == "device":
        chunks = device_chunks(orc, spec, t0, t1, C)
        ctx = ctxs[1]
        k.kv_pack(ctx, src, torch.from_numpy(ta).cuda(), t0, t1, C, chunks)
    else:
        chunks = pinned_chunks(orc, spec, t0, t1, C)
        ctx = ctxs[1 if which == "staged" else 2]
        k.kv_store(ctx, src, torch.from_numpy(ta).cuda(), t0, t1, C, chunks)
    torch.cuda.synchronize()
    for i, (c, w) in enumerate(zip(chunks, want)):
        assert first_mismatch(np_of(c), w) is None, (spec, C, t0, t1, which, i)
    dst = device_pool(spec)
    fn = k.kv_unpack if which == "device" else k.kv_load
    fn(ctx, dst, torch.from_numpy(tb).cuda(), t0, t1, C, chunks)
    torch.cuda.synchronize()
    for l in range(spec.num_layers):
        assert first_mismatch(np_of(dst.layers[l]), want_l[l]) is None, (spec, C, t0, t1, which, l)
    assert k.kv_get_device_error(ctx) == -1


N_ENGINE_CASES = 36


@pytest.mark.parametrize("seed", range(N_ENGINE_CASES))
def test_random_case_engines_and_grids(orc, seed):
    """The same random shapes through every engine and launch shape: device
    pack/unpack with the default engine, TMA row/flat copies
    (KVX_FLAG_DEVICE_TMA) or 16-byte loads/stores (KVX_FLAG_DEVICE_LSU); a CTA
    cap drawn at random (a persistent grid; a ring of stages for TMA); staged
    mode with slots of one to four layers of a chunk (batches that split
    chunks by layers); zero-copy with a random cap; and kv_store_noalloc."""
    k = kvx()
    spec, used, C, t0, t1 = draw(7000 + seed)
    r = synth.rng(9000 + seed)
    P = spec.pages_per_block
    src_np = host_layers(spec, 11000 + seed)
    src = device_pool(spec, src_np)
    ta = synth.permuted_table(spec.num_blocks // P, used, 13 + seed)
    tb = synth.permuted_table(spec.num_blocks // P, used, 14 + seed)
    want, _ = oracle_store(orc, spec, src_np, ta, t0, t1, C)
    want_l, _ = oracle_load(orc, spec, [np.full(spec.layer_bytes, POISON, np.uint8)] * spec.num_layers,
                            tb, t0, t1, C, want)
    which = ("device", "staged", "zerocopy", "noalloc")[seed % 4]
    max_ctas = int(r.choice([0, 1, 3, 7, 19, 64]))
    flags = 0
    slot_bytes = 0
    mode = 2
    if which == "device":
        flags = int(r.choice([0, k.KVX_FLAG_DEVICE_TMA, k.KVX_FLAG_DEVICE_LSU]))
    elif which == "staged":
        mode = 1
        layer = 2 * min(C, t1 - t0) * spec.num_heads * spec.head_dim * spec.elem_bytes
        slot_bytes = (layer * int(r.integers(1, 5)) + 15) // 16 * 16
    ctx = None if which == "noalloc" else k.kv_ctx_create(0, store_mode=mode, load_mode=mode, max_ctas=max_ctas,
                                                         flags=flags, staging_slot_bytes=slot_bytes)
    try:
        ta_d, tb_d = torch.from_numpy(ta).cuda(), torch.from_numpy(tb).cuda()
        if which == "device":
            chunks = device_chunks(orc, spec, t0, t1, C)
            k.kv_pack(ctx, src, ta_d, t0, t1, C, chunks)
        else:
            chunks = pinned_chunks(orc, spec, t0, t1, C)
            if which == "noalloc":
                k.kv_store_noalloc(src, ta_d, t0, t1, C, chunks)
            else:
                k.kv_store(ctx, src, ta_d, t0, t1, C, chunks)
        torch.cuda.synchronize()
        what = (spec, C, t0, t1, which, max_ctas, flags, slot_bytes)
        for i, (c, w) in enumerate(zip(chunks, want)):
            assert first_mismatch(np_of(c), w) is None, (what, i)
        if which == "noalloc":
            return
        dst = device_pool(spec)
        fn = k.kv_unpack if which == "device" else k.kv_load
        fn(ctx, dst, tb_d, t0, t1, C, chunks)
        torch.cuda.synchronize()
        for l in range(spec.num_layers):
            assert first_mismatch(np_of(dst.layers[l]), want_l[l]) is None, (what, l)
        assert k.kv_get_device_error(ctx) == -1
    finally:
        if ctx is not None:
            k.kv_ctx_destroy(ctx)
