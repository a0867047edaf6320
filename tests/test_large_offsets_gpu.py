"""Pages past 4 GiB into a layer: byte offsets that do not fit 32 bits.

Each layer of the pool holds 66,048 pages of 64 KiB (4.33 GB), so a page id
of 65,536 or more starts beyond 2^32 bytes.  The load and store tables draw
most of their pages from that high end (the rest from the low end), the range
ends on a partial block, and every engine moves it: zero-copy and staged
host transfers, device pack/unpack on the default engine, on TMA copies and
on 16-byte loads/stores, and kv_store_noalloc.  HND and NHD pages, and logical
blocks of two pages (so a block-table entry past 32,767 names a page past
4 GiB), are all covered.

Every chunk byte is compared with the oracle; the restored pages with the
oracle's restore into a poisoned pool (tail slots of the partial block must
stay poisoned); and pages around the 4 GiB boundary that no table names must
be untouched.  The oracle runs on a mini-pool of the pages the tables name,
gathered by PyTorch indexing, with an identity table.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import POISON, first_mismatch, gather_pages, kvx, np_of
from paper_2609_15021_gb300 import synth

pytestmark = pytest.mark.gpu

L, B, H, D, E, C = 2, 16, 8, 128, 2, 256
N_PAGES = 66_048                       # 4,328,521,728 bytes per layer
PAGE = 2 * H * B * D * E               # 65,536
HIGH = (1 << 32) // PAGE               # first page that starts past 2^32 bytes
T1 = 4 * C - 37                        # four chunks, the last one ragged, ending inside a block


@pytest.fixture(scope="module")
def pools():
    need = 2 * L * N_PAGES * PAGE
    free, _ = torch.cuda.mem_get_info()
    if free < need + (4 << 30):
        pytest.skip(f"needs {need >> 30} GiB of device memory")
    src = [synth.normal_bf16_(torch.empty(N_PAGES * PAGE, dtype=torch.uint8, device="cuda"), 4242 + l)
           for l in range(L)]
    dst = [torch.empty(N_PAGES * PAGE, dtype=torch.uint8, device="cuda") for _ in range(L)]
    torch.cuda.synchronize()
    yield src, dst
    del src, dst
    torch.cuda.empty_cache()


def _table(n_blocks: int, P: int, seed: int) -> np.ndarray:
    """Logical-block ids, three quarters above the 4 GiB boundary, in seeded order."""
    high_block = -(-HIGH // P)
    n_hi = 3 * n_blocks // 4
    r = synth.rng(seed)
    hi = r.choice(np.arange(high_block, N_PAGES // P), size=n_hi, replace=False)
    lo = r.choice(np.arange(0, 64), size=n_blocks - n_hi, replace=False)
    return r.permutation(np.concatenate([hi, lo])).astype(np.int32)


def _pages_of(table: np.ndarray, P: int) -> np.ndarray:
    return (table.astype(np.int64)[:, None] * P + np.arange(P)).reshape(-1)


CASES = [
    ("hnd", "zerocopy"), ("hnd", "staged"), ("hnd", "device"), ("hnd", "device_tma"), ("hnd", "device_lsu"),
    ("hnd", "noalloc"), ("nhd", "zerocopy"), ("nhd", "staged"), ("nhd", "device"), ("nhd", "device_lsu"),
    ("hnd_p2", "zerocopy"), ("hnd_p2", "device"),
]


@pytest.mark.parametrize("layout,engine", CASES)
def test_pages_past_4gib(orc, pools, layout, engine):
    k = kvx()
    src_layers, dst_layers = pools
    lay = oracle.NHD if layout == "nhd" else oracle.HND
    P = 2 if layout == "hnd_p2" else 1
    n_blocks = -(-T1 // (B * P))
    ta = _table(n_blocks, P, 31 + len(layout) + len(engine))
    tb = _table(n_blocks, P, 57 + len(layout) + len(engine))
    assert _pages_of(ta, P).max() * PAGE >= 1 << 32 and _pages_of(tb, P).max() * PAGE >= 1 << 32
    for t in dst_layers:
        t.fill_(POISON)
    src = k.KvPool(src_layers, N_PAGES, B, H, D, E, lay, P)
    dst = k.KvPool(dst_layers, N_PAGES, B, H, D, E, lay, P)
    spec = oracle.PoolSpec(L, N_PAGES, B, H, D, E, lay, P)
    sizes = [orc.chunk_bytes(spec, n) for n in oracle.chunk_tokens_of(0, T1, C)]
    on_device = engine.startswith("device")
    chunks = [torch.full((n,), POISON, dtype=torch.uint8, device="cuda" if on_device else "cpu") for n in sizes]
    if not on_device:
        chunks = [c.pin_memory() for c in chunks]
    ta_d, tb_d = torch.from_numpy(ta).cuda(), torch.from_numpy(tb).cuda()
    torch.cuda.synchronize()
    flags = {"device_tma": k.KVX_FLAG_DEVICE_TMA, "device_lsu": k.KVX_FLAG_DEVICE_LSU}.get(engine, 0)
    mode = 1 if engine == "staged" else 2
    ctx = None if engine == "noalloc" else k.kv_ctx_create(0, store_mode=mode, load_mode=mode, flags=flags)
    try:
        if engine == "noalloc":
            k.kv_store_noalloc(src, ta_d, 0, T1, C, chunks)
        elif on_device:
            k.kv_pack(ctx, src, ta_d, 0, T1, C, chunks)
            k.kv_unpack(ctx, dst, tb_d, 0, T1, C, chunks)
        else:
            k.kv_store(ctx, src, ta_d, 0, T1, C, chunks)
            k.kv_load(ctx, dst, tb_d, 0, T1, C, chunks)
        torch.cuda.synchronize()
        if ctx is not None:
            assert k.kv_get_device_error(ctx) == -1
    finally:
        if ctx is not None:
            k.kv_ctx_destroy(ctx)

    n_pages = n_blocks * P
    mini = oracle.PoolSpec(L, n_pages, B, H, D, E, lay, P)
    ident = np.arange(n_blocks, dtype=np.int32)
    mini_src = [gather_pages(t, PAGE, _pages_of(ta, P)) for t in src_layers]
    want = [np.full(n, POISON, np.uint8) for n in sizes]
    assert orc.store(mini, mini_src, ident, 0, T1, C, want)[0] == oracle.OK
    for i, (c, w) in enumerate(zip(chunks, want)):
        assert first_mismatch(np_of(c), w) is None, (layout, engine, "chunk", i)
    if engine == "noalloc":
        return
    loaded = [np.full(mini.layer_bytes, POISON, np.uint8) for _ in range(L)]
    assert orc.load(mini, loaded, ident, 0, T1, C, want)[0] == oracle.OK
    for l in range(L):
        got = gather_pages(dst_layers[l], PAGE, _pages_of(tb, P))
        assert first_mismatch(got, loaded[l]) is None, (layout, engine, "layer", l)
    named = set(_pages_of(tb, P).tolist())
    edge = [p for p in (HIGH - 2, HIGH - 1, HIGH, HIGH + 1, N_PAGES - 2, N_PAGES - 1) if p not in named]
    for l in range(L):
        assert np.all(gather_pages(dst_layers[l], PAGE, edge) == POISON), (layout, engine, l)
