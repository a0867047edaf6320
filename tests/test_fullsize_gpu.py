"""Full-size 27B-class workloads (62 layers, 8 KV heads, head_dim 128, bf16, 16-token
pages, 256-token chunks) at 32k and 128k tokens, through the default context the
benchmark uses: every chunk is hashed on the host, sampled chunks are compared
with the oracle byte for byte, and sampled pages outside the load table must be
untouched.  The oracle runs on a mini-pool of exactly the pages a sampled chunk
reads (gathered from the device pool by PyTorch indexing)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import POISON, first_mismatch, gather_pages, kvx, np_of, sha
from paper_2609_15021_gb300 import synth

pytestmark = pytest.mark.gpu

L, B, H, D, E, C = 62, 16, 8, 128, 2, 256


@pytest.mark.parametrize("ctx_tokens,pool_blocks", [(32768, 4096), (131072, 10240)])
def test_fullsize_store_restore_sampled(orc, ctx_tokens, pool_blocks):
    k = kvx()
    spec = oracle.PoolSpec(L, pool_blocks, B, H, D, E, oracle.HND)
    need = 2 * L * spec.layer_bytes
    free, _ = torch.cuda.mem_get_info()
    if free < need + (4 << 30):
        pytest.skip(f"needs {need >> 30} GiB of device memory")
    n_used = ctx_tokens // B
    src_layers = [synth.normal_bf16_(torch.empty(spec.layer_bytes, dtype=torch.uint8, device="cuda"),
                                     synth.SEED + l) for l in range(L)]
    src = k.KvPool(src_layers, pool_blocks, B, H, D, E)
    dst_layers = [torch.full((spec.layer_bytes,), POISON, dtype=torch.uint8, device="cuda") for _ in range(L)]
    dst = k.KvPool(dst_layers, pool_blocks, B, H, D, E)
    ta = synth.permuted_table(pool_blocks, n_used, seed=1)
    tb = synth.permuted_table(pool_blocks, n_used, seed=2)
    n_chunks = ctx_tokens // C
    cb = orc.chunk_bytes(spec, C)
    slab = torch.empty(n_chunks * cb, dtype=torch.uint8).pin_memory()
    chunks = [slab[i * cb:(i + 1) * cb] for i in range(n_chunks)]
    ctx = k.kv_ctx_create(0)
    try:
        stream = torch.cuda.Stream()
        with torch.cuda.stream(stream):
            k.kv_store(ctx, src, torch.from_numpy(ta).cuda(), 0, ctx_tokens, C, chunks)
            k.kv_load(ctx, dst, torch.from_numpy(tb).cuda(), 0, ctx_tokens, C, chunks)
        stream.synchronize()
        assert k.kv_get_device_error(ctx) == -1
    finally:
        k.kv_ctx_destroy(ctx)
    bpc = C // B
    r = synth.rng(ctx_tokens)
    sample = sorted({0, 1, n_chunks // 2, n_chunks - 1, *map(int, r.integers(0, n_chunks, 3))})
    mini = oracle.PoolSpec(L, bpc, B, H, D, E, oracle.HND)
    ident = np.arange(bpc, dtype=np.int32)
    for c in sample:
        pages_a = ta[c * bpc:(c + 1) * bpc]
        pool_np = [gather_pages(t, spec.page_bytes, pages_a) for t in src_layers]
        want = [np.full(cb, POISON, np.uint8)]
        assert orc.store(mini, pool_np, ident, 0, C, C, want, n_threads=8)[0] == 0
        got = np_of(chunks[c])
        assert sha(got) == sha(want[0]), (c, first_mismatch(got, want[0]))
        pages_b = tb[c * bpc:(c + 1) * bpc]
        loaded = [np.full(mini.layer_bytes, POISON, np.uint8) for _ in range(L)]
        assert orc.load(mini, loaded, ident, 0, C, C, want, n_threads=8)[0] == 0
        for l in (0, 1, L // 2, L - 1):
            assert first_mismatch(gather_pages(dst_layers[l], spec.page_bytes, pages_b), loaded[l]) is None, (c, l)
    unused = np.setdiff1d(np.arange(pool_blocks), tb)
    probe = synth.rng(7).choice(unused, size=min(8, unused.size), replace=False)
    for l in (0, L - 1):
        assert np.all(gather_pages(dst_layers[l], spec.page_bytes, probe) == POISON)
