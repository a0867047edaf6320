"""Frozen per-chunk SHA-256 of the tiny paged-KV workload (tests/golden/cfg1_tiny_hashes.txt,
written by tests/golden/make_cfg1_hashes.py from the oracle).

CPU: the oracle still produces the frozen hashes (a regression fixture for the
oracle and for the portable input generators).  GPU: the CUDA path's chunks
and restored layers hash to the same values in every transfer mode and with
both device-side engines.
"""
import importlib.util
import os

import numpy as np
import pytest

from paper_2609_15021_gb300 import synth

_HERE = os.path.dirname(os.path.abspath(__file__))
_spec = importlib.util.spec_from_file_location("make_cfg1_hashes", os.path.join(_HERE, "golden", "make_cfg1_hashes.py"))
g = importlib.util.module_from_spec(_spec)
_spec.loader.exec_module(g)


def test_oracle_reproduces_frozen_hashes():
    assert g.expected() == g.read()


def test_portable_generators():
    x = synth.normal_bf16_bytes(1 << 16, 3).view("<u2").astype(np.uint32) << 16
    v = x.view(np.float32)
    assert abs(float(v.mean())) < 0.02 and abs(float(v.std()) - 1.0) < 0.02
    assert np.all(np.abs(v) <= 6.0)                    # Irwin-Hall(12) - 6 lies in [-6, 6]
    t = synth.portable_table(64, 32, 5)
    assert len(set(t.tolist())) == 32 and t.min() >= 0 and t.max() < 64
    assert np.array_equal(synth.portable_table(64, 64, 5)[:32], t)   # a prefix of one permutation


@pytest.mark.gpu
@pytest.mark.parametrize("mode,flags", [("zerocopy", 0), ("staged", 0), ("staged", "KVX_FLAG_DEVICE_LSU"),
                                        ("device", 0), ("device", "KVX_FLAG_DEVICE_LSU")])
def test_cuda_path_matches_frozen_hashes(mode, flags):
    import torch
    from gpu_util import kvx, np_of
    k = kvx()
    want = g.read()
    layers, ta, tb = g.inputs()
    S = g.SPEC
    src = k.KvPool([torch.from_numpy(a).cuda() for a in layers], S.num_blocks, S.block_tokens, S.num_heads,
                   S.head_dim, S.elem_bytes)
    dst = k.KvPool([torch.full((S.layer_bytes,), synth.POISON, dtype=torch.uint8, device="cuda")
                    for _ in range(S.num_layers)], S.num_blocks, S.block_tokens, S.num_heads, S.head_dim,
                   S.elem_bytes)
    ta_d, tb_d = torch.from_numpy(ta).cuda(), torch.from_numpy(tb).cuda()
    cb = S.num_layers * 2 * g.C * S.num_heads * S.row_bytes
    n = g.TOKENS // g.C
    dev = "cuda" if mode == "device" else "cpu"
    chunks = [torch.full((cb,), synth.POISON, dtype=torch.uint8, device=dev) for _ in range(n)]
    if dev == "cpu":
        chunks = [c.pin_memory() for c in chunks]
    torch.cuda.synchronize()
    m = {"zerocopy": k.KVX_MODE_ZEROCOPY, "staged": k.KVX_MODE_STAGED, "device": k.KVX_MODE_AUTO}[mode]
    ctx = k.kv_ctx_create(0, store_mode=m, load_mode=m, flags=getattr(k, flags) if flags else 0)
    try:
        stream = torch.cuda.Stream()
        if mode == "device":
            k.kv_pack(ctx, src, ta_d, 0, g.TOKENS, g.C, chunks, stream=stream)
            k.kv_unpack(ctx, dst, tb_d, 0, g.TOKENS, g.C, chunks, stream=stream)
        else:
            k.kv_store(ctx, src, ta_d, 0, g.TOKENS, g.C, chunks, stream=stream)
            k.kv_load(ctx, dst, tb_d, 0, g.TOKENS, g.C, chunks, stream=stream)
        stream.synchronize()
        assert k.kv_get_device_error(ctx) == -1
    finally:
        k.kv_ctx_destroy(ctx)
    got = {f"chunk{i}": g.sha(np_of(c)) for i, c in enumerate(chunks)}
    got.update({f"restored_layer{l}": g.sha(np_of(t)) for l, t in enumerate(dst.layers)})
    assert got == want
