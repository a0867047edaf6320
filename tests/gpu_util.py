"""Helpers for the GPU tests: seeded pools on the device, pinned chunks, and the
oracle's expected bytes for the same inputs.  All inputs come from
paper_2609_15021_gb300.synth; all expected values come from oracle/."""
from __future__ import annotations

import hashlib

import numpy as np
import torch

import oracle
from paper_2609_15021_gb300 import synth

POISON = synth.POISON


def kvx():
    from paper_2609_15021_gb300 import kvxfer
    return kvxfer


def spec_of(pool) -> oracle.PoolSpec:
    return oracle.PoolSpec(len(pool.layers), pool.num_blocks, pool.block_tokens, pool.num_heads,
                           pool.head_dim, pool.elem_bytes, pool.layout)


def device_pool(spec: oracle.PoolSpec, host_layers=None, fill=POISON):
    """A KvPool on cuda:0, one uint8 tensor per layer, from host bytes or a fill byte."""
    k = kvx()
    if host_layers is None:
        layers = [torch.full((spec.layer_bytes,), fill, dtype=torch.uint8, device="cuda")
                  for _ in range(spec.num_layers)]
    else:
        layers = [torch.from_numpy(h).to("cuda") for h in host_layers]
    return k.KvPool(layers, spec.num_blocks, spec.block_tokens, spec.num_heads, spec.head_dim,
                    spec.elem_bytes, spec.layout, spec.pages_per_block)


def host_layers(spec: oracle.PoolSpec, seed: int):
    return [synth.splitmix64_bytes(spec.layer_bytes, seed + 104729 * l) for l in range(spec.num_layers)]


def pinned_chunks(orc, spec, t0, t1, C, extra=0, fill=POISON):
    return [torch.full((orc.chunk_bytes(spec, n) + extra,), fill, dtype=torch.uint8).pin_memory()
            for n in oracle.chunk_tokens_of(t0, t1, C)]


def device_chunks(orc, spec, t0, t1, C, extra=0, fill=POISON):
    return [torch.full((orc.chunk_bytes(spec, n) + extra,), fill, dtype=torch.uint8, device="cuda")
            for n in oracle.chunk_tokens_of(t0, t1, C)]


def np_of(t: torch.Tensor) -> np.ndarray:
    return t.detach().to("cpu").numpy().copy()


def oracle_store(orc, spec, layers_np, table, t0, t1, C):
    chunks = [np.full(orc.chunk_bytes(spec, n), POISON, np.uint8) for n in oracle.chunk_tokens_of(t0, t1, C)]
    rc, bad = orc.store(spec, layers_np, np.asarray(table, np.int32), t0, t1, C, chunks)
    assert rc == oracle.OK
    return chunks, bad


def oracle_load(orc, spec, layers_np, table, t0, t1, C, chunks_np):
    out = [l.copy() for l in layers_np]
    rc, bad = orc.load(spec, out, np.asarray(table, np.int32), t0, t1, C, chunks_np)
    assert rc == oracle.OK
    return out, bad


def sha(b) -> str:
    return hashlib.sha256(np.ascontiguousarray(b).tobytes()).hexdigest()


def first_mismatch(a: np.ndarray, b: np.ndarray):
    if a.shape != b.shape:
        return f"shape {a.shape} vs {b.shape}"
    d = np.nonzero(a != b)[0]
    return None if d.size == 0 else f"{d.size} bytes differ, first at {int(d[0])}: {a[d[0]]} vs {b[d[0]]}"


def gather_pages(layer: torch.Tensor, page_bytes: int, pages) -> np.ndarray:
    """Host copy of the listed pages of one device layer, concatenated."""
    idx = torch.as_tensor(np.asarray(pages, dtype=np.int64), device=layer.device)
    return np_of(layer.view(-1, page_bytes).index_select(0, idx)).reshape(-1)
