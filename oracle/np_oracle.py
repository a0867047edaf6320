"""Second, independent formulation of the oracle in NumPy advanced indexing.

TEST INFRASTRUCTURE ONLY (see the package docstring).

Where ``kv_oracle.c`` walks (chunk, layer, kv, token, head) and copies one row
at a time, this module views every pool layer as a 5-D array, picks all tokens
of the range at once with the block table (paper Sec. 3.1: a logical block maps
to pages of the pool; Sec. 3.2: store gathers them, load scatters them back)
and moves the [kv] axis in front of the token axis to obtain the chunk layout
[layer][kv][token][head][row].
"""
from __future__ import annotations

import numpy as np

HND = 0
NHD = 1


def _view(layer: np.ndarray, spec) -> np.ndarray:
    if spec.layout == HND:
        shape = (spec.num_blocks, 2, spec.num_heads, spec.block_tokens, spec.row_bytes)
    else:
        shape = (spec.num_blocks, 2, spec.block_tokens, spec.num_heads, spec.row_bytes)
    return layer.reshape(shape)


def _token_coords(table, t_begin, t_end, block_tokens, pages_per_block=1):
    """Page and slot of every token: the table names logical blocks of
    pages_per_block consecutive pages (Sec. 3.1's packed sub-pages)."""
    t = np.arange(t_begin, t_end, dtype=np.int64)
    kernel_page = t // block_tokens
    logical = np.asarray(table, dtype=np.int64)[kernel_page // pages_per_block]
    pages = logical * pages_per_block + kernel_page % pages_per_block
    slots = t % block_tokens
    return pages, slots


def np_chunk_bytes(spec, tokens: int) -> int:
    return spec.num_layers * 2 * tokens * spec.num_heads * spec.row_bytes


def _gather_layer(view, spec, pages, slots) -> np.ndarray:
    """All tokens of one layer, shaped [kv][token][head][row]."""
    if spec.layout == HND:
        g = view[pages, :, :, slots, :]      # advanced axes 0 and 3 -> [token][kv][head][row]
    else:
        g = view[pages, :, slots, :, :]      # advanced axes 0 and 2 -> [token][kv][head][row]
    return np.transpose(g, (1, 0, 2, 3))


def np_store(spec, layers, table, t_begin, t_end, chunk_tokens):
    """Return the list of packed chunks (uint8 arrays) for tokens [t_begin, t_end)."""
    pages, slots = _token_coords(table, t_begin, t_end, spec.block_tokens, max(1, spec.pages_per_block))
    per_layer = [_gather_layer(_view(layers[l], spec), spec, pages, slots)
                 for l in range(spec.num_layers)]
    allk = np.stack(per_layer)                # [L][kv][T][H][row]
    out = []
    start = t_begin
    while start < t_end:
        stop = min((start // chunk_tokens + 1) * chunk_tokens, t_end)
        part = allk[:, :, start - t_begin:stop - t_begin]
        out.append(np.ascontiguousarray(part).reshape(-1))
        start = stop
    return out


def np_load(spec, layers, table, t_begin, t_end, chunk_tokens, chunks):
    """Scatter ``chunks`` into copies of ``layers``; returns the new layers."""
    pages, slots = _token_coords(table, t_begin, t_end, spec.block_tokens, max(1, spec.pages_per_block))
    H, R, L = spec.num_heads, spec.row_bytes, spec.num_layers
    parts = []
    start, i = t_begin, 0
    while start < t_end:
        stop = min((start // chunk_tokens + 1) * chunk_tokens, t_end)
        parts.append(chunks[i][: L * 2 * (stop - start) * H * R].reshape(L, 2, stop - start, H, R))
        start, i = stop, i + 1
    allk = np.concatenate(parts, axis=2) if parts else np.zeros((L, 2, 0, H, R), np.uint8)
    out = []
    for l in range(L):
        new = layers[l].copy()
        view = _view(new, spec)
        vals = np.transpose(allk[l], (1, 0, 2, 3))   # [token][kv][head][row]
        if spec.layout == HND:
            view[pages, :, :, slots, :] = vals
        else:
            view[pages, :, slots, :, :] = vals
        out.append(new)
    return out
