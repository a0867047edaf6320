"""Python binding of libkvxfer.so (ctypes): argument marshalling only.

Every function has the name of the C entry point it calls (``include/kvxfer.h``;
the measuring probes of ``include/kvxfer_probe.h`` live in ``probe.py``, over a
library of their own); all data movement happens in the library's CUDA
kernels and copies.  Tensors are PyTorch tensors (device memory, pinned host
buffers, streams); a C status other than ``KVX_OK`` raises ``KvxError``.

The library must have been built (``paper_2609_15021_gb300._build.build()``):
importing this module without it raises ``ImportError`` -- there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import Sequence

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib", "libkvxfer.so")

KVX_OK, KVX_EINVAL, KVX_EALIGN, KVX_ERANGE = 0, -1, -2, -3
KVX_ENOTPINNED, KVX_ECUDA, KVX_ENOMEM, KVX_EDEVICE = -4, -5, -6, -7
KVX_LAYOUT_HND, KVX_LAYOUT_NHD = 0, 1
KVX_MODE_AUTO, KVX_MODE_STAGED, KVX_MODE_ZEROCOPY = 0, 1, 2
KVX_FLAG_TIME_KERNELS, KVX_FLAG_UNORDERED, KVX_FLAG_DEVICE_TMA, KVX_FLAG_DEVICE_LSU = 0x1, 0x2, 0x4, 0x8
KVX_FLAG_NO_HOST_TOUCH = 0x10
KVX_FLAGS_ALL = 0x1F
KVX_ETIMEOUT = -10
KVX_MAX_LAYERS = 128

MODE_NAMES = {KVX_MODE_AUTO: "auto", KVX_MODE_STAGED: "staged", KVX_MODE_ZEROCOPY: "zerocopy"}

# Every symbol the headers declare; a test checks the library exports them all.
EXPORTED = (
    "kv_ctx_create", "kv_ctx_destroy", "kv_chunk_layout", "kv_store", "kv_load", "kv_pack", "kv_unpack",
    "kv_state_store", "kv_state_load", "kv_get_device_error", "kv_ctx_stats", "kv_ctx_reset_stats",
    "kv_ctx_modes", "kv_last_cuda_error", "kv_last_error_message", "kv_status_string", "kv_abi_version",
    "kv_store_noalloc",
    "kv_host_alloc", "kv_host_free", "kv_pool_view_check",
    "kv_chunk_keys", "kv_tier_create", "kv_tier_create_on", "kv_tier_destroy", "kv_tier_reserve", "kv_tier_reserve_many", "kv_tier_commit", "kv_tier_commit_many",
    "kv_tier_acquire", "kv_tier_release", "kv_tier_acquire_many", "kv_tier_release_many", "kv_tier_prefix_hits", "kv_tier_stats", "kv_fault_inject",
    "kv_tier_open_shared", "kv_tier_poll", "kv_tier_reclaim", "kv_host_alloc_numa", "kv_host_alloc_ex",
    "kv_host_pool_info", "kv_host_touch", "kv_tier_wait",
)
KVX_ENOENT, KVX_EBUSY = -8, -9
KVX_TIER_CREATE, KVX_TIER_NO_PIN = 0x1, 0x2
KVX_NO_STREAM = -1  # the handle value of KVX_NO_STREAM


class KvxError(RuntimeError):
    def __init__(self, status: int, where: str, message: str):
        super().__init__(f"{where}: {message} (status {status})")
        self.status = status


class kvx_opts(ctypes.Structure):
    _fields_ = [("store_mode", ctypes.c_int32), ("load_mode", ctypes.c_int32),
                ("staging_slots", ctypes.c_int32), ("staging_slot_bytes", ctypes.c_int64),
                ("max_ctas", ctypes.c_int32), ("flags", ctypes.c_uint32), ("wait_cycles", ctypes.c_int64)]


class kvx_pool(ctypes.Structure):
    _fields_ = [("num_layers", ctypes.c_int32), ("layer_base", ctypes.POINTER(ctypes.c_void_p)),
                ("num_blocks", ctypes.c_int64), ("block_tokens", ctypes.c_int32),
                ("num_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("elem_bytes", ctypes.c_int32), ("layout", ctypes.c_int32),
                ("pages_per_block", ctypes.c_int32)]


class kvx_host_pool_info(ctypes.Structure):
    _fields_ = [("bytes", ctypes.c_int64), ("mapped_bytes", ctypes.c_int64), ("huge_page_bytes", ctypes.c_int64),
                ("numa_node", ctypes.c_int32), ("source", ctypes.c_int32)]


class kvx_chunk_layout(ctypes.Structure):
    _fields_ = [("chunk_tokens", ctypes.c_int32), ("tokens", ctypes.c_int32),
                ("chunk_bytes", ctypes.c_int64), ("layer_stride", ctypes.c_int64),
                ("kv_stride", ctypes.c_int64), ("token_stride", ctypes.c_int64),
                ("head_stride", ctypes.c_int64), ("page_bytes", ctypes.c_int64)]


class kvx_stats(ctypes.Structure):
    _fields_ = [("kernel_launches", ctypes.c_int64), ("memcpy_calls", ctypes.c_int64),
                ("timed_launches", ctypes.c_int64 * 2), ("kernel_ms", ctypes.c_double * 2),
                ("kernel_bytes", ctypes.c_int64 * 2)]


class kvx_tier_stats(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int64) for n in ("slots", "slot_bytes", "entries", "pinned", "hits", "misses",
                                                 "evictions")]


def _declare(lib):
    P, vp, i32, i64 = ctypes.POINTER, ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    st = ctypes.c_int
    sig = {
        "kv_ctx_create": (st, [ctypes.c_int, P(kvx_opts), P(vp)]),
        "kv_ctx_destroy": (None, [vp]),
        "kv_chunk_layout": (st, [P(kvx_pool), i32, i32, P(kvx_chunk_layout)]),
        "kv_store": (st, [vp, P(kvx_pool), vp, i64, i64, i64, i32, P(vp), i64, vp]),
        "kv_load": (st, [vp, P(kvx_pool), vp, i64, i64, i64, i32, P(vp), i64, vp]),
        "kv_pack": (st, [vp, P(kvx_pool), vp, i64, i64, i64, i32, P(vp), i64, vp]),
        "kv_unpack": (st, [vp, P(kvx_pool), vp, i64, i64, i64, i32, P(vp), i64, vp]),
        "kv_state_store": (st, [vp, i32, P(vp), i64, i64, i64, vp, vp]),
        "kv_state_load": (st, [vp, i32, P(vp), i64, i64, i64, vp, vp]),
        "kv_get_device_error": (st, [vp, P(i64)]),
        "kv_ctx_stats": (st, [vp, P(kvx_stats)]),
        "kv_ctx_reset_stats": (st, [vp]),
        "kv_ctx_modes": (st, [vp, P(i32), P(i32)]),
        "kv_last_cuda_error": (ctypes.c_int, []),
        "kv_last_error_message": (ctypes.c_char_p, []),
        "kv_status_string": (ctypes.c_char_p, [ctypes.c_int]),
        "kv_abi_version": (ctypes.c_int, []),
        "kv_store_noalloc": (st, [P(kvx_pool), vp, i64, i64, i64, i32, P(vp), i64, vp, vp]),
        "kv_host_alloc": (st, [i64, P(vp)]),
        "kv_host_free": (None, [vp]),
        "kv_host_alloc_numa": (st, [i32, i64, P(vp), P(i32)]),
        "kv_host_alloc_ex": (st, [i64, i32, ctypes.c_uint32, P(vp), P(i32)]),
        "kv_host_pool_info": (st, [vp, P(kvx_host_pool_info)]),
        "kv_pool_view_check": (st, [P(kvx_pool), i32, P(i64), P(i64)]),
        "kv_chunk_keys": (st, [P(i32), i64, i32, ctypes.c_uint64, P(ctypes.c_uint64), i64]),
        "kv_tier_create": (st, [i64, i64, P(vp)]),
        "kv_tier_create_on": (st, [vp, i64, i64, P(vp)]),
        "kv_tier_open_shared": (st, [ctypes.c_char_p, i64, i64, ctypes.c_uint32, P(vp)]),
        "kv_tier_poll": (st, [vp]),
        "kv_tier_reclaim": (st, [vp, P(i64)]),
        "kv_tier_destroy": (None, [vp]),
        "kv_tier_reserve": (st, [vp, ctypes.c_uint64, P(vp)]),
        "kv_tier_reserve_many": (st, [vp, P(ctypes.c_uint64), i64, P(vp), P(i64)]),
        "kv_tier_commit": (st, [vp, ctypes.c_uint64, vp]),
        "kv_tier_commit_many": (st, [vp, P(ctypes.c_uint64), i64, vp]),
        "kv_tier_acquire": (st, [vp, ctypes.c_uint64, vp, P(vp)]),
        "kv_tier_release": (st, [vp, ctypes.c_uint64, vp]),
        "kv_tier_acquire_many": (st, [vp, P(ctypes.c_uint64), i64, vp, P(vp)]),
        "kv_tier_release_many": (st, [vp, P(ctypes.c_uint64), i64, vp]),
        "kv_tier_prefix_hits": (st, [vp, P(ctypes.c_uint64), i64, P(i64)]),
        "kv_tier_wait": (st, [vp, P(ctypes.c_uint64), i64, i64, P(i64)]),
        "kv_tier_stats": (st, [vp, P(kvx_tier_stats)]),
        "kv_fault_inject": (st, [ctypes.c_char_p, i32]),
        "kv_host_touch": (st, [P(vp), P(i64), i64]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    return lib


def load_library(path: str = _LIB_PATH):
    if not os.path.exists(path):
        raise ImportError(f"libkvxfer.so is not built ({path}); run paper_2609_15021_gb300._build.build()")
    return _declare(ctypes.CDLL(path))


_lib = load_library()


def library_path() -> str:
    return _LIB_PATH


def _check(status: int, where: str):
    if status != KVX_OK:
        msg = _lib.kv_status_string(status).decode()
        if status == KVX_ECUDA:
            msg += f" (cuda error {_lib.kv_last_cuda_error()}: {_lib.kv_last_error_message().decode()})"
        elif _lib.kv_last_error_message():
            msg += f" ({_lib.kv_last_error_message().decode()})"
        raise KvxError(status, where, msg)


def _stream_handle(stream) -> int | None:
    if stream is None:
        import torch
        raw = getattr(torch._C, "_cuda_getCurrentRawStream", None)  # the handle without a Stream object
        if raw is not None:
            return raw(torch.cuda.current_device()) or None
        return torch.cuda.current_stream().cuda_stream or None
    if isinstance(stream, int):
        return stream or None
    return stream.cuda_stream or None


def _ptr(x) -> int:
    return x if isinstance(x, int) else x.data_ptr()


def _nbytes(x) -> int:
    return x.numel() * x.element_size()


def _check_tensor(x, what: str, need_bytes: int | None = None) -> None:
    """Binding-side checks of a tensor argument that the C ABI (raw pointers) cannot make:
    contiguity and, where known, its size.  Plain integers are taken as raw pointers."""
    if isinstance(x, int):
        return
    if not x.is_contiguous():
        raise ValueError(f"{what} must be contiguous")
    if need_bytes is not None and _nbytes(x) < need_bytes:
        raise ValueError(f"{what} holds {_nbytes(x)} bytes, needs {need_bytes}")


# ---------------------------------------------------------------- pools


@dataclass
class KvPool:
    """A paged KV pool: one contiguous device buffer per layer."""

    layers: Sequence  # torch tensors (any dtype), one per layer, num_blocks * page_bytes each
    num_blocks: int
    block_tokens: int
    num_heads: int
    head_dim: int
    elem_bytes: int
    layout: int = KVX_LAYOUT_HND
    pages_per_block: int = 1  # pages per logical block named by the block table

    def __post_init__(self):
        for i, t in enumerate(self.layers):
            _check_tensor(t, f"layer {i}", self.num_blocks * self.page_bytes)
        self._bases = (ctypes.c_void_p * max(1, len(self.layers)))(*[_ptr(t) for t in self.layers])
        self._c = kvx_pool(len(self.layers), ctypes.cast(self._bases, ctypes.POINTER(ctypes.c_void_p)),
                           self.num_blocks, self.block_tokens, self.num_heads, self.head_dim,
                           self.elem_bytes, self.layout, self.pages_per_block)

    @classmethod
    def from_tensors(cls, layers, num_heads: int, block_tokens: int, layout: int = KVX_LAYOUT_HND,
                     pages_per_block: int = 1) -> "KvPool":
        """Describe a pool from per-layer tensors shaped [pages, 2, H, B, D] (HND) or
        [pages, 2, B, H, D] (NHD), or packed [blocks, P, 2, ...]; every tensor's view
        is checked against the declared layout (kv_pool_view_check)."""
        t = layers[0]
        head_dim = int(t.shape[-1])
        pages = t.numel() // (2 * num_heads * block_tokens * head_dim)
        shape_only = kvx_pool(len(layers), None, pages, block_tokens, num_heads, head_dim, t.element_size(),
                              layout, pages_per_block)
        for x in layers:  # layout first: a wrong view is named by what is wrong with it
            _view_check(shape_only, x)
        return cls(list(layers), pages, block_tokens, num_heads, head_dim, t.element_size(), layout,
                   pages_per_block)

    @property
    def row_bytes(self) -> int:
        return self.head_dim * self.elem_bytes

    @property
    def page_bytes(self) -> int:
        return 2 * self.num_heads * self.block_tokens * self.row_bytes

    @property
    def c(self) -> kvx_pool:
        return self._c


# ---------------------------------------------------------------- context


def kv_ctx_create(device: int = 0, store_mode: int = KVX_MODE_AUTO, load_mode: int = KVX_MODE_AUTO,
                  staging_slots: int = 0, staging_slot_bytes: int = 0, max_ctas: int = 0,
                  flags: int = 0, wait_cycles: int = 0) -> int:
    opts = kvx_opts(store_mode, load_mode, staging_slots, staging_slot_bytes, max_ctas, flags, wait_cycles)
    out = ctypes.c_void_p()
    _check(_lib.kv_ctx_create(device, ctypes.byref(opts), ctypes.byref(out)), "kv_ctx_create")
    return out.value


def kv_ctx_destroy(ctx: int) -> None:
    _lib.kv_ctx_destroy(ctx)


def kv_chunk_layout(pool: KvPool, chunk_tokens: int, tokens_in_chunk: int) -> kvx_chunk_layout:
    out = kvx_chunk_layout()
    _check(_lib.kv_chunk_layout(ctypes.byref(pool.c), chunk_tokens, tokens_in_chunk, ctypes.byref(out)),
           "kv_chunk_layout")
    return out


def _view_check(cpool: kvx_pool, tensor) -> None:
    nd = tensor.dim()
    shape = (ctypes.c_int64 * nd)(*tensor.shape)
    strides = (ctypes.c_int64 * nd)(*[s * tensor.element_size() for s in tensor.stride()])
    _check(_lib.kv_pool_view_check(ctypes.byref(cpool), nd, shape, strides), "kv_pool_view_check")


def kv_pool_view_check(pool: KvPool, tensor) -> None:
    """Raise KvxError unless `tensor`'s shape and strides are the layout `pool` declares."""
    _view_check(pool.c, tensor)


class ChunkList:
    """A fixed sequence of chunks (tensors, or raw addresses) with their
    addresses marshalled and their sizes read once, for transfers made again and
    again over the same chunks.  kv_store / kv_load / kv_pack / kv_unpack /
    kv_store_noalloc take it wherever they take a list of chunks; element i is
    the call's i-th chunk, as in a list, and a slice is a ChunkList over a run
    of the same chunks, sharing the marshalled addresses.  Per call only the
    sizes the range needs are compared (vectorised).  The chunks must keep
    their storage while the list is in use (it holds references to them)."""

    def __init__(self, chunks, nbytes: int | None = None, *, _parent=None, _start=0, _stop=None, _array=None):
        """chunks: tensors or raw addresses; nbytes: the size of every raw
        address's chunk, if known (tensors report their own)."""
        import numpy as np
        if _parent is not None:
            self._items, self._arr, self._sizes = _parent._items, _parent._arr, _parent._sizes
            self._start, self._n = _start, _stop - _start
            return
        if _array is not None:  # a ctypes address array the library filled in (tier slots)
            self._arr, n = _array, len(chunks)
            self._items = list(chunks)
        else:
            self._items = list(chunks)
            n = len(self._items)
            self._arr = (ctypes.c_void_p * max(1, n))(*[_ptr(c) for c in self._items])
        unknown = np.iinfo(np.int64).max
        sizes = np.full(n, unknown if nbytes is None else nbytes, dtype=np.int64)
        for i, c in enumerate(self._items):
            if not isinstance(c, int):
                _check_tensor(c, f"chunk {i}")
                sizes[i] = _nbytes(c)
        self._sizes, self._start, self._n = sizes, 0, n

    def __len__(self) -> int:
        return self._n

    def __getitem__(self, key):
        if isinstance(key, slice):
            a, b, step = key.indices(self._n)
            if step != 1:
                raise ValueError("a ChunkList slice must be contiguous")
            return ChunkList(None, _parent=self, _start=self._start + a, _stop=self._start + max(a, b))
        if not -self._n <= key < self._n:
            raise IndexError(key)
        return self._items[self._start + key % self._n]

    def _pointer(self):
        return ctypes.cast(ctypes.byref(self._arr, self._start * ctypes.sizeof(ctypes.c_void_p)),
                           ctypes.POINTER(ctypes.c_void_p))

    def _check_sizes(self, per_token: int, chunk_tokens: int, tok_begin: int, tok_end: int) -> None:
        import numpy as np
        first = tok_begin // chunk_tokens
        used = min(self._n, -(-tok_end // chunk_tokens) - first)
        if used <= 0:
            return
        need = np.full(used, per_token * chunk_tokens, dtype=np.int64)
        last = first + used - 1
        need[-1] = per_token * min(chunk_tokens, tok_end - last * chunk_tokens)
        sizes = self._sizes[self._start:self._start + used]
        bad = np.nonzero(sizes < need)[0]
        if bad.size:
            i = int(bad[0])
            raise ValueError(f"chunk {i} holds {int(sizes[i])} bytes, needs {int(need[i])}")


def _ptr_array(chunks):
    if isinstance(chunks, ChunkList):
        return chunks._pointer()
    return (ctypes.c_void_p * max(1, len(chunks)))(*[_ptr(c) for c in chunks])


def _check_transfer_tensors(pool: KvPool, block_table, tok_begin, tok_end, chunk_tokens, chunks) -> None:
    """The table is int32 and every chunk the range uses holds its bytes: a chunk
    smaller than that would be written past its end by the kernels."""
    if not isinstance(block_table, int):
        import torch
        if block_table.dtype != torch.int32:
            raise TypeError(f"block table must be int32, not {block_table.dtype}")
        _check_tensor(block_table, "block table")
    if chunk_tokens < 1 or tok_end <= tok_begin:
        return
    first = tok_begin // chunk_tokens
    per_token = pool.c.num_layers * 2 * pool.num_heads * pool.row_bytes
    if isinstance(chunks, ChunkList):
        chunks._check_sizes(per_token, chunk_tokens, tok_begin, tok_end)
        return
    for i, c in enumerate(chunks):
        start = (first + i) * chunk_tokens
        if start >= tok_end:
            break
        _check_tensor(c, f"chunk {i}", per_token * min(chunk_tokens, tok_end - start))


def _transfer(fn, name, ctx, pool, block_table, tok_begin, tok_end, chunk_tokens, chunks, stream,
              table_len=None):
    _check_transfer_tensors(pool, block_table, tok_begin, tok_end, chunk_tokens, chunks)
    arr = _ptr_array(chunks)
    n_tab = block_table.numel() if table_len is None else table_len
    _check(fn(ctx, ctypes.byref(pool.c), _ptr(block_table), n_tab, tok_begin, tok_end, chunk_tokens,
              arr, len(chunks), _stream_handle(stream)), name)


def kv_store(ctx, pool: KvPool, block_table, tok_begin: int, tok_end: int, chunk_tokens: int,
             host_chunks, stream=None, table_len: int | None = None) -> None:
    """Gather tokens [tok_begin, tok_end) into pinned host chunks, ordered on `stream`."""
    _transfer(_lib.kv_store, "kv_store", ctx, pool, block_table, tok_begin, tok_end, chunk_tokens,
              host_chunks, stream, table_len)


def kv_load(ctx, pool: KvPool, block_table, tok_begin: int, tok_end: int, chunk_tokens: int,
            host_chunks, stream=None, table_len: int | None = None) -> None:
    """Scatter pinned host chunks into the pages of `block_table`, ordered on `stream`."""
    _transfer(_lib.kv_load, "kv_load", ctx, pool, block_table, tok_begin, tok_end, chunk_tokens,
              host_chunks, stream, table_len)


def kv_pack(ctx, pool: KvPool, block_table, tok_begin: int, tok_end: int, chunk_tokens: int,
            dev_chunks, stream=None, table_len: int | None = None) -> None:
    _transfer(_lib.kv_pack, "kv_pack", ctx, pool, block_table, tok_begin, tok_end, chunk_tokens,
              dev_chunks, stream, table_len)


def kv_unpack(ctx, pool: KvPool, block_table, tok_begin: int, tok_end: int, chunk_tokens: int,
              dev_chunks, stream=None, table_len: int | None = None) -> None:
    _transfer(_lib.kv_unpack, "kv_unpack", ctx, pool, block_table, tok_begin, tok_end, chunk_tokens,
              dev_chunks, stream, table_len)


def kv_store_noalloc(pool: KvPool, block_table, tok_begin: int, tok_end: int, chunk_tokens: int,
                     host_chunks, dev_first_bad_block=None, stream=None, table_len: int | None = None) -> None:
    """kv_store for callers that cannot allocate: no context, static device staging (see kvxfer.h)."""
    _check_transfer_tensors(pool, block_table, tok_begin, tok_end, chunk_tokens, host_chunks)
    arr = _ptr_array(host_chunks)
    n_tab = block_table.numel() if table_len is None else table_len
    err = None if dev_first_bad_block is None else _ptr(dev_first_bad_block)
    _check(_lib.kv_store_noalloc(ctypes.byref(pool.c), _ptr(block_table), n_tab, tok_begin, tok_end,
                                 chunk_tokens, arr, len(host_chunks), err, _stream_handle(stream)),
           "kv_store_noalloc")


KVX_NOALLOC_SCRATCH_BYTES = 64 << 20


def kv_host_alloc(nbytes: int) -> int:
    """Exact-size page-locked, mapped host allocation (raises, never falls back to pageable)."""
    out = ctypes.c_void_p()
    _check(_lib.kv_host_alloc(nbytes, ctypes.byref(out)), "kv_host_alloc")
    return out.value


KVX_NUMA_NEAREST, KVX_NUMA_ANY = -1, -2
KVX_HOST_DRIVER, KVX_HOST_HUGE = 0x1, 0x2
KVX_HOST_SOURCE_DRIVER, KVX_HOST_SOURCE_MAPPED = 0, 1


def kv_host_pool_info(ptr: int) -> dict:
    """What backs a pool from kv_host_alloc / _numa / _ex (see kvxfer.h)."""
    out = kvx_host_pool_info()
    _check(_lib.kv_host_pool_info(ptr, ctypes.byref(out)), "kv_host_pool_info")
    return {"bytes": out.bytes, "mapped_bytes": out.mapped_bytes, "huge_page_bytes": out.huge_page_bytes,
            "numa_node": out.numa_node,
            "source": "driver" if out.source == KVX_HOST_SOURCE_DRIVER else "mapped"}


def kv_host_alloc_numa(nbytes: int, numa_node: int = KVX_NUMA_NEAREST) -> tuple[int, int]:
    """kv_host_alloc on one host NUMA node (default: the one nearest the current GPU).
    Returns (pointer, node of the first page or -1)."""
    out = ctypes.c_void_p()
    node = ctypes.c_int32(-1)
    _check(_lib.kv_host_alloc_numa(numa_node, nbytes, ctypes.byref(out), ctypes.byref(node)), "kv_host_alloc_numa")
    return out.value, node.value


def kv_host_alloc_ex(nbytes: int, numa_node: int = KVX_NUMA_ANY, flags: int = 0) -> tuple[int, int]:
    """kv_host_alloc with the placement and the allocator chosen (see kvxfer.h).
    Returns (pointer, node of the first page or -1)."""
    out = ctypes.c_void_p()
    node = ctypes.c_int32(-1)
    _check(_lib.kv_host_alloc_ex(nbytes, numa_node, flags, ctypes.byref(out), ctypes.byref(node)), "kv_host_alloc_ex")
    return out.value, node.value


def kv_host_free(ptr: int) -> None:
    _lib.kv_host_free(ptr)


def kv_host_touch(buffers) -> None:
    """Read one byte of every host page of each buffer (tensors, numpy arrays, or
    (pointer, bytes) pairs) on the library's touch threads; see kvxfer.h."""
    ptrs, sizes = [], []
    for b in buffers:
        if isinstance(b, tuple):
            p, n = b
        elif hasattr(b, "data_ptr"):
            _check_tensor(b, "buffer")
            p, n = b.data_ptr(), _nbytes(b)
        else:
            p, n = b.ctypes.data, b.nbytes
        ptrs.append(p)
        sizes.append(n)
    arr = (ctypes.c_void_p * max(1, len(ptrs)))(*ptrs)
    sz = (ctypes.c_int64 * max(1, len(sizes)))(*sizes)
    _check(_lib.kv_host_touch(arr, sz, len(ptrs)), "kv_host_touch")


class HostBuffer:
    """A kv_host_alloc allocation with a uint8 CPU tensor view (``.tensor``) over it.

    Views of ``.tensor`` keep the allocation alive; ``close()`` frees it at once
    and must only be called when no view is used any more."""

    def __init__(self, nbytes: int, numa_node: int | None = None, driver: bool = False, huge: bool = False):
        """numa_node: None for no placement, else on that node (KVX_NUMA_NEAREST:
        the node nearest the current GPU); see .numa_node.  driver: the driver's
        pinned allocator, stated (KVX_HOST_DRIVER; the default without a
        placement).  huge: the library's huge-page mapping (KVX_HOST_HUGE), for
        copy-engine transfers."""
        import torch
        self.nbytes = nbytes
        self.numa_node = None
        if driver and (huge or numa_node is not None):
            raise ValueError("the driver's allocator takes no NUMA placement and no huge pages")
        if driver:
            self.ptr, _ = kv_host_alloc_ex(nbytes, KVX_NUMA_ANY, KVX_HOST_DRIVER)
        elif huge:
            self.ptr, node = kv_host_alloc_ex(nbytes, KVX_NUMA_ANY if numa_node is None else numa_node, KVX_HOST_HUGE)
            self.numa_node = None if numa_node is None else node
        elif numa_node is None:
            self.ptr = kv_host_alloc(nbytes)
        else:
            self.ptr, self.numa_node = kv_host_alloc_numa(nbytes, numa_node)
        raw = (ctypes.c_uint8 * nbytes).from_address(self.ptr)
        raw._owner = self  # the tensor holds `raw`, `raw` holds this buffer
        self.tensor = torch.frombuffer(raw, dtype=torch.uint8, count=nbytes)

    def info(self) -> dict:
        return kv_host_pool_info(self.ptr)

    def close(self):
        if self.ptr:
            self.tensor = None
            kv_host_free(self.ptr)
            self.ptr = 0

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class StateLayers:
    """Per-layer recurrent-state buffers (one device tensor, or raw pointer, per layer)
    with their base pointers marshalled once, for state copies made every turn.
    kv_state_store / kv_state_load take this or a plain sequence of tensors."""

    def __init__(self, layers):
        self.layers = list(layers)
        self._arr = _ptr_array(self.layers)

    def __len__(self) -> int:
        return len(self.layers)


def _layer_array(layers):
    return layers._arr if isinstance(layers, StateLayers) else _ptr_array(layers)


def kv_state_store(ctx, layers, num_slots: int, slot_bytes: int, slot: int, host_obj, stream=None) -> None:
    _check(_lib.kv_state_store(ctx, len(layers), _layer_array(layers), num_slots, slot_bytes, slot, _ptr(host_obj),
                               _stream_handle(stream)), "kv_state_store")


def kv_state_load(ctx, layers, num_slots: int, slot_bytes: int, slot: int, host_obj, stream=None) -> None:
    _check(_lib.kv_state_load(ctx, len(layers), _layer_array(layers), num_slots, slot_bytes, slot, _ptr(host_obj),
                              _stream_handle(stream)), "kv_state_load")


def kv_get_device_error(ctx) -> int:
    v = ctypes.c_int64(-1)
    _check(_lib.kv_get_device_error(ctx, ctypes.byref(v)), "kv_get_device_error")
    return v.value


def kv_ctx_stats(ctx) -> dict:
    s = kvx_stats()
    _check(_lib.kv_ctx_stats(ctx, ctypes.byref(s)), "kv_ctx_stats")
    out = {}
    for name, _ in kvx_stats._fields_:
        v = getattr(s, name)
        out[name] = list(v) if isinstance(v, ctypes.Array) else v
    return out


def kv_ctx_reset_stats(ctx) -> None:
    _check(_lib.kv_ctx_reset_stats(ctx), "kv_ctx_reset_stats")


def kv_ctx_modes(ctx) -> tuple[int, int]:
    a, b = ctypes.c_int32(), ctypes.c_int32()
    _check(_lib.kv_ctx_modes(ctx, ctypes.byref(a), ctypes.byref(b)), "kv_ctx_modes")
    return a.value, b.value


def kv_abi_version() -> int:
    return _lib.kv_abi_version()


def kv_status_string(status: int) -> str:
    return _lib.kv_status_string(status).decode()


# ---------------------------------------------------------------- convenience


def kv_fault_inject(point: str | None, after_calls: int = 0) -> None:
    """Make the (after_calls+1)-th next CUDA call at `point` fail (host side); None disarms."""
    _check(_lib.kv_fault_inject(point.encode() if point else None, after_calls), "kv_fault_inject")


def kv_chunk_keys(tokens, chunk_tokens: int, salt: int = 0) -> list[int]:
    """Prefix-chained keys of the chunks of a token sequence (a sequence of ints)."""
    import numpy as np
    t = np.ascontiguousarray(np.asarray(tokens, dtype=np.int32))
    n = -(-len(t) // chunk_tokens) if len(t) else 0
    keys = (ctypes.c_uint64 * max(1, n))()
    _check(_lib.kv_chunk_keys(t.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), len(t), chunk_tokens,
                              salt & (2**64 - 1), keys, n), "kv_chunk_keys")
    return list(keys[:n])


class KvTier:
    """The shared host tier (see kvxfer.h): fixed chunk slots in one pinned pool, LRU."""

    def __init__(self, slot_bytes: int = 0, n_slots: int = 0, base: int | None = None,
                 shared_name: str | None = None, create: bool = False, pin: bool = True):
        """Private tier over a new pinned pool (or over `base`), or, with shared_name, a tier
        shared by the processes of this host (create it, or open an existing one)."""
        out = ctypes.c_void_p()
        if shared_name is not None:
            flags = (KVX_TIER_CREATE if create else 0) | (0 if pin else KVX_TIER_NO_PIN)
            _check(_lib.kv_tier_open_shared(shared_name.encode(), slot_bytes, n_slots, flags, ctypes.byref(out)),
                   "kv_tier_open_shared")
        elif base is None:
            _check(_lib.kv_tier_create(slot_bytes, n_slots, ctypes.byref(out)), "kv_tier_create")
        else:
            _check(_lib.kv_tier_create_on(base, slot_bytes, n_slots, ctypes.byref(out)), "kv_tier_create_on")
        self.handle = out.value
        if not slot_bytes:
            slot_bytes = self.stats()["slot_bytes"]
        self.slot_bytes = slot_bytes

    def poll(self):
        _check(_lib.kv_tier_poll(self.handle), "kv_tier_poll")

    def close(self):
        if self.handle:
            _lib.kv_tier_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _slot_tensor(self, ptr: int):
        import torch
        raw = (ctypes.c_uint8 * self.slot_bytes).from_address(ptr)
        raw._owner = self  # a slot view keeps the tier (and its pool) alive
        return torch.frombuffer(raw, dtype=torch.uint8, count=self.slot_bytes)

    @staticmethod
    def _stream(stream):
        if stream == KVX_NO_STREAM:
            return ctypes.c_void_p(KVX_NO_STREAM & (2**64 - 1))
        return _stream_handle(stream)

    def reserve(self, key: int):
        """Host tensor view of the slot to write `key` into (pinned until commit)."""
        out = ctypes.c_void_p()
        _check(_lib.kv_tier_reserve(self.handle, key, ctypes.byref(out)), "kv_tier_reserve")
        return self._slot_tensor(out.value)

    def _slots(self, out, n: int, as_chunk_list: bool):
        if as_chunk_list:
            return ChunkList([out[j] for j in range(n)], self.slot_bytes, _array=out)
        return [self._slot_tensor(out[j]) for j in range(n)]

    def reserve_many(self, keys, as_chunk_list: bool = False):
        """Slots for `keys`, reserved in order under one lock: host tensor views,
        or with as_chunk_list a ChunkList of the slots' addresses (no tensor per
        slot; what the transfer calls take).  If a key cannot be reserved,
        KvxError is raised with `.reserved`: the slots of the keys before it,
        which stay reserved (commit or release them)."""
        n = len(keys)
        arr = (ctypes.c_uint64 * max(1, n))(*keys)
        out = (ctypes.c_void_p * max(1, n))()
        done = ctypes.c_int64()
        status = _lib.kv_tier_reserve_many(self.handle, arr, n, out, ctypes.byref(done))
        slots = self._slots(out, done.value, as_chunk_list)
        try:
            _check(status, "kv_tier_reserve_many")
        except KvxError as e:
            e.reserved = slots
            raise
        return slots

    def commit(self, key: int, stream=None):
        _check(_lib.kv_tier_commit(self.handle, key, self._stream(stream)), "kv_tier_commit")

    def commit_many(self, keys, stream=None):
        arr = (ctypes.c_uint64 * max(1, len(keys)))(*keys)
        _check(_lib.kv_tier_commit_many(self.handle, arr, len(keys), self._stream(stream)), "kv_tier_commit_many")

    def acquire(self, key: int, stream=None):
        out = ctypes.c_void_p()
        _check(_lib.kv_tier_acquire(self.handle, key, self._stream(stream), ctypes.byref(out)), "kv_tier_acquire")
        return self._slot_tensor(out.value)

    def release(self, key: int, stream=None):
        _check(_lib.kv_tier_release(self.handle, key, self._stream(stream)), "kv_tier_release")

    def acquire_many(self, keys, stream=None, as_chunk_list: bool = False):
        """Slots of committed `keys`, pinned, `stream` waiting for their commits:
        host tensor views, or with as_chunk_list a ChunkList of their addresses."""
        arr = (ctypes.c_uint64 * max(1, len(keys)))(*keys)
        out = (ctypes.c_void_p * max(1, len(keys)))()
        _check(_lib.kv_tier_acquire_many(self.handle, arr, len(keys), self._stream(stream), out),
               "kv_tier_acquire_many")
        return self._slots(out, len(keys), as_chunk_list)

    def release_many(self, keys, stream=None):
        arr = (ctypes.c_uint64 * max(1, len(keys)))(*keys)
        _check(_lib.kv_tier_release_many(self.handle, arr, len(keys), self._stream(stream)), "kv_tier_release_many")

    def prefix_hits(self, keys) -> int:
        arr = (ctypes.c_uint64 * max(1, len(keys)))(*keys)
        out = ctypes.c_int64()
        _check(_lib.kv_tier_prefix_hits(self.handle, arr, len(keys), ctypes.byref(out)), "kv_tier_prefix_hits")
        return out.value

    def wait(self, keys, timeout_s: float = 60.0) -> int:
        """Wait until every key is readable (see kv_tier_wait); returns len(keys), or
        raises KvxError (KVX_ETIMEOUT) with `.hits`, the readable prefix at the end."""
        arr = (ctypes.c_uint64 * max(1, len(keys)))(*keys)
        out = ctypes.c_int64()
        status = _lib.kv_tier_wait(self.handle, arr, len(keys), int(timeout_s * 1e9), ctypes.byref(out))
        try:
            _check(status, "kv_tier_wait")
        except KvxError as e:
            e.hits = out.value
            raise
        return out.value

    def reclaim(self) -> int:
        """Drop what processes that no longer exist left pinned or half written; slots changed."""
        out = ctypes.c_int64(0)
        _check(_lib.kv_tier_reclaim(self.handle, ctypes.byref(out)), "kv_tier_reclaim")
        return out.value

    def stats(self) -> dict:
        s = kvx_tier_stats()
        _check(_lib.kv_tier_stats(self.handle, ctypes.byref(s)), "kv_tier_stats")
        return {n: getattr(s, n) for n, _ in kvx_tier_stats._fields_}


class KvTransfer:
    """Owns one kvx_ctx; the methods forward to the functions above."""

    def __init__(self, device: int = 0, **opts):
        self.ctx = kv_ctx_create(device, **opts)

    def close(self):
        if self.ctx:
            kv_ctx_destroy(self.ctx)
            self.ctx = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def store(self, pool, table, t0, t1, chunk_tokens, host_chunks, stream=None):
        kv_store(self.ctx, pool, table, t0, t1, chunk_tokens, host_chunks, stream)

    def load(self, pool, table, t0, t1, chunk_tokens, host_chunks, stream=None):
        kv_load(self.ctx, pool, table, t0, t1, chunk_tokens, host_chunks, stream)

    def pack(self, pool, table, t0, t1, chunk_tokens, dev_chunks, stream=None):
        kv_pack(self.ctx, pool, table, t0, t1, chunk_tokens, dev_chunks, stream)

    def unpack(self, pool, table, t0, t1, chunk_tokens, dev_chunks, stream=None):
        kv_unpack(self.ctx, pool, table, t0, t1, chunk_tokens, dev_chunks, stream)

    def device_error(self) -> int:
        return kv_get_device_error(self.ctx)

    def stats(self) -> dict:
        return kv_ctx_stats(self.ctx)

    def modes(self) -> tuple[int, int]:
        return kv_ctx_modes(self.ctx)
