"""CPU oracle for the paged-KV <-> packed-host-chunk byte move.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The product path (``paper_2609_15021_gb300``) never imports it and
shares no code with it.

Two independent formulations of the same definition (paper Sec. 2.1 Table 1 and
Sec. 3.1: paged KV with HND pages, fixed-token host chunks; Sec. 3.2: store is
a gather of pages into a chunk, load the scatter back into fresh pages):

* ``kv_oracle.c``  -- nested loops with one ``memcpy`` per head row, compiled
  with gcc and called through ctypes (``store`` / ``load`` / ``state_copy``).
* ``np_oracle.py`` -- NumPy advanced indexing over the whole token range
  (``np_store`` / ``np_load``).

Both take host NumPy ``uint8`` arrays.  A pool layer is the raw bytes of
``[num_blocks][2][H][B][D*e]`` (HND) or ``[num_blocks][2][B][H][D*e]`` (NHD);
a chunk is the raw bytes of ``[L][2][T_c][H][D*e]``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass

import numpy as np

from .np_oracle import np_load, np_store, np_chunk_bytes  # noqa: F401

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "kv_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "libkvoracle.so")

HND = 0
NHD = 1

# the oracle's own status values (kv_oracle.c)
OK, EINVAL, EALIGN, ERANGE = 0, -1, -2, -3


@dataclass(frozen=True)
class PoolSpec:
    num_layers: int
    num_blocks: int
    block_tokens: int
    num_heads: int
    head_dim: int
    elem_bytes: int
    layout: int = HND
    pages_per_block: int = 1  # pages per logical block named by the table

    @property
    def row_bytes(self) -> int:
        return self.head_dim * self.elem_bytes

    @property
    def page_bytes(self) -> int:
        return 2 * self.num_heads * self.block_tokens * self.row_bytes

    @property
    def layer_bytes(self) -> int:
        return self.num_blocks * self.page_bytes


class _OrPool(ctypes.Structure):
    _fields_ = [
        ("num_layers", ctypes.c_int32),
        ("num_blocks", ctypes.c_int64),
        ("block_tokens", ctypes.c_int32),
        ("num_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("elem_bytes", ctypes.c_int32),
        ("layout", ctypes.c_int32),
        ("pages_per_block", ctypes.c_int32),
    ]


def build(src: str = _SRC, out: str = _LIB, force: bool = False) -> str:
    """Compile the C oracle with gcc into a shared library; returns its path."""
    os.makedirs(os.path.dirname(out), exist_ok=True)
    if not force and os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(src):
        return out
    tmp = out + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-pthread", "-o", tmp, src])
    os.replace(tmp, out)
    return out


class COracle:
    """ctypes front end of one compiled copy of kv_oracle.c."""

    def __init__(self, lib_path: str | None = None):
        self.lib = ctypes.CDLL(lib_path or build())
        p = ctypes.POINTER
        for name in ("oracle_store", "oracle_load"):
            f = getattr(self.lib, name)
            f.restype = ctypes.c_int
            f.argtypes = [p(_OrPool), p(ctypes.c_void_p), p(ctypes.c_int32), ctypes.c_int64,
                          ctypes.c_int64, ctypes.c_int64, ctypes.c_int32, p(ctypes.c_void_p),
                          ctypes.c_int64, ctypes.c_int, p(ctypes.c_int64)]
        self.lib.oracle_chunk_bytes.restype = ctypes.c_int64
        self.lib.oracle_chunk_bytes.argtypes = [p(_OrPool), ctypes.c_int64]
        self.lib.oracle_state_copy.restype = ctypes.c_int
        self.lib.oracle_state_copy.argtypes = [ctypes.c_int32, p(ctypes.c_void_p), ctypes.c_int64,
                                               ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p,
                                               ctypes.c_int]

    @staticmethod
    def _pool(spec: PoolSpec) -> _OrPool:
        return _OrPool(spec.num_layers, spec.num_blocks, spec.block_tokens, spec.num_heads,
                       spec.head_dim, spec.elem_bytes, spec.layout, spec.pages_per_block)

    @staticmethod
    def _ptrs(arrays) -> ctypes.Array:
        for a in arrays:
            assert a.dtype == np.uint8 and a.flags["C_CONTIGUOUS"]
        return (ctypes.c_void_p * max(1, len(arrays)))(*[a.ctypes.data for a in arrays])

    def chunk_bytes(self, spec: PoolSpec, tokens: int) -> int:
        return int(self.lib.oracle_chunk_bytes(ctypes.byref(self._pool(spec)), tokens))

    def _run(self, fn, spec, layers, table, t_begin, t_end, chunk_tokens, chunks, n_threads):
        assert len(layers) == spec.num_layers
        table = np.ascontiguousarray(table, dtype=np.int32)
        bad = ctypes.c_int64(-1)
        rc = fn(ctypes.byref(self._pool(spec)), self._ptrs(layers),
                table.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), len(table),
                t_begin, t_end, chunk_tokens, self._ptrs(chunks), len(chunks), n_threads,
                ctypes.byref(bad))
        return rc, bad.value

    def store(self, spec, layers, table, t_begin, t_end, chunk_tokens, chunks, n_threads=1):
        """Gather pool pages into ``chunks`` in place; returns (status, first bad block)."""
        return self._run(self.lib.oracle_store, spec, layers, table, t_begin, t_end,
                         chunk_tokens, chunks, n_threads)

    def load(self, spec, layers, table, t_begin, t_end, chunk_tokens, chunks, n_threads=1):
        """Scatter ``chunks`` into pool pages in place; returns (status, first bad block)."""
        return self._run(self.lib.oracle_load, spec, layers, table, t_begin, t_end,
                         chunk_tokens, chunks, n_threads)

    def state_copy(self, layers, slot_bytes, slot, host_obj, to_host):
        num_slots = layers[0].size // slot_bytes
        return int(self.lib.oracle_state_copy(len(layers), self._ptrs(layers), num_slots,
                                              slot_bytes, slot, host_obj.ctypes.data,
                                              1 if to_host else 0))


_default: COracle | None = None


def c_oracle() -> COracle:
    global _default
    if _default is None:
        _default = COracle()
    return _default


def store(*args, **kw):
    return c_oracle().store(*args, **kw)


def load(*args, **kw):
    return c_oracle().load(*args, **kw)


def chunk_tokens_of(t_begin: int, t_end: int, chunk_tokens: int) -> list[int]:
    """Tokens held by each chunk of [t_begin, t_end) (the last one may be short)."""
    out = []
    c = t_begin // chunk_tokens
    while c * chunk_tokens < t_end:
        out.append(min(chunk_tokens, t_end - c * chunk_tokens))
        c += 1
    return out
