"""ctypes binding of libkvxfer_probe.so (``include/kvxfer_probe.h``): the
paper's copy-ordering probes and a host-link streaming probe.

These are measuring instruments for the tests and the benchmark, built as a
library of their own beside libkvxfer.so (``_build.build()`` makes both).
Importing this module without the library raises ``ImportError``.
"""
from __future__ import annotations

import ctypes
import os

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib", "libkvxfer_probe.so")

KVX_PROBE_RAW, KVX_PROBE_WAIT_THEN_COPY, KVX_PROBE_ASYNC_ON_STREAM = 0, 1, 2
KVX_PROBE_MAX_CYCLES = 4_000_000_000

# Every symbol kvxfer_probe.h declares; a test checks the library exports them all.
EXPORTED = ("kvx_probe_delayed_fill", "kvx_probe_delayed_copy", "kvx_probe_copy", "kvx_probe_stream_copy",
            "kvx_probe_last_cuda_error")


def _load():
    if not os.path.exists(_LIB_PATH):
        raise ImportError(f"libkvxfer_probe.so is not built ({_LIB_PATH}); run paper_2609_15021_gb300._build.build()")
    lib = ctypes.CDLL(_LIB_PATH)
    vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    for name, res, args in (("kvx_probe_delayed_fill", ctypes.c_int, [vp, i64, i32, i64, vp]),
                            ("kvx_probe_delayed_copy", ctypes.c_int, [vp, vp, i64, i64, vp]),
                            ("kvx_probe_copy", ctypes.c_int, [vp, vp, i64, i32, vp]),
                            ("kvx_probe_stream_copy", ctypes.c_int, [vp, vp, i64, i32, vp]),
                            ("kvx_probe_last_cuda_error", ctypes.c_int, [])):
        f = getattr(lib, name)
        f.restype, f.argtypes = res, args
    return lib


_lib = _load()


def library_path() -> str:
    return _LIB_PATH


def _check(status: int, where: str) -> None:
    from . import kvxfer
    if status != kvxfer.KVX_OK:
        msg = kvxfer.kv_status_string(status)
        if status == kvxfer.KVX_ECUDA:
            msg += f" (cuda error {_lib.kvx_probe_last_cuda_error()})"
        raise kvxfer.KvxError(status, where, msg)


def _stream(stream):
    from . import kvxfer
    return kvxfer._stream_handle(stream)


def _ptr(x) -> int:
    return x if isinstance(x, int) else x.data_ptr()


def kvx_probe_delayed_fill(dev, nbytes: int, value: int, cycles: int, stream=None) -> None:
    _check(_lib.kvx_probe_delayed_fill(_ptr(dev), nbytes, value, cycles, _stream(stream)), "kvx_probe_delayed_fill")


def kvx_probe_delayed_copy(dst, src, nbytes: int, cycles: int, stream=None) -> None:
    _check(_lib.kvx_probe_delayed_copy(_ptr(dst), _ptr(src), nbytes, cycles, _stream(stream)),
           "kvx_probe_delayed_copy")


def kvx_probe_copy(dst, src, nbytes: int, how: int, stream=None) -> None:
    _check(_lib.kvx_probe_copy(_ptr(dst), _ptr(src), nbytes, how, _stream(stream)), "kvx_probe_copy")


def kvx_probe_stream_copy(dst, src, nbytes: int, ctas: int, stream=None) -> None:
    _check(_lib.kvx_probe_stream_copy(_ptr(dst), _ptr(src), nbytes, ctas, _stream(stream)), "kvx_probe_stream_copy")
