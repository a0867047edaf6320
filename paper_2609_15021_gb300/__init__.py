"""GB300-native paged-KV <-> pinned-host-chunk transfer (libkvxfer).

The compute path is ``libkvxfer.so`` (hand-written CUDA for sm_103a behind a C
ABI, ``include/kvxfer.h``); ``kvxfer`` is its ctypes binding.  Import the
binding explicitly (``from paper_2609_15021_gb300 import kvxfer``): it raises
ImportError when the library has not been built.
"""
__all__ = ["kvxfer", "synth"]
