"""The C-ABI library without a GPU: it loads, exports every declared symbol, and
its host-only logic (chunk geometry, argument checks) behaves as documented."""
import ctypes
import os
import re
import time

import pytest

import oracle
from paper_2609_15021_gb300 import _build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def k():
    _build.build()
    from paper_2609_15021_gb300 import kvxfer
    return kvxfer


def declared_functions(header=None):
    names = set()
    for h in os.listdir(os.path.join(ROOT, "include")):
        if not h.endswith(".h") or (header and h != header):
            continue
        text = open(os.path.join(ROOT, "include", h)).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        for m in re.finditer(r"^\s*(?:const\s+)?[A-Za-z_][\w\s\*]*?\b([a-z]\w*)\s*\(", text, flags=re.M):
            names.add(m.group(1))
    return names - {"if", "while", "for", "return", "sizeof"}


def test_exports_every_declared_symbol(k):
    declared = declared_functions("kvxfer.h")
    assert "kv_store" in declared and "kv_store_noalloc" in declared
    lib = ctypes.CDLL(k.library_path())
    missing = [n for n in sorted(declared) if not hasattr(lib, n)]
    assert not missing, missing
    assert set(k.EXPORTED) == declared


def test_probe_library_exports_its_header_and_the_transfer_library_no_probe(k):
    """The measuring probes live in libkvxfer_probe.so only."""
    from paper_2609_15021_gb300 import probe
    declared = declared_functions("kvxfer_probe.h")
    assert "kvx_probe_copy" in declared and "kvx_probe_stream_copy" in declared
    lib = ctypes.CDLL(probe.library_path())
    missing = [n for n in sorted(declared) if not hasattr(lib, n)]
    assert not missing, missing
    assert set(probe.EXPORTED) == declared
    product = ctypes.CDLL(k.library_path())
    assert not [n for n in declared if hasattr(product, n)]
    assert declared_functions() == declared | set(k.EXPORTED)


def declared_constants():
    """{name: value} of every numeric #define and enum member KVX_* in include/*.h."""
    out = {}
    for h in os.listdir(os.path.join(ROOT, "include")):
        if not h.endswith(".h"):
            continue
        text = re.sub(r"/\*.*?\*/", "", open(os.path.join(ROOT, "include", h)).read(), flags=re.S)
        for m in re.finditer(r"#define\s+(KVX_\w+)\s+\(?(-?(?:0x[0-9A-Fa-f]+|\d+))(?:u|ll|LL)?\b(?:\s*<<\s*(\d+))?",
                             text):
            v = int(m.group(2), 0)
            out[m.group(1)] = v << int(m.group(3)) if m.group(3) else v
        for m in re.finditer(r"\b(KVX_[A-Z0-9_]+)\s*=\s*(-?\d+)", text):
            out[m.group(1)] = int(m.group(2))
    return out


def test_binding_constants_match_headers(k):
    from paper_2609_15021_gb300 import probe
    declared = declared_constants()
    for name in ("KVX_OK", "KVX_ETIMEOUT", "KVX_FLAG_DEVICE_LSU", "KVX_FLAGS_ALL", "KVX_PROBE_MAX_CYCLES",
                 "KVX_NOALLOC_SCRATCH_BYTES", "KVX_TIER_NO_PIN", "KVX_MODE_ZEROCOPY"):
        assert name in declared, name
    def binding(n):
        return probe if n.startswith("KVX_PROBE_") else k
    mismatched = {n: (v, getattr(binding(n), n)) for n, v in declared.items()
                  if hasattr(binding(n), n) and getattr(binding(n), n) != v}
    assert not mismatched, mismatched
    missing = sorted(n for n in declared if not hasattr(binding(n), n) and n not in ("KVX_ABI_VERSION",))
    assert not missing, missing
    flags = [v for n, v in declared.items() if n.startswith("KVX_FLAG_")]
    assert declared["KVX_FLAGS_ALL"] == sum(flags) and all(v & (v - 1) == 0 for v in flags)


def test_abi_version_and_strings(k):
    assert k.kv_abi_version() == 3
    assert k.kv_status_string(k.KVX_ENOTPINNED) == "host buffer is not page-locked"
    assert k.kv_status_string(123) == "unknown status"


def _pool(k, L=62, N=4096, B=16, H=8, D=128, e=2, layout=0):
    return k.KvPool([0] * L, N, B, H, D, e, layout)


@pytest.mark.parametrize("shape", [(62, 4096, 16, 8, 128, 2), (2, 64, 16, 2, 64, 2), (16, 100, 32, 4, 256, 1),
                                   (3, 7, 4, 3, 24, 2)])
@pytest.mark.parametrize("tokens_frac", [1.0, 0.5, 0.0])
def test_chunk_layout_matches_oracle_geometry(k, orc, shape, tokens_frac):
    L, N, B, H, D, e = shape
    C = 4 * B
    T = int(C * tokens_frac)
    lay = k.kv_chunk_layout(_pool(k, *shape), C, T)
    spec = oracle.PoolSpec(L, N, B, H, D, e)
    assert lay.chunk_bytes == orc.chunk_bytes(spec, T)
    assert lay.head_stride == D * e
    assert lay.token_stride == H * D * e
    assert lay.kv_stride == T * H * D * e
    assert lay.layer_stride == 2 * T * H * D * e
    assert lay.page_bytes == spec.page_bytes


def test_chunk_layout_errors(k):
    with pytest.raises(k.KvxError) as e:
        k.kv_chunk_layout(_pool(k, B=16), 24, 24)      # C not a multiple of B
    assert e.value.status == k.KVX_EALIGN
    with pytest.raises(k.KvxError) as e:
        k.kv_chunk_layout(_pool(k, D=12, e=1), 32, 32)  # 12-byte rows
    assert e.value.status == k.KVX_EALIGN
    with pytest.raises(k.KvxError) as e:
        k.kv_chunk_layout(_pool(k), 256, 257)           # more tokens than the chunk
    assert e.value.status == k.KVX_EINVAL
    with pytest.raises(k.KvxError) as e:
        k.kv_chunk_layout(_pool(k, L=k.KVX_MAX_LAYERS + 1), 256, 1)
    assert e.value.status == k.KVX_EINVAL
    with pytest.raises(k.KvxError) as e:
        k.kv_chunk_layout(_pool(k, layout=7), 256, 1)
    assert e.value.status == k.KVX_EINVAL


def test_pool_view_check(k):
    """Layout views are checked against the declaration (paper Sec. 3.1: an NHD/HND
    mismatch must be rejected, not silently mis-copied)."""
    import torch
    N, H, B, D = 12, 8, 16, 128
    hnd = torch.empty(N, 2, H, B, D, dtype=torch.bfloat16)
    nhd = torch.empty(N, 2, B, H, D, dtype=torch.bfloat16)
    pool = k.KvPool.from_tensors([hnd, hnd], H, B, k.KVX_LAYOUT_HND)
    assert (pool.num_blocks, pool.head_dim, pool.elem_bytes) == (N, D, 2)
    k.KvPool.from_tensors([nhd], H, B, k.KVX_LAYOUT_NHD)
    with pytest.raises(k.KvxError) as e:                  # NHD bytes declared HND
        k.KvPool.from_tensors([nhd], H, B, k.KVX_LAYOUT_HND)
    assert e.value.status == k.KVX_EINVAL and "dimension 3 (tokens per page) is 8" in str(e.value)
    with pytest.raises(k.KvxError) as e:                  # an NHD tensor viewed with HND's shape
        k.KvPool.from_tensors([nhd.transpose(2, 3)], H, B, k.KVX_LAYOUT_HND)
    assert "stride" in str(e.value)
    packed = torch.empty(N // 3, 3, 2, H, B, D, dtype=torch.bfloat16)   # 3 pages per logical block
    k.KvPool.from_tensors([packed], H, B, k.KVX_LAYOUT_HND, pages_per_block=3)
    with pytest.raises(k.KvxError) as e:
        k.KvPool.from_tensors([packed], H, B, k.KVX_LAYOUT_HND, pages_per_block=4)
    assert e.value.status in (k.KVX_EINVAL, k.KVX_EALIGN)
    with pytest.raises(k.KvxError):
        k.kv_pool_view_check(pool, torch.empty(N, 2, H, B * D, dtype=torch.bfloat16))


def test_null_context_rejected_before_cuda(k):
    pool = _pool(k)
    arr = (ctypes.c_void_p * 1)(0)
    for fn in (k._lib.kv_store, k._lib.kv_load, k._lib.kv_pack, k._lib.kv_unpack):
        assert fn(None, ctypes.byref(pool.c), 0, 0, 0, 0, 256, arr, 0, None) == k.KVX_EINVAL
    assert k._lib.kv_get_device_error(None, None) == k.KVX_EINVAL
    assert k._lib.kv_ctx_create(0, None, None) == k.KVX_EINVAL


def test_bad_options_rejected(k):
    for kw in ({"store_mode": 9}, {"staging_slots": 1}, {"staging_slot_bytes": 17}, {"max_ctas": -1},
               {"flags": 0x100}, {"flags": k.KVX_FLAG_DEVICE_TMA | k.KVX_FLAG_DEVICE_LSU}):
        with pytest.raises(k.KvxError) as e:
            k.kv_ctx_create(0, **kw)
        assert e.value.status == k.KVX_EINVAL


def test_no_gpu_context_reports_cuda_error(k):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    with pytest.raises(k.KvxError) as e:
        k.kv_ctx_create(0)
    assert e.value.status in (k.KVX_ECUDA, k.KVX_EINVAL)


def test_binding_rejects_what_raw_pointers_cannot_show(k):
    """The C ABI takes raw pointers; the binding checks what only the tensors know:
    the table's dtype, contiguity, and that each chunk and layer holds its bytes."""
    import torch
    L, N, B, H, D, e, C = 2, 8, 16, 2, 64, 2, 32
    page = 2 * H * B * D * e
    with pytest.raises(ValueError, match="layer 1 holds"):
        k.KvPool([torch.empty(N * page, dtype=torch.uint8), torch.empty(N * page - 16, dtype=torch.uint8)],
                 N, B, H, D, e)
    pool = k.KvPool([torch.empty(N * page, dtype=torch.uint8) for _ in range(L)], N, B, H, D, e)
    cb = L * 2 * C * H * D * e
    chunks = [torch.empty(cb, dtype=torch.uint8) for _ in range(2)]
    with pytest.raises(TypeError, match="int32"):
        k.kv_store(0, pool, torch.zeros(4, dtype=torch.int64), 0, 64, C, chunks)
    table = torch.zeros(4, dtype=torch.int32)
    with pytest.raises(ValueError, match="chunk 1 holds"):
        k.kv_load(0, pool, table, 0, 64, C, [chunks[0], chunks[1][:-16]])
    with pytest.raises(ValueError, match="contiguous"):
        k.kv_pack(0, pool, table, 0, 64, C, [chunks[0], torch.empty(2, cb, dtype=torch.uint8)[:, 0]])
    # a short last chunk only needs its own tokens' bytes
    short = torch.empty(L * 2 * 10 * H * D * e, dtype=torch.uint8)
    k._check_transfer_tensors(pool, table, 0, 42, C, [chunks[0], short])
    with pytest.raises(ValueError, match="chunk 1 holds"):
        k._check_transfer_tensors(pool, table, 0, 43, C, [chunks[0], short])


def test_state_layers_marshalled_once(k):
    """StateLayers builds the layer-pointer array once; the state copies pass it
    through unchanged (a null context is rejected before any device call)."""
    ptrs = [0x10000, 0x20000, 0x30000]
    sl = k.StateLayers(ptrs)
    assert len(sl) == 3
    arr = k._layer_array(sl)
    assert [arr[i] for i in range(3)] == ptrs and k._layer_array(sl) is arr
    assert [k._layer_array(ptrs)[i] for i in range(3)] == ptrs  # a plain sequence: marshalled per call
    for fn in (k.kv_state_store, k.kv_state_load):
        for layers in (sl, ptrs):
            with pytest.raises(k.KvxError) as e:
                fn(None, layers, 2, 4096, 0, 0x40000, stream=0)
            assert e.value.status == k.KVX_EINVAL


def test_chunk_list_marshals_once_and_checks_sizes_per_call(k):
    """A ChunkList checks contiguity once, keeps the chunks' addresses, slices
    without copying them, and per call rejects a chunk too small for the
    tokens it must hold, with the same message as a plain list."""
    import torch
    L, N, B, H, D, e, C = 2, 8, 16, 2, 64, 2, 32
    pool = k.KvPool([torch.empty(N * 2 * H * B * D * e, dtype=torch.uint8) for _ in range(L)], N, B, H, D, e)
    cb = L * 2 * C * H * D * e
    items = [torch.empty(cb, dtype=torch.uint8) for _ in range(4)] + [torch.empty(cb // 2, dtype=torch.uint8)]
    cl = k.ChunkList(items)
    table = torch.zeros(8, dtype=torch.int32)
    assert len(cl) == 5 and cl[1] is items[1] and cl[-1] is items[4]
    ptrs = k._ptr_array(cl)
    assert [ptrs[i] for i in range(5)] == [t.data_ptr() for t in items]
    k._check_transfer_tensors(pool, table, 0, 4 * C + 16, C, cl)        # a short last chunk: half a chunk
    for chunks in (cl, items):
        with pytest.raises(ValueError, match="chunk 4 holds 16384 bytes, needs 17408"):
            k._check_transfer_tensors(pool, table, 0, 4 * C + 17, C, chunks)
    sub = cl[1:3]
    assert len(sub) == 2 and sub[0] is items[1]
    sp = k._ptr_array(sub)
    assert (sp[0], sp[1]) == (items[1].data_ptr(), items[2].data_ptr())
    k._check_transfer_tensors(pool, table, C, 3 * C, C, sub)            # chunks 1 and 2 of the range
    assert len(cl[4:9]) == 1 and len(cl[3:1]) == 0
    with pytest.raises(ValueError, match="contiguous"):
        cl[::2]
    with pytest.raises(ValueError, match="contiguous"):
        k.ChunkList([torch.empty(2, cb, dtype=torch.uint8)[:, 0]])
    raw = k.ChunkList([16 * 1000, 16 * 2000])                           # raw addresses: size unknown, not checked
    k._check_transfer_tensors(pool, table, 0, 2 * C, C, raw)
    with pytest.raises(k.KvxError) as ex:                                # reaches the C ABI: no context
        k.kv_store(None, pool, table, 0, 2 * C, C, cl[:2], stream=0)
    assert ex.value.status == k.KVX_EINVAL


def test_host_alloc_numa_arguments(k):
    import torch
    out = ctypes.c_void_p()
    node = ctypes.c_int32(5)
    for numa, n in ((0, 0), (-2, 4096), (1 << 20, 4096)):
        assert k._lib.kv_host_alloc_numa(numa, n, ctypes.byref(out), ctypes.byref(node)) == k.KVX_EINVAL
    assert k._lib.kv_host_alloc_numa(0, 4096, None, None) == k.KVX_EINVAL
    assert k._lib.kv_host_alloc_numa(1000, 4096, ctypes.byref(out), None) == k.KVX_EINVAL   # no such node
    assert out.value is None and node.value == -1
    if not torch.cuda.is_available():                   # node 0 exists; pinning needs a GPU
        assert k._lib.kv_host_alloc_numa(0, 4096, ctypes.byref(out), None) == k.KVX_ECUDA
        assert out.value is None
    ex = k._lib.kv_host_alloc_ex
    assert ex(4096, k.KVX_NUMA_ANY, 0x4, ctypes.byref(out), None) == k.KVX_EINVAL          # unknown flag
    assert ex(4096, 0, k.KVX_HOST_DRIVER, ctypes.byref(out), None) == k.KVX_EINVAL         # driver + node
    assert ex(4096, k.KVX_NUMA_ANY, k.KVX_HOST_DRIVER | k.KVX_HOST_HUGE, ctypes.byref(out),
              None) == k.KVX_EINVAL                                                         # driver + huge
    assert ex(4096, -3, 0, ctypes.byref(out), None) == k.KVX_EINVAL
    assert k._lib.kv_host_alloc_numa(k.KVX_NUMA_ANY, 4096, ctypes.byref(out), None) == k.KVX_EINVAL


_FAULT_PROBE = r"""
import ctypes, json, sys
sys.path.insert(0, sys.argv[1])
from paper_2609_15021_gb300 import kvxfer as k
out = ctypes.c_void_p()
res = []
for _ in range(3):
    code = k._lib.kv_host_alloc(4096, ctypes.byref(out))
    res.append([code, k._lib.kv_last_error_message().decode()])
    k._lib.kv_host_free(out)
print(json.dumps(res))
"""


def _run_with_fault_env(value):
    import json
    import subprocess
    import sys
    env = dict(os.environ, KVX_FAULT=value)
    r = subprocess.run([sys.executable, "-c", _FAULT_PROBE, ROOT], env=env, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0, r.stderr
    return json.loads(r.stdout.strip().splitlines()[-1]), r.stderr


@pytest.mark.parametrize("value, injected_at", [("host_alloc", 0), ("host_alloc:1", 1), ("host_alloc:0", 0)])
def test_fault_armed_from_environment(k, value, injected_at):
    """KVX_FAULT arms a fault point when the library loads: exactly the
    (n + 1)-th pinned allocation fails as injected, the others do not."""
    res, _ = _run_with_fault_env(value)
    injected = [code == k.KVX_ENOMEM and "injected" in msg for code, msg in res]
    assert injected == [i == injected_at for i in range(3)]


@pytest.mark.parametrize("value", ["no_such_point", "host_alloc:x", "host_alloc:-1", ":3", "host_alloc:"])
def test_malformed_fault_environment_is_reported_and_ignored(k, value):
    res, err = _run_with_fault_env(value)
    assert "ignoring KVX_FAULT" in err
    assert not any("injected" in msg for _, msg in res)


def test_host_touch_reads_ranges_and_checks_arguments(k):
    """kv_host_touch on the CPU: any readable host memory, several ranges (one
    empty), repeated calls; argument errors return KVX_EINVAL before any read."""
    import numpy as np
    bufs = [np.ones(5 << 20, np.uint8), np.zeros(0, np.uint8), np.full(12345, 7, np.uint8)]
    for _ in range(3):
        k.kv_host_touch(bufs)
    k.kv_host_touch([])
    lib = k._lib
    ptrs = (ctypes.c_void_p * 2)(bufs[0].ctypes.data, None)
    assert lib.kv_host_touch(ptrs, (ctypes.c_int64 * 2)(16, 0), 2) == k.KVX_OK       # null with size 0: skipped
    assert lib.kv_host_touch(ptrs, (ctypes.c_int64 * 2)(16, 16), 2) == k.KVX_EINVAL  # null with a size
    assert lib.kv_host_touch(ptrs, (ctypes.c_int64 * 2)(-1, 0), 2) == k.KVX_EINVAL
    assert lib.kv_host_touch(ptrs, (ctypes.c_int64 * 2)(16, 0), -1) == k.KVX_EINVAL
    assert lib.kv_host_touch(None, None, 0) == k.KVX_OK


def test_host_touch_from_many_threads_at_once(k):
    """Eight host threads touch their own buffers at once through the one pool
    of touch threads (the ctypes calls release the GIL): every call returns
    KVX_OK, none waits for another's pages beyond its bound, and a thread's
    buffer is read, not written."""
    import threading
    import numpy as np
    bufs = [np.full((3 << 20) + 4096 * i, i, np.uint8) for i in range(8)]
    status, t0 = [None] * 8, time.monotonic()

    def run(i):
        arr = (ctypes.c_void_p * 1)(bufs[i].ctypes.data)
        sizes = (ctypes.c_int64 * 1)(bufs[i].nbytes)
        status[i] = [k._lib.kv_host_touch(arr, sizes, 1) for _ in range(20)]

    threads = [threading.Thread(target=run, args=(i,)) for i in range(8)]
    for t in threads:
        t.start()
    for t in threads:
        t.join(timeout=60)
    assert not any(t.is_alive() for t in threads)
    assert all(st == [k.KVX_OK] * 20 for st in status), status
    assert time.monotonic() - t0 < 30  # far inside one call's 5 s bound per touch
    assert all(int(b.min()) == i == int(b.max()) for i, b in enumerate(bufs))


@pytest.mark.filterwarnings("ignore:This process .* is multi-threaded")
def test_host_touch_in_a_forked_child(k):
    """A child forked after the touch threads started inherits none of them; its
    calls read the pages on the calling thread and return."""
    import numpy as np
    buf = np.ones(8 << 20, np.uint8)
    k.kv_host_touch([buf])          # the parent's threads exist from here on
    pid = os.fork()
    if pid == 0:
        code = 1
        try:
            for _ in range(3):
                k.kv_host_touch([buf])
            code = 0
        finally:
            os._exit(code)
    deadline = time.time() + 60
    while True:
        done, status = os.waitpid(pid, os.WNOHANG)
        if done:
            break
        assert time.time() < deadline, "forked child did not finish its touch"
        time.sleep(0.05)
    assert os.waitstatus_to_exitcode(status) == 0


def test_ctx_options_checked_before_any_device_call(k):
    """Bad options are refused (KVX_EINVAL) before the library looks for a GPU,
    including a negative limit for the kernels' bounded waits."""
    for kw in ({"wait_cycles": -1}, {"max_ctas": -1}, {"flags": 0x80}, {"staging_slot_bytes": 17},
               {"flags": k.KVX_FLAG_DEVICE_TMA | k.KVX_FLAG_DEVICE_LSU}):
        with pytest.raises(k.KvxError) as e:
            k.kv_ctx_create(0, **kw)
        assert e.value.status == k.KVX_EINVAL, kw


def test_tier_wait_with_no_keys_returns_at_once(k):
    t = k.KvTier(64, 2, shared_name=f"/kvx_wait0_{os.getpid()}", create=True, pin=False)
    try:
        t0 = time.perf_counter()
        assert t.wait([], timeout_s=5.0) == 0
        assert time.perf_counter() - t0 < 1.0
    finally:
        t.close()
