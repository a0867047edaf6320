// no_alloc.cu -- kv_store_noalloc: the staged store with its staging buffer in
// a static device array instead of memory the library allocates.
//
// Some callers cannot call cudaMalloc: an engine whose memory pool owns all
// of the GPU's free memory and must not see allocations it does not track, or
// code that must not let cudaMalloc / cudaFree synchronise the device in the
// middle of a pipeline.  They keep inputs and outputs in their own buffers,
// but the staged store also needs scratch memory to pack chunks before the
// copy engines move them to the host.  This entry point takes that scratch
// from g_scratch, a file-scope array of fixed size that every GPU which loads
// this part of the library holds until the process exits.  It creates no
// context, stream or event, and allocates no device, pinned or heap memory.
//
// In host code g_scratch is only a host-side stand-in for the symbol, not a
// device address: it must not be passed to a kernel.  The device address is
// looked up with cudaGetSymbolAddress the first time a call runs in a CUDA
// context and kept for that context, under the context's ID: CUDA gives every
// context an ID that is never reused in the process, so a call in another
// context (a driver-API context the caller made current, or the new primary
// context after cudaDeviceReset) looks the address up again instead of using
// one from a context that may no longer exist.

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdio.h>

#include <algorithm>
#include <mutex>

#include "kvx_internal.h"

using namespace kvx;

namespace {

constexpr int64_t kSink = 256;  // head of the array: error word when the caller passes none
constexpr int kCachedContexts = 64;

static __device__ __align__(256) uint8_t g_scratch[kSink + KVX_NOALLOC_SCRATCH_BYTES];

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

struct Resolved {
  unsigned long long ctx_id;
  uint8_t* addr;
};

std::mutex g_mu;
Resolved g_resolved[kCachedContexts] = {};  // guarded by g_mu; addr == nullptr: empty
int g_next_entry = 0;                       // guarded by g_mu: next entry to replace

kvx_status fail_cuda(cudaError_t e, const char* what) {
  set_last_cuda_error((int)e);
  set_error_text(what);
  cudaGetLastError();
  return KVX_ECUDA;
}

template <typename Fn>
Fn driver_entry(const char* name) {
  void* f = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion(name, &f, 12000, cudaEnableDefault, &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return (Fn)f;
}

// ID of the CUDA context current on this thread, making the runtime's primary
// context of `device` current first if none is.
kvx_status current_context_id(int device, unsigned long long* id) {
  static const CtxGetCurrentFn get_current = driver_entry<CtxGetCurrentFn>("cuCtxGetCurrent");
  static const CtxGetIdFn get_id = driver_entry<CtxGetIdFn>("cuCtxGetId");
  if (!get_current || !get_id) {
    set_error_text("the CUDA driver offers no cuCtxGetCurrent / cuCtxGetId");
    return KVX_ECUDA;
  }
  CUcontext c = nullptr;
  if (get_current(&c) != CUDA_SUCCESS) c = nullptr;
  if (!c) {
    // no context yet on this thread: the runtime makes its primary context current
    const cudaError_t e = cudaSetDevice(device);
    if (e != cudaSuccess) return fail_cuda(e, "cudaSetDevice (making a context current)");
    if (get_current(&c) != CUDA_SUCCESS || !c) {
      set_error_text("no CUDA context is current");
      return KVX_ECUDA;
    }
  }
  if (get_id(c, id) != CUDA_SUCCESS) {
    set_error_text("cuCtxGetId of the current context failed");
    return KVX_ECUDA;
  }
  return KVX_OK;
}

// Device address of g_scratch in the current context (of `device`).  The
// first lookup in a context also loads what a call runs there (the array and
// the pack kernels), so that later calls need no device memory that CUDA's
// lazy loading would otherwise take at their first use.
kvx_status scratch_address(int device, uint8_t** out) {
  unsigned long long id = 0;
  kvx_status st = current_context_id(device, &id);
  if (st != KVX_OK) return st;
  std::lock_guard<std::mutex> lock(g_mu);
  for (const Resolved& r : g_resolved)
    if (r.addr && r.ctx_id == id) {
      *out = r.addr;
      return KVX_OK;
    }
  void* p = nullptr;
  cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
  if (e != cudaSuccess) return fail_cuda(e, "cudaGetSymbolAddress of the static staging array failed");
  e = load_pack_kernels();
  if (e != cudaSuccess) return fail_cuda(e, "loading the pack kernels");
  g_resolved[g_next_entry] = {id, (uint8_t*)p};
  g_next_entry = (g_next_entry + 1) % kCachedContexts;
  *out = (uint8_t*)p;
  return KVX_OK;
}

}  // namespace

extern "C" kvx_status kv_store_noalloc(const kvx_pool* pool, const int32_t* block_table, int64_t table_len,
                                       int64_t tok_begin, int64_t tok_end, int32_t chunk_tokens,
                                       void* const* host_chunks, int64_t n_chunks, int64_t* dev_first_bad_block,
                                       kvx_stream_t stream_handle) {
  return guarded([&]() -> kvx_status {
    cudaStream_t stream = (cudaStream_t)stream_handle;
    int device = 0;
    cudaError_t e = cudaGetDevice(&device);
    if (e != cudaSuccess) return fail_cuda(e, "cudaGetDevice");
    // Set-up first, so that a call with an empty range makes it and nothing else.
    uint8_t* base = nullptr;
    kvx_status st = scratch_address(device, &base);
    if (st != KVX_OK) return st;
    Geometry g;
    int64_t n = 0;
    st = check_transfer(device, pool, block_table, table_len, tok_begin, tok_end, chunk_tokens, host_chunks,
                        n_chunks, stream, kHostChunks, KVX_MODE_STAGED, &g, &n, nullptr);
    if (st != KVX_OK || n == 0) return st;
    const int64_t layer_bytes_max =
        2ll * std::min<int64_t>(chunk_tokens, tok_end - tok_begin) * pool->num_heads * g.row;
    if (layer_bytes_max > KVX_NOALLOC_SCRATCH_BYTES) {
      char msg[160];
      snprintf(msg, sizeof(msg), "one layer of one chunk needs %lld bytes; the static staging array holds %lld",
               (long long)layer_bytes_max, (long long)KVX_NOALLOC_SCRATCH_BYTES);
      set_error_text(msg);
      return KVX_ERANGE;
    }
    if (dev_first_bad_block) {
      if ((uintptr_t)dev_first_bad_block & 7) return KVX_EALIGN;
      cudaPointerAttributes a;
      if (cudaPointerGetAttributes(&a, dev_first_bad_block) != cudaSuccess) {
        cudaGetLastError();
        return KVX_EDEVICE;
      }
      if (a.type != cudaMemoryTypeDevice || a.device != device) return KVX_EDEVICE;
    }
    uint8_t* staging = base + kSink;
    long long* err = dev_first_bad_block ? (long long*)dev_first_bad_block : (long long*)base;

    // Batches of (chunk, layer range) pieces that fit the array, each packed and
    // then copied out on the caller's stream.  Stream order alone keeps a batch
    // from overwriting the array before the previous batch's copies have read it.
    const int64_t first_chunk = tok_begin / chunk_tokens;
    const int64_t bpc = chunk_tokens / pool->block_tokens;
    struct Piece {
      int64_t i;
      int32_t l0, nl;
      int64_t bytes;
    } batch[kMaxJobs];
    int nb = 0;
    int64_t used = 0;
    auto tokens_of = [&](int64_t i) {
      return std::min<int64_t>(chunk_tokens, tok_end - (first_chunk + i) * chunk_tokens);
    };
    auto layer_bytes = [&](int64_t i) { return 2ll * tokens_of(i) * pool->num_heads * g.row; };
    auto flush = [&]() -> kvx_status {
      if (nb == 0) return KVX_OK;
      MoveParams p;
      init_params(&p, err, pool, g, block_table, chunk_tokens);
      int64_t off = 0;
      for (int q = 0; q < nb; ++q) {
        push_job(&p, staging + off, (first_chunk + batch[q].i) * bpc, (int32_t)tokens_of(batch[q].i), batch[q].l0,
                 batch[q].nl);
        off += batch[q].bytes;
      }
      // one warp per unit, as for the library's other HBM-bound launches
      const int64_t grid = std::max<int64_t>(1, (p.total_units + kThreads / 32 - 1) / (kThreads / 32));
      cudaError_t le = launch_move(kPack, pool->layout, p, (int)grid, stream);
      if (le != cudaSuccess) return fail_cuda(le, "pack kernel launch");
      int64_t soff = 0;
      for (int q = 0; q < nb;) {
        const int64_t i = batch[q].i;
        uint8_t* h = (uint8_t*)host_chunks[i] + (int64_t)batch[q].l0 * layer_bytes(i);
        int64_t len = 0;
        int r = q;
        while (r < nb && batch[r].i == i) len += batch[r++].bytes;  // one chunk = one allocation
        cudaError_t ce = cudaMemcpyAsync(h, staging + soff, (size_t)len, cudaMemcpyDeviceToHost, stream);
        if (ce != cudaSuccess) return fail_cuda(ce, "cudaMemcpyAsync staging -> host chunk");
        soff += len;
        q = r;
      }
      nb = 0;
      used = 0;
      return KVX_OK;
    };
    for (int64_t i = 0; i < n; ++i) {
      const int64_t ls = layer_bytes(i);
      int32_t l = 0;
      while (l < pool->num_layers) {
        const int64_t room = (KVX_NOALLOC_SCRATCH_BYTES - used) / ls;
        if (room < 1 || nb == kMaxJobs) {
          st = flush();
          if (st != KVX_OK) return st;
          continue;
        }
        const int32_t nl = (int32_t)std::min<int64_t>(room, pool->num_layers - l);
        batch[nb++] = {i, l, nl, nl * ls};
        used += nl * ls;
        l += nl;
      }
    }
    return flush();
  });
}
