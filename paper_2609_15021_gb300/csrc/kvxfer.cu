// kvxfer.cu -- host side of libkvxfer: argument checks, chunk planning and the
// stream/event pipeline around the pack/unpack kernels.
//
// Ordering contract (paper Sec. 3.2 and Fig. 2): the paper's corruption came
// from a host<->device copy issued with no dependency on the caller's current
// stream, which in PyTorch is a non-blocking stream and therefore not covered
// by legacy default-stream synchronisation.  Here kernel-only moves (zero-copy
// and device chunks) and state copies are enqueued on the caller's stream
// itself, so stream order is the dependency (the paper's same-stream
// control).  The staged pipeline overlaps packing and copying on two side
// streams: the call records an event on the caller's stream after the work
// already enqueued there, both side streams wait on it, and the caller's
// stream then waits on events recorded after the last piece of work.  Staging
// slots are reused only after an event shows their previous consumer finished
// (the premature-reuse hazard the paper cites among related reports, Sec. 3.2).

#include <cuda_runtime.h>
#include <limits.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <unistd.h>

#include <algorithm>
#include <atomic>
#include <chrono>
#include <mutex>
#include <new>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "kvx_internal.h"

using namespace kvx;

namespace {
// NVTX range around an entry point: a profiler timeline shows each call's
// host-side checks and enqueue (free when no tool is attached).
struct TraceRange {
  explicit TraceRange(const char* name) { nvtxRangePushA(name); }
  ~TraceRange() { nvtxRangePop(); }
};
}  // namespace

namespace kvx {
thread_local int g_last_cuda_error = 0;
thread_local char g_last_error_text[256] = "";
void set_last_cuda_error(int e) { g_last_cuda_error = e; }
void record_cuda_error(int e, const char* call, int line) {
  g_last_cuda_error = e;
  snprintf(g_last_error_text, sizeof(g_last_error_text), "%s: %s (kvxfer.cu:%d)", call,
           cudaGetErrorString((cudaError_t)e), line);
}
}  // namespace kvx

// Host-side fault injection (kv_fault_inject): the armed point fails its
// n-th next call with cudaErrorUnknown instead of calling CUDA.
namespace {
std::mutex g_fault_mu;
char g_fault_point[32] = "";               // guarded by g_fault_mu
std::atomic<int> g_fault_countdown{-1};    // -1: unarmed; written under g_fault_mu

bool fault_now(const char* point) {
  // Unarmed is the common case and takes no lock; the armed state is re-read under it.
  if (g_fault_countdown.load(std::memory_order_relaxed) < 0) return false;
  std::lock_guard<std::mutex> lock(g_fault_mu);
  const int n = g_fault_countdown.load(std::memory_order_relaxed);
  if (n < 0 || strcmp(point, g_fault_point) != 0) return false;
  g_fault_countdown.store(n - 1, std::memory_order_relaxed);  // 0 fires now and disarms
  if (n > 0) return false;
  g_fault_point[0] = 0;
  return true;
}
}  // namespace

namespace kvx {
bool fault_point(const char* point) { return fault_now(point); }
}  // namespace kvx

#define KVX_CUDA_AT(point, call)                                                   \
  do {                                                                             \
    cudaError_t e_ = fault_now(point) ? cudaErrorUnknown : (call);                 \
    if (e_ != cudaSuccess) {                                                       \
      record_cuda_error((int)e_, #call, __LINE__);                                 \
      cudaGetLastError();                                                          \
      return KVX_ECUDA;                                                            \
    }                                                                              \
  } while (0)
#define KVX_CUDA(call) KVX_CUDA_AT("", call)

namespace {

constexpr int32_t kDefaultSlots = 4;
// 4 x 128 MiB: measured on GB300 at 128k tokens, staged stores and restores
// run at 200.0 GB/s against 198.3 with 32 MiB slots, and the host enqueues a
// 32k-token store in 0.6 ms instead of 10.4 (a quarter of the launches, each
// carrying its layers' tensor maps).
constexpr int64_t kDefaultSlotBytes = 128ll << 20;
constexpr long long kNoError = LLONG_MAX;

struct TimedLaunch {
  cudaEvent_t a, b;
  int64_t bytes;
  int dir;
};

}  // namespace

struct kvx_ctx {
  int device = 0;
  kvx_opts opts{};
  int32_t store_mode = KVX_MODE_STAGED;
  int32_t load_mode = KVX_MODE_STAGED;
  int num_sms = 1;
  int move_occ[2][2] = {{1, 1}, {1, 1}};
  int seg_occ = 1;
  int link_ctas = 1;  // default CTA cap of launches that cross the host link
  cudaStream_t s_kern = nullptr;  // pack / unpack kernels
  cudaStream_t s_copy = nullptr;  // host-link copies of the staged mode
  cudaStream_t s_aux = nullptr;   // error-word readback
  cudaEvent_t ev_in = nullptr;
  cudaEvent_t ev_kern_done = nullptr;
  cudaEvent_t ev_copy_done = nullptr;
  int32_t nslots = kDefaultSlots;
  int64_t slot_bytes = kDefaultSlotBytes;
  std::vector<uint8_t*> slots;
  std::vector<cudaEvent_t> ev_ready;  // slot written (by pack or by an H2D copy)
  std::vector<cudaEvent_t> ev_free;   // slot consumed (by a D2H copy or by unpack)
  int32_t next_slot = 0;
  long long* d_err = nullptr;  // 16-byte allocation: error word, then the timeout flag
  int* d_timeout = nullptr;
  std::mutex mu;
  // end of this context's last transfer call (host clock, ns), for the host touch
  int64_t last_call_ns = 0;
  int64_t launches = 0, memcpys = 0;
  int64_t timed[2] = {0, 0}, timed_bytes[2] = {0, 0};
  double timed_ms[2] = {0.0, 0.0};
  std::vector<TimedLaunch> pending;
  std::vector<cudaEvent_t> spare_events;
  // tensor maps of the last HND pool moved by the tensor-map engine
  std::vector<uint8_t> tmaps;
  std::vector<const void*> tmap_bases;
  int64_t tmap_shape[6] = {0, 0, 0, 0, 0, 0};
  bool tmap_ok = false;
};

namespace {

// Makes ctx->device current for the duration of a call and restores the
// caller's device afterwards.
struct DeviceGuard {
  int prev = -1;
  bool ok = false;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) != cudaSuccess) {
      cudaGetLastError();
      prev = -1;
    }
    ok = (prev == dev) || (cudaSetDevice(dev) == cudaSuccess);
    if (!ok) cudaGetLastError();
  }
  ~DeviceGuard() {
    int cur = -1;
    if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
  }
};

int32_t pages_per_block(const kvx_pool* P) { return P->pages_per_block > 1 ? P->pages_per_block : 1; }

bool mul_ok(int64_t a, int64_t b, int64_t* out) {
  if (a < 0 || b < 0) return false;
  if (a != 0 && b > INT64_MAX / a) return false;
  *out = a * b;
  return true;
}

kvx_status check_device_range(int device, const void* p, int64_t bytes) {
  if (!p) return KVX_EINVAL;
  if (bytes <= 0) return KVX_OK;
  const uint8_t* ends[2] = {(const uint8_t*)p, (const uint8_t*)p + (bytes - 1)};
  for (const uint8_t* q : ends) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, q) != cudaSuccess) {
      cudaGetLastError();
      return KVX_EDEVICE;
    }
    if (a.type != cudaMemoryTypeDevice || a.device != device) return KVX_EDEVICE;
  }
  return KVX_OK;
}

// Page-locked host memory whose first and last byte are mapped for the GPU at
// one consistent offset; *mapped receives the device-side address of p.
kvx_status check_pinned_range(const void* p, int64_t bytes, uint8_t** mapped) {
  if (!p) return KVX_EINVAL;
  cudaPointerAttributes a, b;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return KVX_ENOTPINNED;
  }
  if (a.type != cudaMemoryTypeHost) return KVX_ENOTPINNED;
  *mapped = (uint8_t*)a.devicePointer;
  if (bytes > 1) {
    const uint8_t* last = (const uint8_t*)p + (bytes - 1);
    if (cudaPointerGetAttributes(&b, last) != cudaSuccess) {
      cudaGetLastError();
      return KVX_ENOTPINNED;
    }
    if (b.type != cudaMemoryTypeHost) return KVX_ENOTPINNED;
    if (a.devicePointer && (uint8_t*)b.devicePointer != (uint8_t*)a.devicePointer + (bytes - 1))
      *mapped = nullptr;  // mapping not contiguous: only the copy engines may use it
  }
  return KVX_OK;
}

kvx_status check_stream_device(cudaStream_t s, int device) {
  if (s == nullptr || s == cudaStreamLegacy || s == cudaStreamPerThread) return KVX_OK;
  // cudaStreamGetDevice is not permitted on a capturing stream (it would
  // invalidate the capture): a stream being captured into a graph is taken as is.
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &cap) != cudaSuccess) {
    cudaGetLastError();
    return KVX_EINVAL;
  }
  if (cap != cudaStreamCaptureStatusNone) return KVX_OK;
  int d = -1;
  if (cudaStreamGetDevice(s, &d) != cudaSuccess) {
    cudaGetLastError();
    return KVX_EINVAL;
  }
  return d == device ? KVX_OK : KVX_EDEVICE;
}

kvx_status check_pool_shape(const kvx_pool* P, Geometry* g) {
  if (!P || !P->layer_base) return KVX_EINVAL;
  if (P->num_layers < 1 || P->num_layers > KVX_MAX_LAYERS) return KVX_EINVAL;
  if (P->num_blocks < 1 || P->block_tokens < 1 || P->num_heads < 1 || P->head_dim < 1 ||
      P->elem_bytes < 1)
    return KVX_EINVAL;
  if (P->layout != KVX_LAYOUT_HND && P->layout != KVX_LAYOUT_NHD) return KVX_EINVAL;
  if ((int64_t)P->block_tokens * P->num_heads > (1ll << 30)) return KVX_EINVAL;
  if (P->pages_per_block < 0) return KVX_EINVAL;
  if (P->num_blocks % pages_per_block(P) != 0) return KVX_EALIGN;
  int64_t row, hb, page, layer;
  if (!mul_ok(P->head_dim, P->elem_bytes, &row) || row > (1ll << 30)) return KVX_EINVAL;
  if (!mul_ok((int64_t)P->num_heads * P->block_tokens, 2 * row, &page)) return KVX_EINVAL;
  if (!mul_ok(page, P->num_blocks, &layer)) return KVX_EINVAL;
  (void)hb;
  if (row % 16 != 0) return KVX_EALIGN;
  g->row = row;
  g->page_bytes = page;
  g->layer_bytes = layer;
  return KVX_OK;
}

kvx_status check_pool_memory(int device, const kvx_pool* P, const Geometry& g) {
  for (int l = 0; l < P->num_layers; ++l) {
    const void* b = P->layer_base[l];
    if (!b) return KVX_EINVAL;
    if ((uintptr_t)b & 15) return KVX_EALIGN;
    kvx_status st = check_device_range(device, b, g.layer_bytes);
    if (st != KVX_OK) return st;
  }
  return KVX_OK;
}

int64_t chunk_bytes_of(const kvx_pool* P, const Geometry& g, int64_t tokens) {
  return (int64_t)P->num_layers * 2 * tokens * P->num_heads * g.row;
}

kvx_status check_range(const kvx_pool* P, int64_t table_len, int64_t t0, int64_t t1, int32_t C,
                       int64_t n_chunks, int64_t* n_needed) {
  if (C < 1 || table_len < 0 || n_chunks < 0) return KVX_EINVAL;
  if (t0 < 0 || t1 < t0) return KVX_ERANGE;
  if (C % P->block_tokens != 0) return KVX_EALIGN;
  if (t0 % C != 0) return KVX_EALIGN;
  int64_t cap;
  if (!mul_ok(table_len, (int64_t)P->block_tokens * pages_per_block(P), &cap)) return KVX_EINVAL;
  if (t1 > cap) return KVX_ERANGE;
  const int64_t need = (t1 == t0) ? 0 : (t1 + C - 1) / C - t0 / C;
  if (need > n_chunks) return KVX_ERANGE;
  if (need > INT32_MAX) return KVX_EINVAL;
  *n_needed = need;
  return KVX_OK;
}

cudaEvent_t take_timing_event(kvx_ctx* ctx) {
  if (!ctx->spare_events.empty()) {
    cudaEvent_t e = ctx->spare_events.back();
    ctx->spare_events.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return e;
}

// 64-byte aligned start of the context's tensor-map storage (CUtensorMap alignment).
void* tensor_map_storage(kvx_ctx* ctx) {
  uintptr_t p = (uintptr_t)ctx->tmaps.data();
  return (void*)((p + 63) & ~(uintptr_t)63);
}

// Tensor maps of pool P (cached per pool in the context); null if P cannot be described.
const void* tensor_maps_of(kvx_ctx* ctx, const kvx_pool* P, int64_t row) {
  const int64_t shape[6] = {P->num_layers, P->num_blocks, P->block_tokens, P->num_heads, row, P->layout};
  bool same = ctx->tmap_bases.size() == (size_t)P->num_layers && memcmp(shape, ctx->tmap_shape, sizeof(shape)) == 0;
  for (int l = 0; same && l < P->num_layers; ++l) same = ctx->tmap_bases[l] == P->layer_base[l];
  if (!same) {
    ctx->tmaps.assign((size_t)P->num_layers * kTensorMapBytes + 64, 0);
    ctx->tmap_ok = encode_tensor_maps(P, row, tensor_map_storage(ctx));
    ctx->tmap_bases.assign(P->layer_base, P->layer_base + P->num_layers);
    memcpy(ctx->tmap_shape, shape, sizeof(shape));
  }
  return ctx->tmap_ok ? tensor_map_storage(ctx) : nullptr;
}

// Launch one pack/unpack kernel with optional timing events around it.
// over_link: the launch reads or writes mapped host memory, so the host link,
// not HBM, bounds it and a fraction of the SMs saturates it.
kvx_status launch_move_timed(kvx_ctx* ctx, const kvx_pool* P, int dir, int layout, const MoveParams& p,
                             int64_t bytes, cudaStream_t s, bool over_link) {
  // TMA variants: device-side chunks only, and a K or V half page (the
  // largest unit) of at most 48 KiB: one shared-memory stage per unit, or a
  // ring of 2-3 when a capped grid strides over units.
  // Default: tensor maps for HND pools the TMA unit can describe; one bulk
  // copy per side for NHD pools, whose units are contiguous on both sides
  // (measured on GB300 at 32k tokens: 6.95 / 7.00 TB/s against 6.78 / 6.75
  // with loads/stores); loads/stores otherwise (per-row bulk copies of HND
  // pages without tensor maps are slower).
  const int64_t unit_bytes = (int64_t)p.B * p.H * p.R;
  const uint32_t f = ctx->opts.flags;
  const bool fits = !over_link && unit_bytes <= (48 << 10) && !(f & KVX_FLAG_DEVICE_LSU);
  const void* maps = fits && layout == KVX_LAYOUT_HND ? tensor_maps_of(ctx, P, p.R) : nullptr;
  const bool tma = fits && (maps || layout == KVX_LAYOUT_NHD || (f & KVX_FLAG_DEVICE_TMA));
  // Grid: HBM-bound launches give every unit its own warp (LSU) or CTA (TMA)
  // and let the block scheduler spread them; measured on GB300 this keeps
  // DRAM busier than a persistent grid walking the units in lockstep.
  // Launches over the host link, or capped by the caller (max_ctas), are
  // persistent: each warp or CTA strides over many units.
  int64_t grid = tma ? p.total_units : (p.total_units + (kThreads / 32) - 1) / (kThreads / 32);
  int64_t cap = grid;
  if (ctx->opts.max_ctas > 0)
    cap = ctx->opts.max_ctas;
  else if (over_link)
    cap = std::min<int64_t>(ctx->link_ctas, (int64_t)ctx->num_sms * ctx->move_occ[dir][layout]);
  grid = std::max<int64_t>(1, std::min(std::min(grid, cap), (int64_t)INT_MAX));  // grid.x limit
  int stage_bytes = 0, stages = 0;
  if (tma) {
    // one stage when each CTA moves one unit; else a ring of 3 (2 above 32 KiB)
    stage_bytes = (int)((unit_bytes + 127) / 128 * 128);
    stages = grid >= p.total_units ? 1 : stage_bytes <= (32 << 10) ? 3 : 2;
  }
  cudaEvent_t a = nullptr, b = nullptr;
  const bool timing = (ctx->opts.flags & KVX_FLAG_TIME_KERNELS) != 0;
  if (timing) {
    a = take_timing_event(ctx);
    b = take_timing_event(ctx);
    if (a && b) {
      KVX_CUDA(cudaEventRecord(a, s));
    }
  }
  TmaWait wt{ctx->opts.wait_cycles > 0 ? (long long)ctx->opts.wait_cycles : kDefaultWaitCycles, -1,
             ctx->d_timeout};
  if ((maps || tma) && fault_now("tma_wait")) wt.stall_unit = 0;
  if (maps)
    KVX_CUDA_AT("launch", launch_move_tmap(dir, p, maps, P->num_layers, (int)grid, stage_bytes, stages, wt, s));
  else if (tma)
    KVX_CUDA_AT("launch", launch_move_tma(dir, layout, p, (int)grid, stage_bytes, stages, wt, s));
  else
    KVX_CUDA_AT("launch", launch_move(dir, layout, p, (int)grid, s));
  ctx->launches++;
  if (timing && a && b) {
    KVX_CUDA(cudaEventRecord(b, s));
    ctx->pending.push_back({a, b, 2 * bytes, dir});
  }
  return KVX_OK;
}

void init_move_params(MoveParams* p, long long* err, const kvx_pool* P, const Geometry& g,
                      const int32_t* table, int32_t C) {
  memset(p, 0, sizeof(*p));
  for (int l = 0; l < P->num_layers; ++l) p->layer_base[l] = (uint8_t*)P->layer_base[l];
  p->table = table;
  p->err = err;
  p->num_blocks = P->num_blocks;
  p->page_bytes = g.page_bytes;
  p->blocks_per_chunk = C / P->block_tokens;
  p->ppb = pages_per_block(P);
  p->B = P->block_tokens;
  p->H = P->num_heads;
  p->R = (int32_t)g.row;
  const int64_t vpr = g.row / 16;
  p->fast = (vpr >= 1 && vpr <= 32 && (vpr & (vpr - 1)) == 0) ? 1 : 0;
  if (p->fast) {
    int sh = 0;
    while ((1ll << sh) < vpr) ++sh;
    p->vpr_shift = sh;
    const int rows_per_step = 32 >> sh;
    p->rpi_div_h = rows_per_step / P->num_heads;
    p->rpi_mod_h = rows_per_step % P->num_heads;
  }
}

// A chunk-side region of one launch: layers [l0, l0+nl) of chunk i.
struct Piece {
  int64_t i;       // chunk index within the call
  int32_t l0, nl;
  int64_t bytes;   // nl * 2 * T_i * H * row
};

void add_job(MoveParams* p, uint8_t* chunk_side, int64_t first_block, int32_t tokens, int32_t l0,
             int32_t nl) {
  Job& J = p->jobs[p->n_jobs];
  J.chunk = chunk_side;
  J.first_block = first_block;
  J.tokens = tokens;
  J.l0 = l0;
  const int64_t units = (int64_t)nl * p->blocks_per_chunk * 2;
  p->total_units += units;
  J.unit_end = p->total_units;
  p->n_jobs++;
}

kvx_status ensure_staging(kvx_ctx* ctx) {
  if (!ctx->slots.empty()) return KVX_OK;
  for (int32_t k = 0; k < ctx->nslots; ++k) {
    uint8_t* s = nullptr;
    if (cudaMalloc(&s, (size_t)ctx->slot_bytes) != cudaSuccess) {
      cudaGetLastError();
      for (uint8_t* q : ctx->slots) cudaFree(q);
      ctx->slots.clear();
      return KVX_ENOMEM;
    }
    ctx->slots.push_back(s);
  }
  return KVX_OK;
}

// Everything one kv_store / kv_load / kv_pack / kv_unpack call needs once
// its arguments have been checked.
struct Plan {
  const kvx_pool* P;
  Geometry g;
  const int32_t* table;
  int32_t C;
  int64_t first_chunk;  // chunk index of the first chunk of the range
  int64_t n;            // chunks in the range
  int64_t bpc;          // pages per chunk (C / B)
  int dir;              // kPack or kUnpack
  bool over_link;       // chunks are mapped host memory (zero-copy)
  std::vector<int32_t> tokens;  // tokens held by chunk i
  std::vector<uint8_t*> side;   // chunk i as the kernel (mapped/device) or copy engine sees it
};

// Zero-copy and device chunks: one kernel pass per batch of whole chunks, on
// stream s.
kvx_status enqueue_direct(kvx_ctx* ctx, const Plan& pl, cudaStream_t s) {
  MoveParams p;
  init_move_params(&p, ctx->d_err, pl.P, pl.g, pl.table, pl.C);
  int64_t bytes = 0;
  for (int64_t i = 0; i < pl.n; ++i) {
    add_job(&p, pl.side[i], (pl.first_chunk + i) * pl.bpc, pl.tokens[i], 0, pl.P->num_layers);
    bytes += chunk_bytes_of(pl.P, pl.g, pl.tokens[i]);
    if (p.n_jobs == kMaxJobs || i == pl.n - 1) {
      TraceRange trace("kvx launch: chunks");
      kvx_status st = launch_move_timed(ctx, pl.P, pl.dir, pl.P->layout, p, bytes, s, pl.over_link);
      if (st != KVX_OK) return st;
      p.n_jobs = 0;
      p.total_units = 0;
      bytes = 0;
    }
  }
  return KVX_OK;
}

// Staged: slot-sized batches of (chunk, layer range) pieces.  A store packs
// batch b into slot b % S on s_kern and copies it out on s_copy; a load copies
// batch b in on s_copy and unpacks it on s_kern.  ev_ready[k] marks slot k
// written, ev_free[k] marks it consumed; a slot is rewritten only after its
// last consumer, in this call or an earlier one, has finished.
kvx_status enqueue_staged(kvx_ctx* ctx, const Plan& pl) {
  const kvx_pool* P = pl.P;
  std::vector<Piece> batch;
  int64_t used = 0;
  auto layer_bytes = [&](int64_t i) { return 2ll * pl.tokens[i] * P->num_heads * pl.g.row; };
  auto flush = [&]() -> kvx_status {
    if (batch.empty()) return KVX_OK;
    TraceRange trace(pl.dir == kPack ? "kvx staged batch: pack, copy out" : "kvx staged batch: copy in, unpack");
    const int k = ctx->next_slot;
    ctx->next_slot = (ctx->next_slot + 1) % ctx->nslots;
    uint8_t* slot = ctx->slots[k];
    MoveParams p;
    init_move_params(&p, ctx->d_err, P, pl.g, pl.table, pl.C);
    int64_t off = 0;
    for (const Piece& pc : batch) {
      add_job(&p, slot + off, (pl.first_chunk + pc.i) * pl.bpc, pl.tokens[pc.i], pc.l0, pc.nl);
      off += pc.bytes;
    }
    const int64_t bytes = off;
    // Copies of the batch: one per piece, merged only within one chunk.  Two
    // chunks that happen to be adjacent in the address space may still be
    // separate pinned allocations, and one copy may not span two of them.
    auto copies = [&](bool to_host) -> kvx_status {
      int64_t soff = 0;
      size_t q = 0;
      while (q < batch.size()) {
        const Piece& a = batch[q];
        uint8_t* h = pl.side[a.i] + (int64_t)a.l0 * layer_bytes(a.i);
        int64_t len = a.bytes;
        size_t r = q + 1;
        while (r < batch.size() && batch[r].i == a.i) {
          len += batch[r].bytes;
          ++r;
        }
        if (to_host)
          KVX_CUDA_AT("memcpy", cudaMemcpyAsync(h, slot + soff, (size_t)len, cudaMemcpyDeviceToHost, ctx->s_copy));
        else
          KVX_CUDA_AT("memcpy", cudaMemcpyAsync(slot + soff, h, (size_t)len, cudaMemcpyHostToDevice, ctx->s_copy));
        ctx->memcpys++;
        soff += len;
        q = r;
      }
      return KVX_OK;
    };
    kvx_status st;
    if (pl.dir == kPack) {
      KVX_CUDA(cudaStreamWaitEvent(ctx->s_kern, ctx->ev_free[k], 0));
      st = launch_move_timed(ctx, P, kPack, P->layout, p, bytes, ctx->s_kern, false);
      if (st != KVX_OK) return st;
      KVX_CUDA(cudaEventRecord(ctx->ev_ready[k], ctx->s_kern));
      KVX_CUDA(cudaStreamWaitEvent(ctx->s_copy, ctx->ev_ready[k], 0));
      st = copies(true);
      if (st != KVX_OK) return st;
      KVX_CUDA(cudaEventRecord(ctx->ev_free[k], ctx->s_copy));
    } else {
      KVX_CUDA(cudaStreamWaitEvent(ctx->s_copy, ctx->ev_free[k], 0));
      st = copies(false);
      if (st != KVX_OK) return st;
      KVX_CUDA(cudaEventRecord(ctx->ev_ready[k], ctx->s_copy));
      KVX_CUDA(cudaStreamWaitEvent(ctx->s_kern, ctx->ev_ready[k], 0));
      st = launch_move_timed(ctx, P, kUnpack, P->layout, p, bytes, ctx->s_kern, false);
      if (st != KVX_OK) return st;
      KVX_CUDA(cudaEventRecord(ctx->ev_free[k], ctx->s_kern));
    }
    batch.clear();
    used = 0;
    return KVX_OK;
  };
  for (int64_t i = 0; i < pl.n; ++i) {
    const int64_t ls = layer_bytes(i);
    int32_t l = 0;
    while (l < P->num_layers) {
      const int64_t room = (ctx->slot_bytes - used) / ls;
      if (room < 1 || (int)batch.size() == kMaxJobs) {
        kvx_status st = flush();
        if (st != KVX_OK) return st;
        continue;
      }
      const int32_t nl = (int32_t)std::min<int64_t>(room, P->num_layers - l);
      batch.push_back({i, l, nl, nl * ls});
      used += nl * ls;
      l += nl;
    }
  }
  return flush();
}

// The caller's stream waits for everything the side streams hold, which
// includes all the work of this call -- also when enqueueing stopped early.
kvx_status join_caller(kvx_ctx* ctx, cudaStream_t stream, bool copy_stream_used) {
  KVX_CUDA(cudaEventRecord(ctx->ev_kern_done, ctx->s_kern));
  KVX_CUDA(cudaStreamWaitEvent(stream, ctx->ev_kern_done, 0));
  if (copy_stream_used) {
    KVX_CUDA(cudaEventRecord(ctx->ev_copy_done, ctx->s_copy));
    KVX_CUDA(cudaStreamWaitEvent(stream, ctx->ev_copy_done, 0));
  }
  return KVX_OK;
}

}  // namespace

namespace kvx {

void set_error_text(const char* text) { snprintf(g_last_error_text, sizeof(g_last_error_text), "%s", text); }

kvx_status check_transfer(int device, const kvx_pool* P, const int32_t* table, int64_t table_len, int64_t t0,
                          int64_t t1, int32_t C, void* const* chunks, int64_t n_chunks, cudaStream_t stream,
                          int where, int mode, Geometry* g, int64_t* n_out, uint8_t** side) {
  kvx_status st = check_pool_shape(P, g);
  if (st != KVX_OK) return st;
  int64_t n = 0;
  st = check_range(P, table_len, t0, t1, C, n_chunks, &n);
  if (st != KVX_OK) return st;
  if (n > 0 && (!table || !chunks)) return KVX_EINVAL;
  st = check_stream_device(stream, device);
  if (st != KVX_OK) return st;
  *n_out = n;
  if (n == 0) return KVX_OK;  // empty range: nothing to order or move
  st = check_pool_memory(device, P, *g);
  if (st != KVX_OK) return st;
  if ((uintptr_t)table & 3) return KVX_EALIGN;
  const int64_t block_span = (int64_t)P->block_tokens * pages_per_block(P);
  const int64_t blocks_needed = (t1 + block_span - 1) / block_span;
  st = check_device_range(device, table, blocks_needed * (int64_t)sizeof(int32_t));
  if (st != KVX_OK) return st;
  const int64_t first_chunk = t0 / C;
  for (int64_t i = 0; i < n; ++i) {
    const int64_t tokens = std::min<int64_t>(C, t1 - (first_chunk + i) * C);
    const int64_t bytes = chunk_bytes_of(P, *g, tokens);
    void* c = chunks[i];
    if (!c) return KVX_EINVAL;
    if ((uintptr_t)c & 15) return KVX_EALIGN;
    uint8_t* s = (uint8_t*)c;
    if (where == kDeviceChunks) {
      st = check_device_range(device, c, bytes);
      if (st != KVX_OK) return st;
    } else {
      uint8_t* mapped = nullptr;
      st = check_pinned_range(c, bytes, &mapped);
      if (st != KVX_OK) return st;
      if (mode == KVX_MODE_ZEROCOPY) {
        if (!mapped) return KVX_ENOTPINNED;
        s = mapped;
      }
    }
    if (side) side[i] = s;
  }
  return KVX_OK;
}

void init_params(MoveParams* p, long long* err, const kvx_pool* P, const Geometry& g, const int32_t* table,
                 int32_t C) {
  init_move_params(p, err, P, g, table, C);
}

void push_job(MoveParams* p, uint8_t* chunk_side, int64_t first_block, int32_t tokens, int32_t l0, int32_t nl) {
  add_job(p, chunk_side, first_block, tokens, l0, nl);
}

int64_t chunk_bytes(const kvx_pool* P, const Geometry& g, int64_t tokens) { return chunk_bytes_of(P, g, tokens); }

}  // namespace kvx

namespace {

int64_t now_ns() {
  return std::chrono::duration_cast<std::chrono::nanoseconds>(std::chrono::steady_clock::now().time_since_epoch())
      .count();
}

// A context that began no transfer for this long reads its host chunks' pages
// before it moves them.  Measured from the previous call's start, since the
// library does not see when the GPU finishes; 1 s keeps a caller that waits
// for each 128k-256k transfer before the next (160-350 ms) from touching at
// every call, and the slowdown after 1 s of idle time was still small (+4 %).
constexpr int64_t kIdleTouchNs = 1000ll * 1000 * 1000;

// The shared body of kv_store / kv_load / kv_pack / kv_unpack.
kvx_status transfer(kvx_ctx* ctx, const kvx_pool* P, const int32_t* table, int64_t table_len, int64_t t0,
                    int64_t t1, int32_t C, void* const* chunks, int64_t n_chunks, cudaStream_t stream,
                    int dir, int where) {
  if (!ctx) return KVX_EINVAL;
  DeviceGuard guard(ctx->device);
  if (!guard.ok) return KVX_ECUDA;
  const int mode = (where == kDeviceChunks) ? KVX_MODE_ZEROCOPY
                                            : (dir == kPack ? ctx->store_mode : ctx->load_mode);
  Plan pl;
  int64_t cap = 0;  // entries the chunk arrays may need (checked below)
  if (C > 0 && t0 >= 0 && t1 > t0) cap = std::min<int64_t>(n_chunks, (t1 + C - 1) / C - t0 / C);
  pl.side.resize((size_t)std::max<int64_t>(cap, 0));
  int64_t n = 0;
  kvx_status st = check_transfer(ctx->device, P, table, table_len, t0, t1, C, chunks, n_chunks, stream, where,
                                 mode, &pl.g, &n, pl.side.data());
  if (st != KVX_OK || n == 0) return st;
  pl.P = P;
  pl.table = table;
  pl.C = C;
  pl.first_chunk = t0 / C;
  pl.n = n;
  pl.bpc = C / P->block_tokens;
  pl.dir = dir;
  pl.over_link = (where == kHostChunks && mode == KVX_MODE_ZEROCOPY);
  pl.tokens.resize((size_t)n);
  for (int64_t i = 0; i < n; ++i)
    pl.tokens[i] = (int32_t)std::min<int64_t>(C, t1 - (pl.first_chunk + i) * C);
  const bool staged = (mode == KVX_MODE_STAGED);
  const int64_t max_layer_bytes = 2ll * std::min<int64_t>(C, t1 - t0) * P->num_heads * pl.g.row;
  if (staged && max_layer_bytes > ctx->slot_bytes) return KVX_EINVAL;

  std::lock_guard<std::mutex> lock(ctx->mu);
  const int64_t now = now_ns();
  if (where == kHostChunks && !(ctx->opts.flags & KVX_FLAG_NO_HOST_TOUCH) && now - ctx->last_call_ns > kIdleTouchNs) {
    TraceRange trace("kvx host touch after idle time");
    touch_before_transfer(chunks, pl.tokens, P, pl.g, stream);
  }
  ctx->last_call_ns = now;
  const bool ordered = (ctx->opts.flags & KVX_FLAG_UNORDERED) == 0;
  // Kernel-only moves (zero-copy or device chunks) run on the caller's stream
  // itself: stream order is the dependency, with no event hop in between.
  if (!staged && ordered) return enqueue_direct(ctx, pl, stream);
  if (staged) {
    st = ensure_staging(ctx);
    if (st != KVX_OK) return st;
  }
  // The staged pipeline overlaps packing and copying on two side streams
  // that wait on an event recorded on the caller's stream.  Without that wait
  // (KVX_FLAG_UNORDERED, the negative control) kernel-only moves also run on
  // a side stream, which is the paper's missing dependency.
  KVX_CUDA_AT("event", cudaEventRecord(ctx->ev_in, stream));
  if (ordered) {
    KVX_CUDA(cudaStreamWaitEvent(ctx->s_kern, ctx->ev_in, 0));
    KVX_CUDA(cudaStreamWaitEvent(ctx->s_copy, ctx->ev_in, 0));
  }
  st = staged ? enqueue_staged(ctx, pl) : enqueue_direct(ctx, pl, ctx->s_kern);
  const kvx_status joined = join_caller(ctx, stream, staged);
  return st != KVX_OK ? st : joined;
}

kvx_status state_copy(kvx_ctx* ctx, int32_t L, void* const* layer_base, int64_t num_slots, int64_t slot_bytes,
                      int64_t slot, void* host_obj, cudaStream_t stream, bool to_host) {
  if (!ctx || !layer_base || !host_obj) return KVX_EINVAL;
  if (L < 1 || L > KVX_MAX_LAYERS || num_slots < 1 || slot_bytes < 1) return KVX_EINVAL;
  if (slot < 0 || slot >= num_slots) return KVX_ERANGE;
  if (slot_bytes % 16 != 0 || ((uintptr_t)host_obj & 15)) return KVX_EALIGN;
  int64_t layer_bytes, obj_bytes;
  if (!mul_ok(num_slots, slot_bytes, &layer_bytes) || !mul_ok(L, slot_bytes, &obj_bytes)) return KVX_EINVAL;
  DeviceGuard guard(ctx->device);
  if (!guard.ok) return KVX_ECUDA;
  kvx_status st = check_stream_device(stream, ctx->device);
  if (st != KVX_OK) return st;
  for (int32_t l = 0; l < L; ++l) {
    if (!layer_base[l]) return KVX_EINVAL;
    if ((uintptr_t)layer_base[l] & 15) return KVX_EALIGN;
    st = check_device_range(ctx->device, layer_base[l], layer_bytes);
    if (st != KVX_OK) return st;
  }
  uint8_t* mapped = nullptr;
  st = check_pinned_range(host_obj, obj_bytes, &mapped);
  if (st != KVX_OK) return st;
  const int mode = to_host ? ctx->store_mode : ctx->load_mode;
  if (mode == KVX_MODE_ZEROCOPY && !mapped) return KVX_ENOTPINNED;

  std::lock_guard<std::mutex> lock(ctx->mu);
  // Ordered copies run on the caller's stream itself (stream order is the
  // dependency); the negative control (KVX_FLAG_UNORDERED) runs them on a side
  // stream that does not wait for the caller's work.
  const bool ordered = (ctx->opts.flags & KVX_FLAG_UNORDERED) == 0;
  if (mode == KVX_MODE_ZEROCOPY) {
    cudaStream_t ks = ordered ? stream : ctx->s_kern;
    SegmentParams p;
    memset(&p, 0, sizeof(p));
    int64_t bytes = 0;
    for (int32_t l = 0; l < L; ++l) {
      uint8_t* dev = (uint8_t*)layer_base[l] + slot * slot_bytes;
      uint8_t* host = mapped + (int64_t)l * slot_bytes;
      Segment& s = p.seg[p.n_seg++];
      s.src = to_host ? dev : host;
      s.dst = to_host ? host : dev;
      p.total_bytes += slot_bytes;
      s.byte_end = p.total_bytes;
      bytes += slot_bytes;
      if (p.n_seg == kMaxSegments || l == L - 1) {
        // Warps of at most 32 KiB units, then the unit size that splits the
        // bytes evenly over those warps in whole rounds: with 32 KiB units a
        // 48-layer state snapshot took 3 rounds of 608 warps where 2.7 suffice.
        constexpr int64_t kMaxUnit = 32 << 10, kWarps = kThreads / 32;
        int64_t grid = (p.total_bytes + kMaxUnit * kWarps - 1) / (kMaxUnit * kWarps);
        int64_t cap = (int64_t)ctx->num_sms * ctx->seg_occ;
        cap = std::min<int64_t>(cap, ctx->opts.max_ctas > 0 ? ctx->opts.max_ctas : ctx->link_ctas);
        grid = std::max<int64_t>(1, std::min(grid, cap));
        const int64_t warps = grid * kWarps;
        const int64_t rounds = (p.total_bytes + warps * kMaxUnit - 1) / (warps * kMaxUnit);
        const int64_t share = (p.total_bytes + warps * rounds - 1) / (warps * rounds);
        p.unit_bytes = std::max<int64_t>(512, (share + 511) / 512 * 512);
        p.total_units = (p.total_bytes + p.unit_bytes - 1) / p.unit_bytes;
        const bool timing = (ctx->opts.flags & KVX_FLAG_TIME_KERNELS) != 0;
        cudaEvent_t a = timing ? take_timing_event(ctx) : nullptr;
        cudaEvent_t b = timing ? take_timing_event(ctx) : nullptr;
        if (a && b) KVX_CUDA(cudaEventRecord(a, ks));
        KVX_CUDA(launch_segments(p, (int)grid, ks));
        ctx->launches++;
        if (a && b) {
          KVX_CUDA(cudaEventRecord(b, ks));
          ctx->pending.push_back({a, b, 2 * bytes, to_host ? 0 : 1});
        }
        memset(&p, 0, sizeof(p));
        bytes = 0;
      }
    }
    if (!ordered) {
      KVX_CUDA(cudaEventRecord(ctx->ev_kern_done, ctx->s_kern));
      KVX_CUDA(cudaStreamWaitEvent(stream, ctx->ev_kern_done, 0));
    }
    return KVX_OK;
  }
  // Staged mode: the slot of each layer is already contiguous, so the copy
  // engines move it directly; no staging buffer is needed.
  cudaStream_t cs = ordered ? stream : ctx->s_copy;
  for (int32_t l = 0; l < L; ++l) {
    uint8_t* dev = (uint8_t*)layer_base[l] + slot * slot_bytes;
    uint8_t* host = (uint8_t*)host_obj + (int64_t)l * slot_bytes;
    if (to_host)
      KVX_CUDA(cudaMemcpyAsync(host, dev, (size_t)slot_bytes, cudaMemcpyDeviceToHost, cs));
    else
      KVX_CUDA(cudaMemcpyAsync(dev, host, (size_t)slot_bytes, cudaMemcpyHostToDevice, cs));
    ctx->memcpys++;
  }
  if (!ordered) {
    KVX_CUDA(cudaEventRecord(ctx->ev_copy_done, ctx->s_copy));
    KVX_CUDA(cudaStreamWaitEvent(stream, ctx->ev_copy_done, 0));
  }
  return KVX_OK;
}

void destroy_ctx(kvx_ctx* ctx) {
  if (!ctx) return;
  {
    DeviceGuard guard(ctx->device);
    if (ctx->s_kern) cudaStreamSynchronize(ctx->s_kern);
    if (ctx->s_copy) cudaStreamSynchronize(ctx->s_copy);
    if (ctx->s_aux) cudaStreamSynchronize(ctx->s_aux);
    for (uint8_t* s : ctx->slots) cudaFree(s);
    for (cudaEvent_t e : ctx->ev_ready) cudaEventDestroy(e);
    for (cudaEvent_t e : ctx->ev_free) cudaEventDestroy(e);
    for (const TimedLaunch& t : ctx->pending) {
      cudaEventDestroy(t.a);
      cudaEventDestroy(t.b);
    }
    for (cudaEvent_t e : ctx->spare_events) cudaEventDestroy(e);
    if (ctx->ev_in) cudaEventDestroy(ctx->ev_in);
    if (ctx->ev_kern_done) cudaEventDestroy(ctx->ev_kern_done);
    if (ctx->ev_copy_done) cudaEventDestroy(ctx->ev_copy_done);
    if (ctx->d_err) cudaFree(ctx->d_err);
    if (ctx->s_kern) cudaStreamDestroy(ctx->s_kern);
    if (ctx->s_copy) cudaStreamDestroy(ctx->s_copy);
    if (ctx->s_aux) cudaStreamDestroy(ctx->s_aux);
    cudaGetLastError();
  }
  delete ctx;
}

int32_t resolve_mode(int32_t m) {
  // Measured on GB300 (Grace host, NVLink-C2C) for a 128k-token 27B-class
  // context: zero-copy moves every step at the pinned-copy peak of both
  // directions (193 / 211 GB/s) from any pinned pool, including a tier in
  // POSIX shared memory; the staged pipeline reaches 0.98-0.99 of that only
  // from a pool wholly on huge pages.  Zero-copy also needs no staging memory,
  // no second pass over HBM and one launch per 64 chunks, and two replicas
  // moving at once get more of the bidirectional link with it.
  return m == KVX_MODE_AUTO ? (int32_t)KVX_MODE_ZEROCOPY : m;
}

}  // namespace

extern "C" {

int kv_abi_version(void) { return KVX_ABI_VERSION; }

int kv_last_cuda_error(void) { return g_last_cuda_error; }

const char* kv_last_error_message(void) { return g_last_error_text; }

const char* kv_status_string(kvx_status s) {
  switch (s) {
    case KVX_OK: return "ok";
    case KVX_EINVAL: return "invalid argument";
    case KVX_EALIGN: return "alignment rule broken";
    case KVX_ERANGE: return "out of range";
    case KVX_ENOTPINNED: return "host buffer is not page-locked";
    case KVX_ECUDA: return "CUDA runtime error";
    case KVX_ENOMEM: return "out of memory";
    case KVX_EDEVICE: return "pointer is not device memory of the context's GPU";
    case KVX_ENOENT: return "no committed tier entry for the key";
    case KVX_EBUSY: return "tier entry still in use";
    case KVX_ETIMEOUT: return "a bounded wait expired";
  }
  return "unknown status";
}

kvx_status kv_ctx_create(int device, const kvx_opts* opts, kvx_ctx** out) {
  return guarded([&]() -> kvx_status {
    if (!out) return KVX_EINVAL;
    *out = nullptr;
    kvx_opts o{};
    if (opts) o = *opts;
    for (int32_t m : {o.store_mode, o.load_mode})
      if (m != KVX_MODE_AUTO && m != KVX_MODE_STAGED && m != KVX_MODE_ZEROCOPY) return KVX_EINVAL;
    if (o.staging_slots != 0 && o.staging_slots < 2) return KVX_EINVAL;
    if (o.staging_slots > 64) return KVX_EINVAL;
    if (o.staging_slot_bytes < 0 || o.staging_slot_bytes % 16 != 0) return KVX_EINVAL;
    if (o.max_ctas < 0 || o.wait_cycles < 0) return KVX_EINVAL;
    if (o.flags & ~KVX_FLAGS_ALL) return KVX_EINVAL;
    if ((o.flags & KVX_FLAG_DEVICE_TMA) && (o.flags & KVX_FLAG_DEVICE_LSU)) return KVX_EINVAL;
    int count = 0;
    if (cudaGetDeviceCount(&count) != cudaSuccess) {
      g_last_cuda_error = (int)cudaGetLastError();
      return KVX_ECUDA;
    }
    if (device < 0 || device >= count) return KVX_EINVAL;
    DeviceGuard guard(device);
    if (!guard.ok) return KVX_ECUDA;
    kvx_ctx* ctx = new (std::nothrow) kvx_ctx;
    if (!ctx) return KVX_ENOMEM;
    ctx->device = device;
    ctx->opts = o;
    ctx->store_mode = resolve_mode(o.store_mode);
    ctx->load_mode = resolve_mode(o.load_mode);
    ctx->nslots = o.staging_slots ? o.staging_slots : kDefaultSlots;
    ctx->slot_bytes = o.staging_slot_bytes ? o.staging_slot_bytes : kDefaultSlotBytes;
    auto fail = [&](cudaError_t e) {
      g_last_cuda_error = (int)e;
      cudaGetLastError();
      destroy_ctx(ctx);
      return e == cudaErrorMemoryAllocation ? KVX_ENOMEM : KVX_ECUDA;
    };
    cudaError_t e;
    if ((e = cudaDeviceGetAttribute(&ctx->num_sms, cudaDevAttrMultiProcessorCount, device)) != cudaSuccess)
      return fail(e);
    // Host-link launches: half the SMs.  A quarter already saturates the link on
    // an idle GPU; half keeps it within 2-4 % of that while a full-GPU GEMM runs
    // beside the transfer (a quarter then loses 16-21 %), for 1-2 % more GEMM time.
    ctx->link_ctas = std::max(1, (ctx->num_sms + 1) / 2);
    if ((e = cudaStreamCreateWithFlags(&ctx->s_kern, cudaStreamNonBlocking)) != cudaSuccess) return fail(e);
    if ((e = cudaStreamCreateWithFlags(&ctx->s_copy, cudaStreamNonBlocking)) != cudaSuccess) return fail(e);
    if ((e = cudaStreamCreateWithFlags(&ctx->s_aux, cudaStreamNonBlocking)) != cudaSuccess) return fail(e);
    for (cudaEvent_t* ev : {&ctx->ev_in, &ctx->ev_kern_done, &ctx->ev_copy_done})
      if ((e = cudaEventCreateWithFlags(ev, cudaEventDisableTiming)) != cudaSuccess) return fail(e);
    for (int32_t k = 0; k < ctx->nslots; ++k) {
      cudaEvent_t a = nullptr, b = nullptr;
      if ((e = cudaEventCreateWithFlags(&a, cudaEventDisableTiming)) != cudaSuccess) return fail(e);
      ctx->ev_ready.push_back(a);
      if ((e = cudaEventCreateWithFlags(&b, cudaEventDisableTiming)) != cudaSuccess) return fail(e);
      ctx->ev_free.push_back(b);
    }
    if ((e = cudaMalloc(&ctx->d_err, 16)) != cudaSuccess) return fail(e);
    ctx->d_timeout = reinterpret_cast<int*>(ctx->d_err + 1);
    const long long init[2] = {kNoError, 0};
    if ((e = cudaMemcpy(ctx->d_err, init, sizeof(init), cudaMemcpyHostToDevice)) != cudaSuccess) return fail(e);
    for (int d = 0; d < 2; ++d)
      for (int l = 0; l < 2; ++l) ctx->move_occ[d][l] = move_ctas_per_sm(d, l);
    ctx->seg_occ = segment_ctas_per_sm();
    if ((e = prepare_tma_kernels()) != cudaSuccess) return fail(e);
    // the host-page touch threads, once per process, at set-up rather than
    // inside a transfer call
    if (!(o.flags & KVX_FLAG_NO_HOST_TOUCH)) start_touch_threads();
    if (ctx->store_mode == KVX_MODE_STAGED || ctx->load_mode == KVX_MODE_STAGED) {
      kvx_status st = ensure_staging(ctx);
      if (st != KVX_OK) {
        destroy_ctx(ctx);
        return st;
      }
    }
    *out = ctx;
    return KVX_OK;
  });
}

void kv_ctx_destroy(kvx_ctx* ctx) { destroy_ctx(ctx); }

kvx_status kv_chunk_layout(const kvx_pool* pool, int32_t chunk_tokens, int32_t tokens_in_chunk,
                           kvx_chunk_layout* out) {
  if (!out) return KVX_EINVAL;
  Geometry g;
  kvx_pool shape{};
  if (!pool) return KVX_EINVAL;
  shape = *pool;
  static void* const dummy[1] = {nullptr};
  if (!shape.layer_base) shape.layer_base = dummy;  // geometry needs no pointers
  kvx_status st = check_pool_shape(&shape, &g);
  if (st != KVX_OK) return st;
  if (chunk_tokens < 1 || tokens_in_chunk < 0 || tokens_in_chunk > chunk_tokens) return KVX_EINVAL;
  if (chunk_tokens % pool->block_tokens != 0) return KVX_EALIGN;
  out->chunk_tokens = chunk_tokens;
  out->tokens = tokens_in_chunk;
  out->head_stride = g.row;
  out->token_stride = (int64_t)pool->num_heads * g.row;
  out->kv_stride = out->token_stride * tokens_in_chunk;
  out->layer_stride = 2 * out->kv_stride;
  out->chunk_bytes = out->layer_stride * pool->num_layers;
  out->page_bytes = g.page_bytes;
  return KVX_OK;
}

kvx_status kv_store(kvx_ctx* ctx, const kvx_pool* pool, const int32_t* block_table, int64_t table_len,
                    int64_t tok_begin, int64_t tok_end, int32_t chunk_tokens, void* const* host_chunks,
                    int64_t n_chunks, kvx_stream_t stream) {
  return guarded([&]() -> kvx_status {
    TraceRange trace("kv_store");
    return transfer(ctx, pool, block_table, table_len, tok_begin, tok_end, chunk_tokens, host_chunks, n_chunks,
                    (cudaStream_t)stream, kPack, kHostChunks);
  });
}

kvx_status kv_load(kvx_ctx* ctx, const kvx_pool* pool, const int32_t* block_table, int64_t table_len,
                   int64_t tok_begin, int64_t tok_end, int32_t chunk_tokens, const void* const* host_chunks,
                   int64_t n_chunks, kvx_stream_t stream) {
  return guarded([&]() -> kvx_status {
    TraceRange trace("kv_load");
    return transfer(ctx, pool, block_table, table_len, tok_begin, tok_end, chunk_tokens,
                    const_cast<void* const*>(host_chunks), n_chunks, (cudaStream_t)stream, kUnpack, kHostChunks);
  });
}

kvx_status kv_pack(kvx_ctx* ctx, const kvx_pool* pool, const int32_t* block_table, int64_t table_len,
                   int64_t tok_begin, int64_t tok_end, int32_t chunk_tokens, void* const* dev_chunks,
                   int64_t n_chunks, kvx_stream_t stream) {
  return guarded([&]() -> kvx_status {
    TraceRange trace("kv_pack");
    return transfer(ctx, pool, block_table, table_len, tok_begin, tok_end, chunk_tokens, dev_chunks, n_chunks,
                    (cudaStream_t)stream, kPack, kDeviceChunks);
  });
}

kvx_status kv_unpack(kvx_ctx* ctx, const kvx_pool* pool, const int32_t* block_table, int64_t table_len,
                     int64_t tok_begin, int64_t tok_end, int32_t chunk_tokens, const void* const* dev_chunks,
                     int64_t n_chunks, kvx_stream_t stream) {
  return guarded([&]() -> kvx_status {
    TraceRange trace("kv_unpack");
    return transfer(ctx, pool, block_table, table_len, tok_begin, tok_end, chunk_tokens,
                    const_cast<void* const*>(dev_chunks), n_chunks, (cudaStream_t)stream, kUnpack, kDeviceChunks);
  });
}

kvx_status kv_state_store(kvx_ctx* ctx, int32_t num_layers, void* const* layer_base, int64_t num_slots,
                          int64_t slot_bytes, int64_t slot, void* host_obj, kvx_stream_t stream) {
  return guarded([&]() -> kvx_status {
    TraceRange trace("kv_state_store");
    return state_copy(ctx, num_layers, layer_base, num_slots, slot_bytes, slot, host_obj, (cudaStream_t)stream,
                      true);
  });
}

kvx_status kv_state_load(kvx_ctx* ctx, int32_t num_layers, void* const* layer_base, int64_t num_slots,
                         int64_t slot_bytes, int64_t slot, const void* host_obj, kvx_stream_t stream) {
  return guarded([&]() -> kvx_status {
    TraceRange trace("kv_state_load");
    return state_copy(ctx, num_layers, layer_base, num_slots, slot_bytes, slot, const_cast<void*>(host_obj),
                      (cudaStream_t)stream, false);
  });
}

kvx_status kv_fault_inject(const char* point, int32_t after_calls) {
  static const char* const points[] = {"launch", "memcpy", "event", "host_alloc", "tier_exit", "tma_wait"};
  std::lock_guard<std::mutex> lock(g_fault_mu);
  if (!point || !point[0]) {
    g_fault_point[0] = 0;
    g_fault_countdown.store(-1, std::memory_order_relaxed);
    return KVX_OK;
  }
  bool known = false;
  for (const char* q : points) known |= strcmp(q, point) == 0;
  if (!known || after_calls < 0) return KVX_EINVAL;
  snprintf(g_fault_point, sizeof(g_fault_point), "%s", point);
  g_fault_countdown.store(after_calls, std::memory_order_relaxed);
  return KVX_OK;
}

}  // extern "C"

namespace {
// KVX_FAULT="<point>[:<after_calls>]" arms one fault point when the library is
// loaded, so that a program which never calls kv_fault_inject (a serving
// engine under test) can be made to fail the same way.  A value naming no
// point, or a count that is not a non-negative integer, is reported on stderr
// and ignored.
struct FaultFromEnv {
  FaultFromEnv() {
    const char* v = getenv("KVX_FAULT");
    if (!v || !v[0]) return;
    char point[32];
    const char* colon = strchr(v, ':');
    const size_t len = colon ? (size_t)(colon - v) : strlen(v);
    long n = 0;
    bool ok = len > 0 && len < sizeof(point);
    if (ok && colon) {
      char* end = nullptr;
      n = strtol(colon + 1, &end, 10);
      ok = end != colon + 1 && *end == 0 && n >= 0 && n <= INT32_MAX;
    }
    if (ok) {
      memcpy(point, v, len);
      point[len] = 0;
      ok = kv_fault_inject(point, (int32_t)n) == KVX_OK;
    }
    if (!ok) fprintf(stderr, "libkvxfer: ignoring KVX_FAULT=%s (expected <point>[:<after_calls>])\n", v);
  }
} g_fault_from_env;
}  // namespace

extern "C" {

kvx_status kv_pool_view_check(const kvx_pool* pool, int32_t ndim, const int64_t* shape,
                              const int64_t* strides_bytes) {
  if (!pool || !shape || !strides_bytes) return KVX_EINVAL;
  Geometry g;
  kvx_pool p = *pool;
  static void* const dummy[1] = {nullptr};
  if (!p.layer_base) p.layer_base = dummy;
  kvx_status st = check_pool_shape(&p, &g);
  if (st != KVX_OK) return st;
  const int64_t P = pages_per_block(pool);
  const int64_t H = pool->num_heads, B = pool->block_tokens, D = pool->head_dim;
  int64_t want[6];
  int nd = 0;
  if (ndim == 6) {
    want[nd++] = pool->num_blocks / P;
    want[nd++] = P;
  } else if (ndim == 5) {
    want[nd++] = pool->num_blocks;
  } else {
    set_error_text("a pool layer view has 5 dimensions, or 6 with packed pages");
    return KVX_EINVAL;
  }
  want[nd++] = 2;
  want[nd++] = pool->layout == KVX_LAYOUT_HND ? H : B;
  want[nd++] = pool->layout == KVX_LAYOUT_HND ? B : H;
  want[nd++] = D;
  static const char* const names_hnd[] = {"pages", "K/V", "heads", "tokens per page", "head_dim"};
  static const char* const names_nhd[] = {"pages", "K/V", "tokens per page", "heads", "head_dim"};
  const char* const* names = pool->layout == KVX_LAYOUT_HND ? names_hnd : names_nhd;
  int64_t stride = pool->elem_bytes;
  for (int d = ndim - 1; d >= 0; --d) {
    const char* name = d >= ndim - 5 ? names[d - (ndim - 5)] : "logical blocks";
    char msg[192];
    if (shape[d] != want[d]) {
      snprintf(msg, sizeof(msg), "dimension %d (%s) is %lld, the %s pool description needs %lld", d, name,
               (long long)shape[d], pool->layout == KVX_LAYOUT_HND ? "HND" : "NHD", (long long)want[d]);
      set_error_text(msg);
      return KVX_EINVAL;
    }
    if (shape[d] > 1 && strides_bytes[d] != stride) {
      snprintf(msg, sizeof(msg), "dimension %d (%s) has stride %lld bytes, the %s layout needs %lld", d, name,
               (long long)strides_bytes[d], pool->layout == KVX_LAYOUT_HND ? "HND" : "NHD", (long long)stride);
      set_error_text(msg);
      return KVX_EINVAL;
    }
    stride *= shape[d];
  }
  return KVX_OK;
}

kvx_status kv_get_device_error(kvx_ctx* ctx, int64_t* first_bad_block) {
  if (!ctx || !first_bad_block) return KVX_EINVAL;
  DeviceGuard guard(ctx->device);
  if (!guard.ok) return KVX_ECUDA;
  std::lock_guard<std::mutex> lock(ctx->mu);
  long long v[2] = {kNoError, 0};
  const long long none[2] = {kNoError, 0};
  KVX_CUDA(cudaMemcpyAsync(v, ctx->d_err, sizeof(v), cudaMemcpyDeviceToHost, ctx->s_aux));
  KVX_CUDA(cudaStreamSynchronize(ctx->s_aux));
  KVX_CUDA(cudaMemcpyAsync(ctx->d_err, none, sizeof(none), cudaMemcpyHostToDevice, ctx->s_aux));
  KVX_CUDA(cudaStreamSynchronize(ctx->s_aux));
  *first_bad_block = (v[0] == kNoError) ? -1 : (int64_t)v[0];
  return (int)v[1] != 0 ? KVX_ETIMEOUT : KVX_OK;
}

kvx_status kv_ctx_stats(kvx_ctx* ctx, kvx_stats* out) {
  return guarded([&]() -> kvx_status {
    if (!ctx || !out) return KVX_EINVAL;
    DeviceGuard guard(ctx->device);
    if (!guard.ok) return KVX_ECUDA;
    std::lock_guard<std::mutex> lock(ctx->mu);
    for (const TimedLaunch& t : ctx->pending) {
      KVX_CUDA(cudaEventSynchronize(t.b));
      float ms = 0.f;
      KVX_CUDA(cudaEventElapsedTime(&ms, t.a, t.b));
      ctx->timed_ms[t.dir] += ms;
      ctx->timed[t.dir]++;
      ctx->timed_bytes[t.dir] += t.bytes;
      ctx->spare_events.push_back(t.a);
      ctx->spare_events.push_back(t.b);
    }
    ctx->pending.clear();
    out->kernel_launches = ctx->launches;
    out->memcpy_calls = ctx->memcpys;
    for (int d = 0; d < 2; ++d) {
      out->timed_launches[d] = ctx->timed[d];
      out->kernel_ms[d] = ctx->timed_ms[d];
      out->kernel_bytes[d] = ctx->timed_bytes[d];
    }
    return KVX_OK;
  });
}

kvx_status kv_ctx_reset_stats(kvx_ctx* ctx) {
  if (!ctx) return KVX_EINVAL;
  kvx_stats tmp;
  kvx_status st = kv_ctx_stats(ctx, &tmp);  // drains pending timings
  if (st != KVX_OK) return st;
  std::lock_guard<std::mutex> lock(ctx->mu);
  ctx->launches = ctx->memcpys = 0;
  for (int d = 0; d < 2; ++d) {
    ctx->timed[d] = ctx->timed_bytes[d] = 0;
    ctx->timed_ms[d] = 0.0;
  }
  return KVX_OK;
}

kvx_status kv_ctx_modes(const kvx_ctx* ctx, int32_t* store_mode, int32_t* load_mode) {
  if (!ctx) return KVX_EINVAL;
  if (store_mode) *store_mode = ctx->store_mode;
  if (load_mode) *load_mode = ctx->load_mode;
  return KVX_OK;
}

}  // extern "C"
