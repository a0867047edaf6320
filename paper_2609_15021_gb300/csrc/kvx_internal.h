// kvx_internal.h -- declarations shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <new>
#include <vector>

#include "kvxfer.h"

namespace kvx {

constexpr int kMaxJobs = 64;      // chunk-side segments per kernel launch
constexpr int kThreads = 256;     // threads per CTA of the move kernels
constexpr int kMaxSegments = 96;  // segments per opaque-copy launch (params < 4 KiB)

enum Dir : int { kPack = 0, kUnpack = 1 };

// One contiguous chunk-side region: layers [l0, l0 + nl) of one chunk.
struct Job {
  uint8_t* chunk;       // chunk-side address of layer l0 (device, staging or mapped host)
  int64_t first_block;  // logical block index of the chunk's first token
  int64_t unit_end;     // exclusive prefix sum of units up to and including this job
  int32_t tokens;       // T_c: tokens held by the chunk
  int32_t l0;           // first layer of the region
};

// Kernel parameters of one pack/unpack launch (passed by value, < 4 KiB).
struct MoveParams {
  uint8_t* layer_base[KVX_MAX_LAYERS];
  Job jobs[kMaxJobs];
  const int32_t* table;        // device block table
  long long* err;              // device error word (lowest bad logical block)
  int64_t num_blocks;          // pages per layer
  int64_t page_bytes;          // 2 * H * B * row
  int64_t total_units;         // units of this launch
  int32_t n_jobs;
  int32_t blocks_per_chunk;    // C / B: kernel pages per chunk
  int32_t ppb;                 // pages per logical block named by the table (>= 1)
  int32_t B, H, R;             // tokens per page, heads, row bytes
  int32_t fast;                // 1 if R/16 is a power of two <= 32
  int32_t vpr_shift;           // log2(R / 16) when fast
  int32_t rpi_div_h, rpi_mod_h; // (32 / (R/16)) / H and % H when fast
};

// One contiguous byte range of an opaque copy (a recurrent-state slot).
struct Segment {
  const uint8_t* src;
  uint8_t* dst;
  int64_t byte_end;  // exclusive prefix sum of segment bytes
};

// The segments of one launch are treated as one byte stream cut into units of
// unit_bytes (a multiple of 512; the last unit may be shorter) that may span
// segment ends, so every warp gets the same share of bytes.
struct SegmentParams {
  Segment seg[kMaxSegments];
  int64_t total_bytes;
  int64_t unit_bytes;
  int64_t total_units;
  int32_t n_seg;
};

// Byte geometry of a pool description.
struct Geometry {
  int64_t row;          // head_dim * elem_bytes
  int64_t page_bytes;   // 2 * H * B * row
  int64_t layer_bytes;  // num_blocks * page_bytes
};

enum Where : int { kHostChunks = 0, kDeviceChunks = 1 };

// Argument checks shared by the pack/unpack entry points (kvxfer.cu): pool
// shape and memory, token range, block table, and every chunk pointer of
// [t0, t1) on `device`.  Fills *g and *n (chunks in the range) and, when
// `side` is not null, side[i] = the address of chunk i that the kernel or
// copy engine uses (mapped address for zero-copy host chunks).  Enqueues
// nothing and allocates nothing.
kvx_status check_transfer(int device, const kvx_pool* P, const int32_t* table, int64_t table_len, int64_t t0,
                          int64_t t1, int32_t C, void* const* chunks, int64_t n_chunks, cudaStream_t stream,
                          int where, int mode, Geometry* g, int64_t* n, uint8_t** side);
void init_params(MoveParams* p, long long* err, const kvx_pool* P, const Geometry& g, const int32_t* table,
                 int32_t C);
void push_job(MoveParams* p, uint8_t* chunk_side, int64_t first_block, int32_t tokens, int32_t l0, int32_t nl);
int64_t chunk_bytes(const kvx_pool* P, const Geometry& g, int64_t tokens);
void set_error_text(const char* text);

// Launchers (pack_kernels.cu).  Return the cudaError_t of the launch.
cudaError_t launch_move(int dir, int layout, const MoveParams& p, int grid, cudaStream_t s);
cudaError_t launch_segments(const SegmentParams& p, int grid, cudaStream_t s);
// Loads the pack kernels into the current context if lazy loading has not yet.
cudaError_t load_pack_kernels();
// Bounded waits of the TMA kernels: the limit of each mbarrier wait in SM
// cycles, the device int set when one expires, and the unit (global index, -1
// for none) whose load a kernel arms without issuing it (fault point "tma_wait").
struct TmaWait {
  long long cycles;
  long long stall_unit;
  int* timeout;
};
constexpr long long kDefaultWaitCycles = 4000000000ll;  // about 2 s at the maximum SM clock
// Bulk-copy (TMA) variant for chunks in device memory (tma_kernels.cu): one
// warp per CTA, `stages` shared-memory stages of stage_bytes each.
cudaError_t launch_move_tma(int dir, int layout, const MoveParams& p, int grid, int stage_bytes, int stages,
                            const TmaWait& wt, cudaStream_t s);
// Sets the TMA kernels' shared-memory limit for the current device (once per
// context creation; never on the launch path).
cudaError_t prepare_tma_kernels();
// Tensor-map variant for HND pools: one TMA box per full page half.
constexpr int kTensorMapBytes = 128;
// Encodes one tensor map per layer of P (kTensorMapBytes each) into `out`;
// false if the pool's shape cannot be described (the row-copy variant is used).
bool encode_tensor_maps(const kvx_pool* P, int64_t row_bytes, void* out);
cudaError_t launch_move_tmap(int dir, const MoveParams& p, const void* maps, int num_layers, int grid,
                             int stage_bytes, int stages, const TmaWait& wt, cudaStream_t s);
int move_ctas_per_sm(int dir, int layout);
int segment_ctas_per_sm();
// Shared tier (tier_kernels.cu): publication of up to kMaxPublish commits in
// one launch.  Thread j makes a system-scope release store of seq0 + j to the
// 8-byte flag at meta + slot[j] * stride + offset (meta: the device address of
// the mapped slot table).
constexpr int kMaxPublish = 512;
struct TierPublish {
  uint8_t* meta;
  int64_t stride, offset;
  uint64_t seq0;
  int32_t n;
  int32_t slot[kMaxPublish];
};
cudaError_t launch_tier_publish(const TierPublish& b, cudaStream_t s);
// Loads the publication kernel (at tier open, never inside a commit).
cudaError_t prepare_tier_kernels();

// Host-page touch (host_touch.cpp).  start_touch_threads starts the
// process-wide reading threads once (kv_ctx_create); touch_before_transfer
// reads one byte per host page of the chunks of a transfer on those threads
// and enqueues on `stream` a host function that waits for the reads, so the
// transfer behind it follows them (nothing while `stream` is capturing; on the
// calling thread where no threads or host function are to be had).  Neither
// throws: the touch is only a speed-up.
void start_touch_threads();
void touch_before_transfer(void* const* chunks, const std::vector<int32_t>& tokens, const kvx_pool* P,
                           const Geometry& g, cudaStream_t stream);

// Records the last CUDA error seen by this thread (kv_last_cuda_error).
void set_last_cuda_error(int e);

// Host-side fault injection (kv_fault_inject): true if the armed point fails now.
bool fault_point(const char* point);

// Runs an entry point's body so that no C++ exception leaves the C ABI: a
// failed host allocation (a caller's absurd count, say) returns KVX_ENOMEM.
template <class F>
kvx_status guarded(F&& body) {
  try {
    return body();
  } catch (const std::bad_alloc&) {
    set_error_text("out of host memory");
    return KVX_ENOMEM;
  } catch (...) {
    set_error_text("unexpected failure inside the library");
    return KVX_EINVAL;
  }
}

}  // namespace kvx
