/*
 * kvxfer.h -- C ABI of the paged-KV <-> pinned-host-chunk transfer library
 * (libkvxfer.so, CUDA, sm_103a).
 *
 * The paper (Sec. 2, Fig. 1) runs full inference replicas, one per GPU, that
 * share one host-memory KV tier.  Each replica keeps its KV cache as a pool of
 * pages (Table 1: paged cache, HND layout); the shared tier holds fixed-token
 * chunks (Table 1: 1,568-token chunks in a 256 GiB RAM pool).  Storing a
 * prefix gathers its pages into packed chunks in pinned host memory; loading
 * it on another replica scatters the chunks into freshly allocated pages
 * (Sec. 3.2).  Every copy is ordered on the caller's current CUDA stream:
 * the paper's diagnosed corruption (Sec. 3.2, Fig. 2) is a copy that omits
 * exactly this dependency.
 *
 * Data layout (all sizes in bytes unless stated; row = head_dim * elem_bytes):
 *   pool layer l   : num_blocks pages, page = [2 (K,V)][H][B][row] for
 *                    KVX_LAYOUT_HND, [2][B][H][row] for KVX_LAYOUT_NHD.
 *   block table    : int32 device array; entry i names logical block i, i.e.
 *                    the pages of tokens [i*P*B, (i+1)*P*B) (P =
 *                    kvx_pool.pages_per_block, 1 unless pages are packed).
 *   chunk c        : tokens [c*C, min((c+1)*C, tok_end)), packed densely as
 *                    [layer][2 (K,V)][token][head][row]; a short last chunk
 *                    holds fewer tokens and is not padded.  The layout does
 *                    not depend on the page layout, so HND and NHD pools
 *                    exchange chunks (Sec. 3.1: a wrong view of the bytes was
 *                    the paper's first corruption).
 *   host chunk i   : the i-th chunk of the call's range, i.e. chunk
 *                    tok_begin/C + i; page-locked host memory, 16-byte
 *                    aligned, at least kv_chunk_layout(...).chunk_bytes long.
 *
 * Threading: a kvx_ctx may be shared by host threads (calls are serialised
 * inside).  Calls are asynchronous with respect to the host.
 *
 * Ordering: zero-copy and device-chunk moves and state copies are enqueued on
 * `stream` itself, so stream order makes them follow the work already there
 * and precede what comes after.  The staged pipeline runs on two side streams
 * that wait on an event recorded on `stream`, and `stream` then waits on
 * events recorded after its last piece of work.
 *
 * CUDA graphs: kv_store, kv_load, kv_pack and kv_unpack allocate nothing per
 * call (the staging ring of KVX_MODE_STAGED is made by kv_ctx_create), and
 * what they enqueue is joined to `stream`.  They may therefore be captured
 * from a capturing `stream` and replayed; the buffers and ranges of the
 * capture are replayed.  While `stream` is capturing, its device is not
 * checked (the query would end the capture).
 *
 * Error behaviour: argument errors return before anything is enqueued and
 * leave every buffer untouched.  A block-table entry outside [0, num_blocks)
 * is found on the device: it names no page, so a store writes zero bytes for
 * its tokens (never stale staging bytes) and a load writes nothing for them;
 * the lowest such logical block index is kept for kv_get_device_error().  A
 * CUDA failure while work is being enqueued returns KVX_ECUDA after making
 * `stream` wait for whatever was already enqueued.  No call aborts the
 * process, traps on the device, or waits without a bound.
 */
#ifndef KVXFER_H
#define KVXFER_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define KVX_ABI_VERSION 3
#define KVX_MAX_LAYERS 128 /* layers per pool description */

/* Same handle as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st* kvx_stream_t;

typedef enum {
  KVX_OK = 0,
  KVX_EINVAL = -1,     /* null pointer, non-positive size, unknown enum value   */
  KVX_EALIGN = -2,     /* tok_begin % C, C % B, row % 16 or a pointer % 16 != 0 */
  KVX_ERANGE = -3,     /* tok_end beyond the table, too few chunks, bad slot    */
  KVX_ENOTPINNED = -4, /* a host buffer is not page-locked host memory          */
  KVX_ECUDA = -5,      /* a CUDA runtime call failed (kv_last_cuda_error)       */
  KVX_ENOMEM = -6,     /* staging or device allocation failed                   */
  KVX_EDEVICE = -7,    /* a device pointer is not device memory of ctx's GPU    */
  KVX_ENOENT = -8,     /* tier: no committed entry for the key                  */
  KVX_EBUSY = -9,      /* tier: the entry is still in use and cannot be rewritten */
  KVX_ETIMEOUT = -10   /* a bounded wait expired: inside a kernel (the kernel
                          returned early and its output is incomplete), or
                          kv_tier_wait's host wait                             */
} kvx_status;

typedef enum { KVX_LAYOUT_HND = 0, KVX_LAYOUT_NHD = 1 } kvx_layout;

/* How host chunks are filled and read.  Both move exactly the same bytes. */
typedef enum {
  KVX_MODE_AUTO = 0,     /* library's measured default: ZEROCOPY both ways
                            (GB300 + Grace: the link's ceiling every step on
                            every pool kind measured; STAGED reaches 0.98-0.99
                            of it only from huge-page pools, KVX_HOST_HUGE,
                            and varies from step to step on others)           */
  KVX_MODE_STAGED = 1,   /* pack into a device staging ring, then
                            cudaMemcpyAsync over the host link on a side stream,
                            pack of batch i+1 overlapping the copy of batch i  */
  KVX_MODE_ZEROCOPY = 2  /* the kernel reads/writes the mapped pinned chunks
                            directly over the host link; no staging            */
} kvx_mode;

/* Options flags */
#define KVX_FLAG_TIME_KERNELS 0x1u /* record CUDA events around every kernel
                                      launch; read with kv_ctx_stats()        */
#define KVX_FLAG_UNORDERED 0x2u    /* NEGATIVE CONTROL ONLY: drop the wait on
                                      the caller's stream, reproducing the
                                      paper's missing dependency (Sec. 3.2).
                                      Results are then undefined.             */
/* Device-side moves (kv_pack, kv_unpack, staged mode) use, by default, the
   TMA kernel when a K or V page half is at most 48 KiB: one tensor-map box
   per page half for HND pools, one bulk copy per side for NHD pools (whose
   page halves are contiguous), staged through shared memory; both measured
   faster than the load/store kernel on GB300.  HND pools that no tensor map
   describes use the 16-byte load/store kernel.  Zero-copy moves always use
   the load/store kernel.  The flags below force one of them for device-side
   moves.                                                                     */
#define KVX_FLAG_DEVICE_TMA 0x4u   /* TMA everywhere it fits, with one bulk
                                      copy per row of HND pages no tensor map
                                      describes                              */
#define KVX_FLAG_DEVICE_LSU 0x8u   /* the 16-byte load/store kernel always   */
/* Host memory after idle time.  Measured on GB300 (Grace host): after the
   pinned pool had sat untouched for 10 s, a 128k-token restore through it took
   337 ms instead of 159 ms (219 ms after 3 s, 165-168 after 1 s), the next one
   159 ms again; the slowdown followed parts of the pool's host memory, not the
   GPU or the link.  A CPU read of one byte per host page of the chunks just
   before the transfer (13.8 ms on one thread for 33 GB) brought it back to
   159 ms.  So when a context has begun no transfer for more than 1 s,
   kv_store and kv_load read one byte of every host page of the chunks they
   are given before moving them.  The reads run on a pool of up to 16
   persistent library threads (started once per process, by the first
   kv_ctx_create), not on the calling thread: the call enqueues on `stream`,
   ahead of its transfer, a host function (cudaLaunchHostFunc) that waits
   until the pages have been read (2-4 ms for 33 GB on GB300), so the transfer
   follows the reads, the call itself returns without waiting, and `stream`
   completes only after the last read.  It is skipped while `stream` is being captured.  If the library
   cannot start threads (or in a forked child, which inherits none) the
   calling thread reads the pages itself before it enqueues.  kv_host_touch
   does the same reads on request.  This flag turns the idle-time touch off. */
#define KVX_FLAG_NO_HOST_TOUCH 0x10u
/* Every defined flag.  kv_ctx_create rejects (KVX_EINVAL) other bits, and
   KVX_FLAG_DEVICE_TMA together with KVX_FLAG_DEVICE_LSU.                     */
#define KVX_FLAGS_ALL 0x1Fu

typedef struct {
  int32_t store_mode;         /* kvx_mode                                       */
  int32_t load_mode;          /* kvx_mode                                       */
  int32_t staging_slots;      /* staged ring depth (>= 2); 0 = 4                */
  int64_t staging_slot_bytes; /* bytes per slot; 0 = 128 MiB; a slot must hold
                                 one layer of one chunk                         */
  int32_t max_ctas;           /* cap on CTAs per kernel launch; 0 = default:
                                 launches that read or write host memory
                                 (zero-copy) run one 8-warp CTA per two SMs,
                                 which saturates the host link even beside the
                                 replica's compute and leaves most of each SM
                                 to it; device-side launches give every
                                 32 KiB unit its own warp or CTA.  With a cap,
                                 each warp or CTA strides over many units       */
  uint32_t flags;             /* KVX_FLAG_*                                     */
  int64_t wait_cycles;        /* limit of every bounded wait inside a kernel, in
                                 SM cycles (the TMA engine's waits for its
                                 global -> shared copies); 0 = 4e9, about 2 s at
                                 the maximum SM clock.  When a wait expires, the
                                 CTA issues no further copy, waits once more
                                 (same limit) for each copy it has started,
                                 then returns; kv_get_device_error reports
                                 KVX_ETIMEOUT and that call's output is
                                 incomplete.  The context stays usable.         */
} kvx_opts;

/* Caller-owned description of one paged KV pool (device memory). */
typedef struct {
  int32_t num_layers;        /* 1 .. KVX_MAX_LAYERS                            */
  void* const* layer_base;   /* host array [num_layers] of device pointers, each
                                16-byte aligned, num_blocks * page_bytes long   */
  int64_t num_blocks;        /* pages per layer                                */
  int32_t block_tokens;      /* B: tokens per page                             */
  int32_t num_heads;         /* H: KV heads                                    */
  int32_t head_dim;          /* D: elements per head vector                    */
  int32_t elem_bytes;        /* e: bytes per element (bf16 = 2, fp8 = 1, ...)  */
  int32_t layout;            /* kvx_layout                                     */
  int32_t pages_per_block;   /* P: pages per logical block named by the block
                                table (0 or 1: the table names pages).  Sec.
                                3.1: a 1,568-token logical block packs 49 pages
                                of 32 tokens; logical block b is pages
                                b*P .. b*P+P-1, so token t lies in page
                                table[(t/B)/P]*P + (t/B)%P.  num_blocks (pages)
                                must be a multiple of P.                        */
} kvx_pool;

/* Byte geometry of one packed chunk holding tokens_in_chunk tokens. */
typedef struct {
  int32_t chunk_tokens;      /* C                                              */
  int32_t tokens;            /* tokens held (<= C)                             */
  int64_t chunk_bytes;       /* L * 2 * tokens * H * row                       */
  int64_t layer_stride;      /* 2 * tokens * H * row                           */
  int64_t kv_stride;         /* tokens * H * row                               */
  int64_t token_stride;      /* H * row                                        */
  int64_t head_stride;       /* row                                            */
  int64_t page_bytes;        /* bytes of one pool page (2 * H * B * row)       */
} kvx_chunk_layout;

/* Counters kept by a context.  Index [0] is the pack direction (kv_store,
   kv_pack, kv_state_store), [1] the unpack direction.  Durations are kept
   only with KVX_FLAG_TIME_KERNELS: a pair of CUDA events is recorded around
   each kernel launch on the stream it runs on. */
typedef struct {
  int64_t kernel_launches;   /* kernels this context has launched              */
  int64_t memcpy_calls;      /* cudaMemcpyAsync calls issued (staged mode)     */
  int64_t timed_launches[2]; /* launches with a recorded duration              */
  double kernel_ms[2];       /* summed durations of timed launches             */
  int64_t kernel_bytes[2];   /* algorithmic bytes of timed launches: every byte
                                read plus every byte written, host or device   */
} kvx_stats;

typedef struct kvx_ctx kvx_ctx;

/*
 * Create a context on `device`: side streams, per-slot events, the staging
 * ring (KVX_MODE_STAGED only, allocated on first use) and a device error word.
 * opts may be NULL (all defaults).  Returns KVX_ENOMEM if an allocation fails.
 */
kvx_status kv_ctx_create(int device, const kvx_opts* opts, kvx_ctx** out);

/* Synchronises the context's streams, then frees everything it owns. */
void kv_ctx_destroy(kvx_ctx* ctx);

/*
 * Geometry of a chunk (Table 1: fixed-token chunks of the shared tier).
 * chunk_tokens must be a positive multiple of pool->block_tokens and
 * 0 <= tokens_in_chunk <= chunk_tokens.  Pure host arithmetic.
 */
kvx_status kv_chunk_layout(const kvx_pool* pool, int32_t chunk_tokens, int32_t tokens_in_chunk,
                           kvx_chunk_layout* out);

/*
 * Check that a framework's view of one pool layer -- its shape and byte
 * strides, outermost dimension first -- is the layout `pool` declares.
 * Sec. 3.1: the paper's first corruption came from reading the same bytes
 * with a different logical shape; its NHD attempt failed a divisibility check
 * because the transfer patch's view and the attention backend's shape and
 * strides disagreed.  A mismatch must be rejected, never silently mis-copied.
 * Accepted views (element strides, C-contiguous, times elem_bytes in bytes):
 *   HND: [num_blocks, 2, H, B, D]       or packed [num_blocks/P, P, 2, H, B, D]
 *   NHD: [num_blocks, 2, B, H, D]       or packed [num_blocks/P, P, 2, B, H, D]
 * (P = pool->pages_per_block).  Pure host check; pool->layer_base is not read.
 * Returns KVX_OK, or KVX_EINVAL with kv_last_error_message naming the first
 * dimension or stride that disagrees.  A view whose H and B are equal and
 * whose layout differs cannot be told apart by shape; its strides still must
 * be the declared layout's.
 */
kvx_status kv_pool_view_check(const kvx_pool* pool, int32_t ndim, const int64_t* shape,
                              const int64_t* strides_bytes);

/*
 * Store (Sec. 3.2 gather; Fig. 2 lower panel ordering): pack tokens
 * [tok_begin, tok_end) of the pages named by block_table into host_chunks.
 *   block_table : device int32 [table_len]; pages of logical blocks 0..
 *   tok_begin   : multiple of chunk_tokens (chunks start on aligned recovery
 *                 boundaries, Sec. 2.2);
 *   tok_end     : tok_begin <= tok_end <= table_len * P * B, where
 *                 P = pool->pages_per_block (1 unless pages are packed into
 *                 logical blocks) and B = pool->block_tokens; beyond that
 *                 KVX_ERANGE.
 *   host_chunks : host array [n_chunks] of pinned host pointers; chunk i gets
 *                 chunk tok_begin/C + i; n_chunks >= ceil(tok_end/C) - tok_begin/C.
 *   stream      : the caller's current stream.  All reads of the pool happen
 *                 after the work already enqueued on it; work enqueued on it
 *                 after this call runs after the chunks are written.
 * The host must synchronise `stream` before reading the chunks (Fig. 2
 * caption: completion must precede host consumption).  Only the first
 * chunk_bytes of each chunk are written.
 */
kvx_status kv_store(kvx_ctx* ctx, const kvx_pool* pool, const int32_t* block_table, int64_t table_len,
                    int64_t tok_begin, int64_t tok_end, int32_t chunk_tokens,
                    void* const* host_chunks, int64_t n_chunks, kvx_stream_t stream);

/*
 * Load (Sec. 3.2 scatter into freshly allocated pages): the inverse of
 * kv_store into the pages named by block_table.  Exactly the page rows of
 * tokens [tok_begin, tok_end) are written; all other pool bytes (other pages,
 * slots past tok_end in a partial last page) are left untouched.  Host chunks
 * must not be modified or freed before `stream` has passed this call.
 * A physical page listed twice in block_table is a caller error (the bytes
 * written there are then unspecified).
 */
kvx_status kv_load(kvx_ctx* ctx, const kvx_pool* pool, const int32_t* block_table, int64_t table_len,
                   int64_t tok_begin, int64_t tok_end, int32_t chunk_tokens,
                   const void* const* host_chunks, int64_t n_chunks, kvx_stream_t stream);

/*
 * Device-side pack / unpack: kv_store / kv_load with chunks in device memory
 * of ctx's GPU (16-byte aligned) instead of pinned host memory.  Same rules,
 * one kernel pass, ordered on `stream`.
 */
kvx_status kv_pack(kvx_ctx* ctx, const kvx_pool* pool, const int32_t* block_table, int64_t table_len,
                   int64_t tok_begin, int64_t tok_end, int32_t chunk_tokens,
                   void* const* dev_chunks, int64_t n_chunks, kvx_stream_t stream);
kvx_status kv_unpack(kvx_ctx* ctx, const kvx_pool* pool, const int32_t* block_table, int64_t table_len,
                     int64_t tok_begin, int64_t tok_end, int32_t chunk_tokens,
                     const void* const* dev_chunks, int64_t n_chunks, kvx_stream_t stream);

/*
 * Recurrent-state snapshot (Sec. 2.2: a recurrent page -- convolution state,
 * recurrent state and padding -- is moved as opaque addressable bytes; a
 * hybrid prefix is recovered only with the snapshot taken at its boundary).
 *   layer_base : host array [num_layers] of device pointers to
 *                [num_slots][slot_bytes] state pools.
 *   host_obj   : pinned host buffer [num_layers][slot_bytes].
 * kv_state_store copies slot `slot` of every layer into host_obj;
 * kv_state_load copies host_obj into slot `slot`.  Ordered on `stream`.
 */
kvx_status kv_state_store(kvx_ctx* ctx, int32_t num_layers, void* const* layer_base, int64_t num_slots,
                          int64_t slot_bytes, int64_t slot, void* host_obj, kvx_stream_t stream);
kvx_status kv_state_load(kvx_ctx* ctx, int32_t num_layers, void* const* layer_base, int64_t num_slots,
                         int64_t slot_bytes, int64_t slot, const void* host_obj, kvx_stream_t stream);

/*
 * kv_store without any allocation (the paper has no counterpart: this entry
 * point exists for callers that cannot allocate device memory).
 *
 * Who needs it: code running under an engine whose memory pool owns all free
 * GPU memory and must not see allocations it does not track, or code that must
 * not let cudaMalloc/cudaFree synchronise the device mid-pipeline.  kv_store
 * needs a context, and a context allocates a staging ring, streams and events.
 * This call creates nothing: it packs into a static device array of
 * KVX_NOALLOC_SCRATCH_BYTES (64 MiB, plus 256 bytes) that every GPU loading
 * this part of the library holds until the process exits, and copies each
 * packed batch to the host chunks with cudaMemcpyAsync, all on `stream` and in
 * stream order (no overlap of packing and copying, unlike kv_store).
 *
 * Arguments, layout, alignment, pinned-memory and range rules are those of
 * kv_store; it runs on the calling thread's current device.  One layer of one
 * chunk (2 * tokens * H * head_dim * elem_bytes) must fit in the array, else
 * KVX_ERANGE (kv_last_error_message names both sizes).
 *   dev_first_bad_block : NULL, or a device int64 that the kernel lowers by
 *                         atomicMin to the lowest logical block whose table
 *                         entry is out of range (initialise it, e.g. to
 *                         INT64_MAX); such tokens are stored as zeros.
 * Set-up: the first call in a CUDA context (on the thread's current device)
 * looks up the array's device address with cudaGetSymbolAddress, loads the
 * pack kernels, and keeps the address for that context.  A call in another
 * context -- a driver-API context the caller made current, or the new primary
 * context after cudaDeviceReset -- repeats this set-up there.  With CUDA's
 * lazy module loading (the default) this set-up is also when the GPU takes the
 * array's 64 MiB, so an engine that reserves all free GPU memory must make one
 * call before it does.  A call with an empty range (tok_begin == tok_end,
 * arguments otherwise valid) makes the set-up and moves nothing: make it at
 * start-up, before the engine reserves GPU memory and before any stream
 * capture.  Later calls in the same context allocate nothing on the device or
 * the host.  All calls share the one array and nothing in it needs to start
 * at zero (every staged byte is written before it is copied).  Calls that
 * overlap on the GPU -- on different streams without an ordering between
 * them -- race on the array: order them.
 */
#define KVX_NOALLOC_SCRATCH_BYTES (64ll << 20)
kvx_status kv_store_noalloc(const kvx_pool* pool, const int32_t* block_table, int64_t table_len,
                            int64_t tok_begin, int64_t tok_end, int32_t chunk_tokens, void* const* host_chunks,
                            int64_t n_chunks, int64_t* dev_first_bad_block, kvx_stream_t stream);

/*
 * Page-locked host memory for a shared chunk pool (Sec. 3.3: the shared tier
 * is one full-size pinned allocation; the paper's 256 GiB + 4096 B request
 * was rounded up to a power of two by the framework's pinned allocator and
 * silently fell back to pageable memory).  kv_host_alloc returns exactly
 * `bytes` of page-locked memory, portable to every device and mapped for
 * zero-copy, from the driver's pinned allocator (cudaHostAlloc, asked for
 * exactly that size).  Measured on GB300 (Grace host): zero-copy transfers,
 * the default mode, held the link peak from such pools in every benchmark
 * run, where pools the library mapped on huge pages stalled at times after
 * other pinning, freeing or forking in the same process.  For copy-engine
 * transfers (KVX_MODE_STAGED) ask for huge pages (kv_host_alloc_ex with
 * KVX_HOST_HUGE): the copy engines reach the link peak only from them.
 * Failure is KVX_ENOMEM or KVX_ECUDA, never a pageable fallback.  Free with
 * kv_host_free (NULL is ignored).
 */
kvx_status kv_host_alloc(int64_t bytes, void** out);
/*
 * kv_host_alloc placed on one host NUMA node.  On a host with several memory
 * nodes the pool belongs on the node next to the GPU that uses it, or every
 * zero-copy access also crosses the link between sockets.  numa_node >= 0
 * names the node; KVX_NUMA_NEAREST asks for the node CUDA reports as closest
 * to the current device (no placement if it reports none).  The library maps
 * the pool itself (huge pages where they fit, as KVX_HOST_HUGE, else base
 * pages) and gives it a preferred-node policy (mbind) before it is faulted in.
 * KVX_EINVAL for a node that does not exist, KVX_ENOMEM if the node has less
 * free memory than `bytes` or the memory cannot be pinned (never a pageable
 * fallback).  *numa_out (may be NULL) receives the node of the first page,
 * or -1 if unknown.  Free with kv_host_free.
 */
#define KVX_NUMA_NEAREST (-1)
kvx_status kv_host_alloc_numa(int32_t numa_node, int64_t bytes, void** out, int32_t* numa_out);
/*
 * Both of the above, with the choices spelled out.  numa_node: KVX_NUMA_ANY
 * (no placement), KVX_NUMA_NEAREST, or a node.  flags:
 *   KVX_HOST_DRIVER  the driver's pinned allocator (the default without a
 *                    placement); numa_node must be KVX_NUMA_ANY.
 *   KVX_HOST_HUGE    the library's own mapping on transparent huge pages,
 *                    rounded up to whole huge pages (never to a power of
 *                    two), for copy-engine transfers.  A pool that whole huge
 *                    pages would overshoot by more than an eighth (for 512 MiB
 *                    pages: anything below 4 GiB that is not a near multiple),
 *                    or that huge pages cannot wholly back, or any pool on a
 *                    host without transparent huge pages, comes from the
 *                    driver's allocator instead (no placement) or from base
 *                    pages (placement).  Not with KVX_HOST_DRIVER.
 * A mapped pool is not inherited by child processes (MADV_DONTFORK): on GB300
 * a fork of the owning process, even to start a subprocess, otherwise
 * stalled the next zero-copy store through it for seconds.  A child must not
 * touch the pool.  kv_host_alloc(b, o) is kv_host_alloc_ex(b, KVX_NUMA_ANY, 0,
 * o, NULL).  kv_host_pool_info tells what a call returned.
 */
#define KVX_NUMA_ANY (-2)
#define KVX_HOST_DRIVER 0x1u
#define KVX_HOST_HUGE 0x2u
kvx_status kv_host_alloc_ex(int64_t bytes, int32_t numa_node, uint32_t flags, void** out, int32_t* numa_out);

/*
 * What backs a pool from the calls above.  A pool of the library's own
 * mapping is either wholly on huge pages or wholly on base pages, never a
 * mixture: on GB300 a pool partly on huge pages zero-copied at 76 GB/s where
 * either kind alone reached 202 GB/s.  When huge pages cannot back the whole
 * pool, the call falls back to the driver's allocator (no placement asked) or
 * to base pages (placement asked).
 */
#define KVX_HOST_SOURCE_DRIVER 0 /* cudaHostAlloc                               */
#define KVX_HOST_SOURCE_MAPPED 1 /* the library's mapping, then cudaHostRegister */
typedef struct {
  int64_t bytes;            /* requested                                        */
  int64_t mapped_bytes;     /* mapped (rounded up to whole pages)               */
  int64_t huge_page_bytes;  /* backed by transparent huge pages when pinned     */
  int32_t numa_node;        /* node of the first page, or -1 if unknown          */
  int32_t source;           /* KVX_HOST_SOURCE_*                                 */
} kvx_host_pool_info;
/* KVX_ENOENT if `host` is not the start of a pool these calls returned. */
kvx_status kv_host_pool_info(const void* host, kvx_host_pool_info* info);
/* Frees kv_host_alloc and kv_host_alloc_numa memory; NULL and pointers the
   library did not allocate are ignored. */
void kv_host_free(void* host);

/*
 * Read one byte of every host page of n ranges (ptrs[i], bytes[i] long) on the
 * library's touch threads and the calling thread, returning when all have been
 * read.  The idle-time touch of kv_store / kv_load (KVX_FLAG_NO_HOST_TOUCH)
 * done ahead of time: a caller that knows a restore is coming (a request that
 * hit the shared tier, say) can warm the chunks' pages before it calls
 * kv_load.  Each range must be readable host memory (pinned or not) for the
 * duration of the call.  KVX_EINVAL for n < 0, a negative size, or a null
 * pointer with a positive size; zero-sized ranges are skipped.  Gives up after
 * 5 s (pages left unread) and still returns KVX_OK: the touch is only a
 * speed-up.
 */
kvx_status kv_host_touch(void* const* ptrs, const int64_t* bytes, int64_t n);

/* ------------------------------------------------------------------------
 * Shared host tier (Table 1: one pinned RAM pool of fixed-token chunks with
 * LRU eviction).  A tier is n_slots fixed-size slots in one pool, each slot
 * holding one chunk under a 64-bit key.  Entries follow the ordering rule of
 * Sec. 3.2: a writer reserves a slot, enqueues kv_store into it, then commits
 * on its stream (an event is recorded there); a reader acquires with its own
 * stream, which is made to wait for that event, enqueues kv_load, then
 * releases on its stream.  A slot is never handed out again while it is
 * pinned or while the GPU may still be writing or reading it (commit and
 * release events not yet complete): the premature reuse of asynchronous-copy
 * buffers the paper cites is ruled out.  All tier calls are host-thread safe.
 * Pass KVX_NO_STREAM when the caller has already synchronised (no event).
 * Tier calls keep their bookkeeping on the host at call time, so a call given
 * a stream that is being captured into a CUDA graph returns KVX_EINVAL and
 * leaves the capture as it was: a replay would repeat its events and
 * publications without the bookkeeping.
 * ------------------------------------------------------------------------ */
#define KVX_NO_STREAM ((kvx_stream_t)(intptr_t)-1)

typedef struct kvx_tier kvx_tier;

typedef struct {
  int64_t slots, slot_bytes, entries, pinned;
  int64_t hits, misses, evictions;
} kvx_tier_stats;

/*
 * Keys of the chunks of a token sequence: key c depends on the salt, on every
 * token of chunks 0..c and on chunk c's length, so a chunk is found only after
 * the same prefix (KV depends on everything before it).  The salt separates
 * namespaces (Sec. 3.2: a new cache salt forces a cold computation; Sec. 4.4:
 * a reused namespace produced spurious hits).  keys must hold
 * ceil(n_tokens / chunk_tokens) entries.  SplitMix64 finaliser as the mixer.
 */
kvx_status kv_chunk_keys(const int32_t* tokens, int64_t n_tokens, int32_t chunk_tokens, uint64_t salt,
                         uint64_t* keys, int64_t n_keys);

/* A tier over one new exact-size pinned pool (kv_host_alloc) of
   slot_bytes * n_slots; slot_bytes a multiple of 16. */
kvx_status kv_tier_create(int64_t slot_bytes, int64_t n_slots, kvx_tier** out);
/* A tier over caller-owned memory (16-byte aligned, slot_bytes * n_slots
   long), not freed by kv_tier_destroy. */
kvx_status kv_tier_create_on(void* base, int64_t slot_bytes, int64_t n_slots, kvx_tier** out);
/*
 * A tier shared by the processes of one host (Fig. 1: complete replicas, each
 * its own process, share one pinned RAM pool).  `name` is a POSIX shared-memory
 * name ("/..."); with KVX_TIER_CREATE the region (slot table, a process-shared
 * robust mutex, and slot_bytes * n_slots of data) is created, otherwise an
 * existing one is opened and slot_bytes / n_slots are ignored.  Each process
 * registers the region as pinned, mapped memory (cudaHostRegister) unless
 * KVX_TIER_NO_PIN (bookkeeping only, no transfers).  An entry committed on a
 * stream becomes readable by every process as soon as the GPU has completed
 * the work enqueued on that stream before the commit: the commit enqueues a
 * one-thread kernel that publishes it into the shared slot table with a
 * system-scope release store, so no further call of the writer's process is
 * needed.  In the writer's own process the entry is readable at once, the
 * reader's stream waiting on the writer's event.  The creator's
 * kv_tier_destroy removes the name; mappings in other processes stay valid.
 * The shared data is kept on base pages.  Zero-copy runs at the link peak on
 * it (measured on GB300); the copy engines (KVX_MODE_STAGED) moved 192 GB/s
 * to it but only 104 GB/s from it, so use zero-copy with a shared tier.
 */
#define KVX_TIER_CREATE 0x1u
#define KVX_TIER_NO_PIN 0x2u
kvx_status kv_tier_open_shared(const char* name, int64_t slot_bytes, int64_t n_slots, uint32_t flags,
                               kvx_tier** out);
/* Settle this process's completed work on the tier (pins held for its queued
   reads are dropped, its completed commits become READY) and turn every
   published commit of any process READY. */
kvx_status kv_tier_poll(kvx_tier* tier);
/* Waits for this process's pending work on the tier, then frees the tier (and
   its pool if kv_tier_create made it). */
void kv_tier_destroy(kvx_tier* tier);

/* Slot for writing `key` (a free slot, or the least recently used committed
   entry that is neither pinned nor in use by queued GPU work).  Pins it until
   kv_tier_commit (or kv_tier_release to give it up).  KVX_ENOMEM if every
   slot is pinned or busy; KVX_EBUSY if `key` itself is. */
kvx_status kv_tier_reserve(kvx_tier* tier, uint64_t key, void** slot);
/* kv_tier_reserve of keys[0..n) in order, under one lock: slots[j] receives
   the slot of keys[j].  It stops at the first key that cannot be reserved and
   returns that key's status; *n_reserved (may be NULL) receives the number
   reserved, which stay reserved (commit them or release them). */
kvx_status kv_tier_reserve_many(kvx_tier* tier, const uint64_t* keys, int64_t n, void** slots,
                                int64_t* n_reserved);
/* Marks a reserved entry readable once the work already enqueued on
   `stream` (the store into it) completes; unpins it.  On a shared tier the
   commit enqueues its publication (see kv_tier_open_shared): a one-thread
   kernel launch per call. */
kvx_status kv_tier_commit(kvx_tier* tier, uint64_t key, kvx_stream_t stream);
/* kv_tier_commit of n keys on one stream at once: one publication launch per
   512 keys and one event for all of them (a 128k-token context is 512 chunks).
   Every key must be reserved by this process and listed once; otherwise
   KVX_ENOENT / KVX_EINVAL and nothing is committed. */
kvx_status kv_tier_commit_many(kvx_tier* tier, const uint64_t* keys, int64_t n, kvx_stream_t stream);
/* Slot of a committed entry; `stream` is made to wait for its commit event.
   Pins it until kv_tier_release.  KVX_ENOENT if absent or not committed. */
kvx_status kv_tier_acquire(kvx_tier* tier, uint64_t key, kvx_stream_t stream, void** slot);
/* kv_tier_acquire of n keys: slots[j] receives the slot of keys[j] (a key may
   be listed more than once: one pin each).  `stream` waits once per distinct
   commit event.  If any key is not readable (KVX_ENOENT) or cannot be pinned
   (KVX_EBUSY), nothing is pinned. */
kvx_status kv_tier_acquire_many(kvx_tier* tier, const uint64_t* keys, int64_t n, kvx_stream_t stream,
                                void** slots);
/* Unpins; the slot stays in use until the work already enqueued on `stream`
   (the load from it) completes. */
kvx_status kv_tier_release(kvx_tier* tier, uint64_t key, kvx_stream_t stream);
/* kv_tier_release of n keys with one event for all of them.  Each listing of
   a key drops one pin this process holds; if any key lacks the pins
   (KVX_EINVAL) or is absent (KVX_ENOENT), nothing is released. */
kvx_status kv_tier_release_many(kvx_tier* tier, const uint64_t* keys, int64_t n, kvx_stream_t stream);
/* Shared tier: drops the pins held by processes that no longer exist and
   frees the entries they were writing or committing (their bytes may be
   incomplete).  *reclaimed (may be null) receives the number of slots changed.
   kv_tier_reserve does the same by itself when it finds no usable slot.
   Liveness is judged by process id within this host's pid namespace; a
   private tier has nothing to reclaim.  An entry can be pinned by at most 8
   processes at once (KVX_EBUSY beyond).  A process that dies inside a tier
   call, holding the table lock, leaves no entry readable under a wrong key:
   the next call in another process takes the lock over and rebuilds the key
   index from the slot table, and the dead process's slot is reclaimed. */
kvx_status kv_tier_reclaim(kvx_tier* tier, int64_t* reclaimed);
/* Number of leading keys with committed entries (the cached prefix). */
kvx_status kv_tier_prefix_hits(kvx_tier* tier, const uint64_t* keys, int64_t n, int64_t* hits);
/*
 * Waits on the host until all n keys have readable entries -- committed, and
 * for another process's commits published by the GPU -- or until timeout_ns
 * has passed (Fig. 1: a replica restores what another replica stored only once
 * the store is complete).  It checks the keys, then sleeps 20 us, doubling to
 * at most 1 ms, holding the tier's lock only while it checks, so many waiting
 * replicas do not hold up the writers.  KVX_OK when every key is readable;
 * KVX_ETIMEOUT when the limit passed first.  *hits (may be NULL) receives the
 * number of leading keys readable at the last check.  Nothing is pinned: the
 * caller acquires the entries afterwards (an entry can be evicted in between).
 */
kvx_status kv_tier_wait(kvx_tier* tier, const uint64_t* keys, int64_t n, int64_t timeout_ns, int64_t* hits);
kvx_status kv_tier_stats(kvx_tier* tier, kvx_tier_stats* out);

/*
 * Lowest logical block index whose table entry was out of range in any call
 * completed since the last query, or -1.  Call after the caller's stream has
 * been synchronised.  Clears the record.  Returns KVX_ETIMEOUT (and still fills
 * *first_bad_block) if a bounded wait inside a kernel of this context expired
 * since the last query (kvx_opts.wait_cycles); that clears too.
 */
kvx_status kv_get_device_error(kvx_ctx* ctx, int64_t* first_bad_block);

/* Counters of this context; waits for timed launches to finish. */
kvx_status kv_ctx_stats(kvx_ctx* ctx, kvx_stats* out);
kvx_status kv_ctx_reset_stats(kvx_ctx* ctx);

/* The mode a context resolved for each direction (after KVX_MODE_AUTO). */
kvx_status kv_ctx_modes(const kvx_ctx* ctx, int32_t* store_mode, int32_t* load_mode);

/* The last CUDA error code seen by this thread inside the library (0 = none). */
int kv_last_cuda_error(void);

/* Text naming the CUDA call behind the last KVX_ECUDA of this thread ("" if
   none).  The string belongs to the library and stays valid until the
   thread's next failing call. */
const char* kv_last_error_message(void);

/*
 * Host-side fault injection for testing error handling without faulting a
 * GPU: the (after_calls + 1)-th next CUDA call at `point` in this process
 * fails with cudaErrorUnknown (cudaErrorMemoryAllocation for "host_alloc")
 * instead of being made.  Points: "launch" (kernel launches), "memcpy"
 * (staged-mode copies), "event" (the staged pipeline's ordering event
 * recorded on the caller's stream), "host_alloc" (kv_host_alloc).  Two more
 * points fail differently.  "tma_wait": the (after_calls + 1)-th next launch
 * of the TMA engine arms the shared-memory stage of its first unit for bytes
 * that no copy brings, so that unit's bounded wait runs out (after
 * kvx_opts.wait_cycles) with no copy in flight: the launch leaves that unit
 * unmoved and kv_get_device_error returns KVX_ETIMEOUT; nothing faults or
 * hangs.  "tier_exit" ends the process (_exit(3)) inside
 * kv_tier_reserve, while it holds a shared tier's table lock, right after it
 * has taken a slot for the new key; it tests how the processes left recover
 * the tier from a replica that died mid-update.  One point is armed at a
 * time; point NULL or "" disarms.  KVX_EINVAL for an unknown point.
 * The environment variable KVX_FAULT="<point>[:<after_calls>]" arms a point
 * the same way when the library is loaded (a malformed value is reported on
 * stderr and ignored), for programs that do not call this function.
 */
kvx_status kv_fault_inject(const char* point, int32_t after_calls);

/* Static text for a status value. */
const char* kv_status_string(kvx_status status);

int kv_abi_version(void);

#ifdef __cplusplus
}
#endif
#endif /* KVXFER_H */
