/*
 * kvxfer_probe.h -- measuring instruments in libkvxfer_probe.so, a library of
 * its own that the tests and the benchmark load beside libkvxfer.so.  It
 * shares no code with the transfer library.
 *
 * Ordering probes.
 * These reproduce the paper's controlled byte experiment (Sec. 3.2; Table 2,
 * "Copy-ordering controls"): a kernel on a non-default stream writes (or
 * reads) a buffer after an imposed delay of the order of 10^8 SM cycles, and
 * a host<->device copy is issued either without a dependency on that stream
 * (the raw fallback: a synchronous cudaMemcpy with cudaMemcpyDefault and no
 * stream argument) or with one of the ordered mechanisms the paper lists
 * (wait for the stream before the same copy; cudaMemcpyAsync on the stream).
 * Unordered + delay must observe stale bytes; ordered must observe final ones.
 *
 * The delay is a clock64() spin bounded by KVX_PROBE_MAX_CYCLES; nothing here
 * waits on a flag or on another kernel.
 */
#ifndef KVXFER_PROBE_H
#define KVXFER_PROBE_H

#include <stdint.h>
#include "kvxfer.h"

#ifdef __cplusplus
extern "C" {
#endif

#define KVX_PROBE_MAX_CYCLES 4000000000LL /* about 2 s at the maximum SM clock */

typedef enum {
  KVX_PROBE_RAW = 0,             /* cudaMemcpy(dst, src, n, cudaMemcpyDefault): no stream */
  KVX_PROBE_WAIT_THEN_COPY = 1,  /* cudaStreamSynchronize(stream), then the same copy     */
  KVX_PROBE_ASYNC_ON_STREAM = 2  /* cudaMemcpyAsync(..., stream)                           */
} kvx_probe_how;

/*
 * On `stream`: spin `cycles` SM cycles (clamped to [0, KVX_PROBE_MAX_CYCLES]),
 * then fill dev[0 .. bytes) with `value`.  dev: device memory.
 */
kvx_status kvx_probe_delayed_fill(void* dev, int64_t bytes, int32_t value, int64_t cycles,
                                  kvx_stream_t stream);

/*
 * On `stream`: spin `cycles` SM cycles, then copy bytes from src to dst
 * (device memory, 16-byte aligned, bytes % 16 == 0).  Used both as a delayed
 * producer (final KV written just before kv_store) and as a delayed consumer
 * (reading a buffer that a copy is about to overwrite).
 */
kvx_status kvx_probe_delayed_copy(void* dst, const void* src, int64_t bytes, int64_t cycles,
                                  kvx_stream_t stream);

/*
 * Copy `bytes` between pinned host memory and device memory with ordering
 * mechanism `how` relative to `stream`.  KVX_PROBE_RAW is the paper's faulty
 * fallback and is kept as a negative control only.
 */
kvx_status kvx_probe_copy(void* dst, const void* src, int64_t bytes, int32_t how, kvx_stream_t stream);

/*
 * Host-link probe: on `stream`, copy `bytes` from src to dst with a plain
 * contiguous streaming kernel on the SMs (16-byte loads and stores, whole
 * 128-byte lines, `ctas` CTAs of 256 threads striding over the range).  Either
 * side may be device memory or page-locked host memory mapped for the GPU, so
 * device -> mapped host measures what SM stores can push over the host link
 * and mapped host -> device what SM loads can pull: the ceiling of zero-copy
 * transfers, beside the copy engines' cudaMemcpyAsync.  Both pointers and
 * `bytes` must be multiples of 16 (KVX_EALIGN); a side that is neither device
 * memory nor mapped over its whole length is KVX_ENOTPINNED.
 */
kvx_status kvx_probe_stream_copy(void* dst, const void* src, int64_t bytes, int32_t ctas, kvx_stream_t stream);

/* The last CUDA error code a probe call of this thread saw (0 = none). */
int kvx_probe_last_cuda_error(void);

#ifdef __cplusplus
}
#endif
#endif /* KVXFER_PROBE_H */
