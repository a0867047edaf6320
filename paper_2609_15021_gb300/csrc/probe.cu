// probe.cu -- libkvxfer_probe.so: measuring instruments for the tests and the
// benchmark, kept out of the transfer library.
//
// * The paper's copy-ordering byte probes (Sec. 3.2, Table 2): a kernel on the
//   caller's stream waits a fixed number of SM cycles and then writes (or
//   reads) a buffer; a host<->device copy is issued with or without a
//   dependency on that stream.  The delay is a clock64() loop capped at
//   KVX_PROBE_MAX_CYCLES; it waits on nothing else.
// * A contiguous streaming copy on the SMs, used between device memory and
//   mapped pinned host memory to measure what the SMs alone can move over the
//   host link (the ceiling of the zero-copy transfers, beside the copy
//   engines' pinned cudaMemcpyAsync peak).
//
// This library shares no code with libkvxfer.so; it includes only the public
// header for kvx_status and kvx_stream_t.

#include <cuda_runtime.h>

#include <mutex>

#include "kvxfer_probe.h"

namespace {

constexpr int kProbeThreads = 256;
constexpr int kStreamInflight = 8;  // 16-byte vectors per thread between loads and stores

thread_local int g_probe_cuda_error = 0;

kvx_status cuda_failed(cudaError_t e) {
  g_probe_cuda_error = (int)e;
  cudaGetLastError();
  return KVX_ECUDA;
}

__device__ __forceinline__ void spin_cycles(long long cycles) {
  if (cycles <= 0) return;
  if (threadIdx.x == 0) {
    const long long t0 = clock64();
    while (clock64() - t0 < cycles) __nanosleep(200);
  }
  __syncthreads();
}

__global__ void delayed_fill_kernel(uint8_t* dev, long long bytes, uint8_t value, long long cycles) {
  spin_cycles(cycles);
  const long long stride = (long long)gridDim.x * blockDim.x;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < bytes; i += stride)
    dev[i] = value;
}

__global__ void delayed_copy_kernel(uint4* dst, const uint4* src, long long n16, long long cycles) {
  spin_cycles(cycles);
  const long long stride = (long long)gridDim.x * blockDim.x;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n16; i += stride)
    dst[i] = src[i];
}

// dst[i] = src[i] for n16 16-byte vectors: each thread keeps kStreamInflight
// vectors in flight, and a warp's lanes cover 512 contiguous bytes per vector
// step, so every 128-byte line is read and written whole.  Streaming
// (evict-first) accesses: every byte is touched once.
__global__ void stream_copy_kernel(uint4* dst, const uint4* src, long long n16) {
  const long long nthreads = (long long)gridDim.x * blockDim.x;
  long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  for (; i + (kStreamInflight - 1) * nthreads < n16; i += kStreamInflight * nthreads) {
    uint4 v[kStreamInflight];
#pragma unroll
    for (int k = 0; k < kStreamInflight; ++k) v[k] = __ldcs(src + i + k * nthreads);
#pragma unroll
    for (int k = 0; k < kStreamInflight; ++k) __stcs(dst + i + k * nthreads, v[k]);
  }
  for (; i < n16; i += nthreads) __stcs(dst + i, __ldcs(src + i));
}

// The probe kernels use no shared memory, but an SM's shared-memory carveout
// is set for the kernels resident on it: asking for the largest carveout lets
// kernels that need shared memory (the TMA engine) start beside a spinning
// probe, so an unordered transfer really runs before the probe finishes.
void prefer_max_shared_carveout() {
  static std::once_flag once;
  std::call_once(once, [] {
    cudaFuncSetAttribute(delayed_fill_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                         cudaSharedmemCarveoutMaxShared);
    cudaFuncSetAttribute(delayed_copy_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                         cudaSharedmemCarveoutMaxShared);
    cudaGetLastError();
  });
}

// One CTA per SM keeps every CTA resident, so the whole grid waits about
// `cycles` once rather than once per wave.
int resident_grid() {
  int dev = 0, sms = 1;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    return 1;
  }
  return sms > 0 ? sms : 1;
}

long long clamp_cycles(int64_t c) {
  if (c < 0) return 0;
  return c > KVX_PROBE_MAX_CYCLES ? KVX_PROBE_MAX_CYCLES : (long long)c;
}

// The address a kernel uses for p: p itself for device memory, the mapped
// device address for page-locked host memory; null for anything else.
void* kernel_address(void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) return p;
  if (a.type == cudaMemoryTypeHost) return a.devicePointer;
  return nullptr;
}

kvx_status device_ptr_ok(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return KVX_EDEVICE;
  }
  return a.type == cudaMemoryTypeDevice ? KVX_OK : KVX_EDEVICE;
}

}  // namespace

extern "C" kvx_status kvx_probe_delayed_fill(void* dev, int64_t bytes, int32_t value, int64_t cycles,
                                             kvx_stream_t stream) {
  if (!dev || bytes <= 0 || value < 0 || value > 255) return KVX_EINVAL;
  kvx_status st = device_ptr_ok(dev);
  if (st != KVX_OK) return st;
  prefer_max_shared_carveout();
  delayed_fill_kernel<<<resident_grid(), kProbeThreads, 0, (cudaStream_t)stream>>>(
      (uint8_t*)dev, bytes, (uint8_t)value, clamp_cycles(cycles));
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? KVX_OK : cuda_failed(e);
}

extern "C" kvx_status kvx_probe_delayed_copy(void* dst, const void* src, int64_t bytes, int64_t cycles,
                                             kvx_stream_t stream) {
  if (!dst || !src || bytes <= 0) return KVX_EINVAL;
  if (((uintptr_t)dst | (uintptr_t)src | (uintptr_t)bytes) & 15) return KVX_EALIGN;
  kvx_status st = device_ptr_ok(dst);
  if (st == KVX_OK) st = device_ptr_ok(src);
  if (st != KVX_OK) return st;
  prefer_max_shared_carveout();
  delayed_copy_kernel<<<resident_grid(), kProbeThreads, 0, (cudaStream_t)stream>>>(
      (uint4*)dst, (const uint4*)src, bytes / 16, clamp_cycles(cycles));
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? KVX_OK : cuda_failed(e);
}

extern "C" kvx_status kvx_probe_copy(void* dst, const void* src, int64_t bytes, int32_t how,
                                     kvx_stream_t stream) {
  if (!dst || !src || bytes <= 0) return KVX_EINVAL;
  cudaError_t e = cudaSuccess;
  switch (how) {
    case KVX_PROBE_RAW:  // the paper's fallback: no stream argument at all
      e = cudaMemcpy(dst, src, (size_t)bytes, cudaMemcpyDefault);
      break;
    case KVX_PROBE_WAIT_THEN_COPY:
      e = cudaStreamSynchronize((cudaStream_t)stream);
      if (e == cudaSuccess) e = cudaMemcpy(dst, src, (size_t)bytes, cudaMemcpyDefault);
      break;
    case KVX_PROBE_ASYNC_ON_STREAM:
      e = cudaMemcpyAsync(dst, src, (size_t)bytes, cudaMemcpyDefault, (cudaStream_t)stream);
      break;
    default:
      return KVX_EINVAL;
  }
  return e == cudaSuccess ? KVX_OK : cuda_failed(e);
}

extern "C" kvx_status kvx_probe_stream_copy(void* dst, const void* src, int64_t bytes, int32_t ctas,
                                            kvx_stream_t stream) {
  if (!dst || !src || bytes <= 0 || ctas < 1) return KVX_EINVAL;
  if (((uintptr_t)dst | (uintptr_t)src | (uintptr_t)bytes) & 15) return KVX_EALIGN;
  void* d = kernel_address(dst);
  void* s = kernel_address(const_cast<void*>(src));
  if (!d || !s) return KVX_ENOTPINNED;
  // both ends must be mapped over their whole length at one offset
  void* d_last = kernel_address((uint8_t*)dst + bytes - 1);
  void* s_last = kernel_address((uint8_t*)const_cast<void*>(src) + bytes - 1);
  if (d_last != (uint8_t*)d + bytes - 1 || s_last != (uint8_t*)s + bytes - 1) return KVX_ENOTPINNED;
  stream_copy_kernel<<<ctas, kProbeThreads, 0, (cudaStream_t)stream>>>((uint4*)d, (const uint4*)s, bytes / 16);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? KVX_OK : cuda_failed(e);
}

extern "C" int kvx_probe_last_cuda_error(void) { return g_probe_cuda_error; }
