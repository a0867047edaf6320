// probe.cu -- the paper's copy-ordering byte probes (Sec. 3.2, Table 2).
//
// A kernel on the caller's stream waits a fixed number of SM cycles and then
// writes (or reads) a buffer; a host<->device copy is issued with or without
// a dependency on that stream.  The delay is a clock64() loop capped at
// KVX_PROBE_MAX_CYCLES; it waits on nothing else.

#include <cuda_runtime.h>

#include <mutex>

#include "kvx_internal.h"
#include "kvxfer_probe.h"

namespace {

constexpr int kProbeThreads = 256;

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
  if (e != cudaSuccess) {
    kvx::set_last_cuda_error((int)e);
    return KVX_ECUDA;
  }
  return KVX_OK;
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
  if (e != cudaSuccess) {
    kvx::set_last_cuda_error((int)e);
    return KVX_ECUDA;
  }
  return KVX_OK;
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
  if (e != cudaSuccess) {
    kvx::set_last_cuda_error((int)e);
    cudaGetLastError();
    return KVX_ECUDA;
  }
  return KVX_OK;
}
