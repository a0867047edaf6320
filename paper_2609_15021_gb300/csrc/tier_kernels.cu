// tier_kernels.cu -- the one kernel of the shared host tier: publication of a
// commit.
//
// Paper Sec. 3.2: a chunk may be consumed only after the copy that produced it
// has completed.  A commit on a stream enqueues this single-thread kernel
// behind the store: it writes the commit's sequence number into the slot
// table, which lives in host memory shared by every process of the tier and
// mapped for the GPU.  The store is a release at system scope, so every byte
// the stream wrote before it (the chunk, written by earlier kernels or copies
// in stream order) is visible to any CPU or GPU that observes the number with
// an acquire load.  Other processes then treat the entry as complete without
// the writer's process having to notice its own GPU work finish.

#include "kvx_internal.h"

namespace kvx {
namespace {

// Thread j publishes commit seq0 + j of slot slot[j]: its flag lies at
// meta + slot[j] * stride + offset.
__global__ void tier_publish_kernel(TierPublish b) {
  const int j = threadIdx.x;
  if (j >= b.n) return;
  unsigned long long* flag = reinterpret_cast<unsigned long long*>(b.meta + (int64_t)b.slot[j] * b.stride + b.offset);
  const unsigned long long seq = b.seq0 + (unsigned long long)j;
  asm volatile("st.release.sys.global.u64 [%0], %1;" ::"l"(flag), "l"(seq) : "memory");
}

}  // namespace

// Loads the kernel's module now.  Left to its first launch, the lazy load
// happened inside a commit and waited for the work already on the GPU.
cudaError_t prepare_tier_kernels() {
  cudaFuncAttributes a;
  return cudaFuncGetAttributes(&a, tier_publish_kernel);
}

cudaError_t launch_tier_publish(const TierPublish& b, cudaStream_t s) {
  if (b.n < 1 || b.n > kMaxPublish) return cudaErrorInvalidValue;
  tier_publish_kernel<<<1, b.n, 0, s>>>(b);
  return cudaGetLastError();
}

}  // namespace kvx
