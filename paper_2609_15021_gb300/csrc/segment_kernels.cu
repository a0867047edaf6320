// segment_kernels.cu -- opaque byte copies (recurrent-state snapshots, paper
// Sec. 2.2: a hybrid model's linear-attention layers keep a fixed-size state
// that is saved and restored whole at aligned boundaries), between state
// slots in HBM and a host object in mapped pinned memory.

#include "copy16.cuh"
#include "kvx_internal.h"

namespace kvx {
namespace {

// Opaque byte segments (recurrent-state slots): warp units of p.unit_bytes
// over the concatenated segments; a unit that crosses a segment end continues
// in the next segment.  Every piece is a multiple of 16 bytes.
__global__ void __launch_bounds__(kThreads) segment_kernel(const __grid_constant__ SegmentParams p) {
  const int lane = threadIdx.x & 31;
  const int64_t nwarps = ((int64_t)gridDim.x * kThreads) >> 5;
  int64_t u = ((int64_t)blockIdx.x * kThreads + threadIdx.x) >> 5;
  int j = 0;
  int64_t seg_begin = 0;
  for (; u < p.total_units; u += nwarps) {
    int64_t b = u * p.unit_bytes;
    const int64_t b_end = min(b + p.unit_bytes, p.total_bytes);
    while (b >= p.seg[j].byte_end) {  // warp-uniform; units ascend per warp
      seg_begin = p.seg[j].byte_end;
      ++j;
    }
    while (b < b_end) {
      const Segment& S = p.seg[j];
      const int64_t n = min(b_end, S.byte_end) - b;
      move_flat<kPack>(const_cast<uint8_t*>(S.src) + (b - seg_begin), S.dst + (b - seg_begin), n, lane);
      b += n;
      if (b >= S.byte_end && b < b_end) {
        seg_begin = S.byte_end;
        ++j;
      }
    }
  }
}

}  // namespace

cudaError_t launch_segments(const SegmentParams& p, int grid, cudaStream_t s) {
  segment_kernel<<<grid, kThreads, 0, s>>>(p);
  return cudaGetLastError();
}

int segment_ctas_per_sm() {
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, segment_kernel, kThreads, 0) != cudaSuccess) {
    cudaGetLastError();
    return 1;
  }
  return n > 0 ? n : 1;
}

}  // namespace kvx
