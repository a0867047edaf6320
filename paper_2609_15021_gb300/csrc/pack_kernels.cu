// pack_kernels.cu -- gather (pack) and scatter (unpack) kernels between the
// paged KV pool and packed chunks, for sm_103a.
//
// Paper Sec. 3.2: storing a prefix gathers its KV pages into the host tier's
// packed chunk, loading scatters the chunk back into freshly allocated pages.
// This is pure byte movement bound by memory bandwidth (HBM for device chunks
// and staging, the host link for mapped pinned chunks), so it runs on the
// load/store units with 16-byte vectors; no tensor cores are involved.
//
// Work unit: one (chunk, layer, page, K|V) region, handled by one warp.  For
// the shapes of a 27B-class model (B = 16 tokens, H = 8 heads, 256-byte rows)
// a unit is 32 KiB: both its page side and its chunk side are contiguous
// 32 KiB extents, the chunk side in [token][head] row order and the page side
// in [head][token] order (HND) or [token][head] order (NHD).  Every 256-byte
// row is read and written whole by 16 lanes, so each 128-byte line is used in
// full on both sides.  Each lane keeps kInflight 16-byte loads in flight
// before storing them.
//
// Out-of-range block-table entries skip their unit and lower a device error
// word (atomicMin of the logical block index); nothing traps.

#include "copy16.cuh"
#include "kvx_internal.h"

namespace kvx {
namespace {

// HND page side [H][B][R] <-> chunk side [nb][H][R], nr = nb * H rows, when
// R / 16 is a power of two no larger than 32: a warp covers 32 / (R/16) whole
// rows per step, each lane a fixed 16-byte column, and the (token, head) pair
// of a lane's row is advanced incrementally (no division in the loop).
template <int DIR>
__device__ __forceinline__ void move_hnd_fast(uint8_t* pg, uint8_t* ck, int nr, const MoveParams& p,
                                              int lane) {
  const int rows_per_step = 32 >> p.vpr_shift;
  const int64_t col = (int64_t)(lane & ((1 << p.vpr_shift) - 1)) * 16;
  const int64_t R = p.R, B = p.B;
  const int H = p.H;
  int r = lane >> p.vpr_shift;  // row in chunk order: r = s * H + h
  int s = r / H;
  int h = r - s * H;
  while (r + (kInflight - 1) * rows_per_step < nr) {
    int64_t po[kInflight], co[kInflight];
#pragma unroll
    for (int i = 0; i < kInflight; ++i) {
      po[i] = ((int64_t)h * B + s) * R + col;
      co[i] = (int64_t)r * R + col;
      r += rows_per_step;
      s += p.rpi_div_h;
      h += p.rpi_mod_h;
      if (h >= H) {
        h -= H;
        ++s;
      }
    }
    move_batch<DIR>(pg, ck, po, co);
  }
  while (r < nr) {
    move_one<DIR>(pg, ck, ((int64_t)h * B + s) * R + col, (int64_t)r * R + col);
    r += rows_per_step;
    s += p.rpi_div_h;
    h += p.rpi_mod_h;
    if (h >= H) {
      h -= H;
      ++s;
    }
  }
}

// HND for any row size that is a multiple of 16 bytes.
template <int DIR>
__device__ __forceinline__ void move_hnd_generic(uint8_t* pg, uint8_t* ck, int nr, const MoveParams& p,
                                                 int lane) {
  const int vpr = p.R / 16;
  const int64_t nv = (int64_t)nr * vpr;
  for (int64_t v = lane; v < nv; v += 32) {
    const int64_t r = v / vpr;
    const int64_t c = (v - r * vpr) * 16;
    const int64_t s = r / p.H;
    const int64_t h = r - s * p.H;
    move_one<DIR>(pg, ck, (h * p.B + s) * p.R + c, r * p.R + c);
  }
}

// At most 64 registers (4 CTAs of 256 threads per SM); no variant spills.
template <int DIR, int LAYOUT>
__global__ void __launch_bounds__(kThreads, 4) move_kernel(const __grid_constant__ MoveParams p) {
  const int lane = threadIdx.x & 31;
  const int64_t nwarps = ((int64_t)gridDim.x * kThreads) >> 5;
  int64_t u = ((int64_t)blockIdx.x * kThreads + threadIdx.x) >> 5;
  int j = 0;
  int64_t job_begin = 0;
  const int64_t half_page = p.page_bytes >> 1;  // K or V part of a page: H * B * R
  const int64_t HR = (int64_t)p.H * p.R;
  for (; u < p.total_units; u += nwarps) {
    while (u >= p.jobs[j].unit_end) {  // warp-uniform; units ascend per warp
      job_begin = p.jobs[j].unit_end;
      ++j;
    }
    const Job& J = p.jobs[j];
    const int64_t local = u - job_begin;
    const int kv = (int)(local & 1);
    const int64_t rest = local >> 1;
    const int jb = (int)(rest % p.blocks_per_chunk);
    const int l = J.l0 + (int)(rest / p.blocks_per_chunk);
    const int tok0 = jb * p.B;
    if (tok0 >= J.tokens) continue;  // past the end of a short last chunk
    const int nb = min(p.B, J.tokens - tok0);
    // kernel page of the unit, the logical block naming it, and the pool page
    const int64_t kpage = J.first_block + jb;
    const int64_t lblk = kpage / p.ppb;
    const int32_t entry = __ldg(p.table + lblk);
    const int64_t page = (int64_t)entry * p.ppb + (kpage - lblk * p.ppb);
    uint8_t* ck = J.chunk + ((int64_t)(l - J.l0) * 2 + kv) * J.tokens * HR + (int64_t)tok0 * HR;
    const int nr = nb * p.H;
    if (entry < 0 || (int64_t)entry >= p.num_blocks / p.ppb) {
      if (lane == 0) atomicMin(p.err, (long long)lblk);
      if (DIR == kPack) {  // the unit's chunk rows (contiguous) read as zeros
        const uint4 z = make_uint4(0, 0, 0, 0);
        for (int64_t off = (int64_t)lane * 16; off < (int64_t)nr * p.R; off += 32 * 16) st16(ck + off, z);
      }
      continue;
    }
    uint8_t* pg = p.layer_base[l] + (int64_t)page * p.page_bytes + kv * half_page;
    if (LAYOUT == KVX_LAYOUT_NHD)
      move_flat<DIR>(pg, ck, (int64_t)nr * p.R, lane);
    else if (p.fast)
      move_hnd_fast<DIR>(pg, ck, nr, p, lane);
    else
      move_hnd_generic<DIR>(pg, ck, nr, p, lane);
  }
}

template <int DIR, int LAYOUT>
int occupancy_of() {
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, move_kernel<DIR, LAYOUT>, kThreads, 0) !=
      cudaSuccess) {
    cudaGetLastError();
    return 1;
  }
  return n > 0 ? n : 1;
}

}  // namespace

cudaError_t launch_move(int dir, int layout, const MoveParams& p, int grid, cudaStream_t s) {
  if (dir == kPack && layout == KVX_LAYOUT_HND)
    move_kernel<kPack, KVX_LAYOUT_HND><<<grid, kThreads, 0, s>>>(p);
  else if (dir == kPack)
    move_kernel<kPack, KVX_LAYOUT_NHD><<<grid, kThreads, 0, s>>>(p);
  else if (layout == KVX_LAYOUT_HND)
    move_kernel<kUnpack, KVX_LAYOUT_HND><<<grid, kThreads, 0, s>>>(p);
  else
    move_kernel<kUnpack, KVX_LAYOUT_NHD><<<grid, kThreads, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t load_pack_kernels() {
  // cudaFuncGetAttributes makes CUDA load a kernel that lazy loading has not loaded yet
  cudaFuncAttributes a;
  cudaError_t e = cudaFuncGetAttributes(&a, move_kernel<kPack, KVX_LAYOUT_HND>);
  if (e == cudaSuccess) e = cudaFuncGetAttributes(&a, move_kernel<kPack, KVX_LAYOUT_NHD>);
  return e;
}

int move_ctas_per_sm(int dir, int layout) {
  if (dir == kPack) return layout == KVX_LAYOUT_HND ? occupancy_of<kPack, KVX_LAYOUT_HND>()
                                                    : occupancy_of<kPack, KVX_LAYOUT_NHD>();
  return layout == KVX_LAYOUT_HND ? occupancy_of<kUnpack, KVX_LAYOUT_HND>()
                                  : occupancy_of<kUnpack, KVX_LAYOUT_NHD>();
}

}  // namespace kvx
