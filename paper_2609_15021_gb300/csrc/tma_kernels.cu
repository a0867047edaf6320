// tma_kernels.cu -- device-side pack / unpack with the Tensor Memory
// Accelerator (TMA), staged through shared memory.
//
// Same work units and byte mapping as move_kernel (pack_kernels.cu): one
// (chunk, layer, page, K|V) unit at a time, here per CTA of one warp.  A unit
// is copied global -> shared with completion on an mbarrier, then shared ->
// global tracked as a bulk group; registers never hold the data.  By default
// every unit gets its own CTA with a single stage (six 32 KiB CTAs fit an SM,
// and the block scheduler keeps DRAM busy as CTAs finish); a grid capped by
// the caller strides each CTA over many units through a ring of stages, so
// the loads of the next units overlap the store of the current one.
//
// Two ways to move the page side of an HND unit (its [head][token][row]
// bytes, which the chunk holds in [token][head][row] order):
//  * tensor maps (TMAP): each pool layer is described to the TMA unit as a
//    5-D tensor (row bytes, head, token, K|V, page) whose head and token
//    dimensions carry each other's strides, so one box copy of a whole page
//    half lands in -- or leaves from -- shared memory already in chunk order;
//  * row copies: one 1-D bulk copy per (head, token) row.
// The chunk side is always one contiguous bulk copy.  Units that cover only
// part of a page (the end of a range) use row copies, so no byte past the
// range is read into a chunk or written to a page.
//
// Only for chunks in device memory (kv_pack / kv_unpack / staged mode).  Every
// mbarrier wait is bounded by a clock limit passed to the kernel.  When a wait
// expires the CTA issues no further load; it waits again, under the same
// limit, on every stage whose load it has issued and not yet consumed (so no
// global -> shared copy it started can still be landing in its shared memory
// when it leaves), waits for its bulk stores, sets the timeout flag and
// returns.  A CTA therefore leaves a load behind only if that load has not
// completed within twice the limit.

#include <cuda.h>
#include <string.h>

#include "kvx_internal.h"

namespace kvx {
namespace {

constexpr int kStagesMax = 4;

struct TensorMaps {
  CUtensorMap m[KVX_MAX_LAYERS];
};
static_assert(sizeof(CUtensorMap) == kTensorMapBytes, "tensor map size");

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(done)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return done != 0;
}
// Bounded wait on an mbarrier phase; false when `limit` SM cycles expired.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, long long limit) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity))
    if (clock64() - t0 > limit) return false;
  return true;
}
__device__ __forceinline__ void bulk_load(void* sdst, const void* gsrc, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_addr(sdst)),
               "l"(gsrc), "r"(bytes), "r"(smem_addr(bar))
               : "memory");
}
__device__ __forceinline__ void bulk_store(void* gdst, const void* ssrc, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(gdst), "r"(smem_addr(ssrc)),
               "r"(bytes)
               : "memory");
}
// One box of a 5-D tensor map at (0, 0, 0, kv, page): a whole K or V page half.
__device__ __forceinline__ void box_load(void* sdst, const CUtensorMap* map, int kv, int page, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.5d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5, "
      "%6}], [%7];" ::"r"(smem_addr(sdst)),
      "l"(map), "r"(0), "r"(0), "r"(0), "r"(kv), "r"(page), "r"(smem_addr(bar))
      : "memory");
}
__device__ __forceinline__ void box_store(const CUtensorMap* map, int kv, int page, const void* ssrc) {
  asm volatile("cp.async.bulk.tensor.5d.global.shared::cta.tile.bulk_group [%0, {%1, %2, %3, %4, %5}], [%6];" ::"l"(
                   map),
               "r"(0), "r"(0), "r"(0), "r"(kv), "r"(page), "r"(smem_addr(ssrc))
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read_0() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read_1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// One unit resolved to addresses.
struct Unit {
  uint8_t* pg;   // page side (K or V half of the page)
  uint8_t* ck;   // chunk side
  int nr;        // rows (tokens x heads)
  int move;      // 0: nothing to move (past a short chunk's end, or a bad page)
  int full;      // the unit covers the whole page half (all B tokens)
  int layer, kv;
  int page;
};

// Same decode as move_kernel; a bad table entry zero-fills the chunk rows
// (pack) with ordinary stores and reports the logical block.  lane < 0: a
// second decode of the same unit (store side), which repeats no side effect.
template <int DIR>
__device__ __forceinline__ Unit decode(const MoveParams& p, int64_t u, int& j, int64_t& job_begin, int lane) {
  Unit r{nullptr, nullptr, 0, 0, 0, 0, 0, 0};
  while (u >= p.jobs[j].unit_end) {
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
  if (tok0 >= J.tokens) return r;
  const int nb = min(p.B, J.tokens - tok0);
  const int64_t HR = (int64_t)p.H * p.R;
  const int64_t kpage = J.first_block + jb;
  const int64_t lblk = kpage / p.ppb;
  const int32_t entry = __ldg(p.table + lblk);
  const int64_t page = (int64_t)entry * p.ppb + (kpage - lblk * p.ppb);
  r.ck = J.chunk + ((int64_t)(l - J.l0) * 2 + kv) * J.tokens * HR + (int64_t)tok0 * HR;
  r.nr = nb * p.H;
  if (entry < 0 || (int64_t)entry >= p.num_blocks / p.ppb) {
    if (lane == 0) atomicMin(p.err, (long long)lblk);
    if (DIR == kPack && lane >= 0) {
      const uint4 z = make_uint4(0, 0, 0, 0);
      for (int64_t off = (int64_t)lane * 16; off < (int64_t)r.nr * p.R; off += 32 * 16)
        *reinterpret_cast<uint4*>(r.ck + off) = z;
    }
    return r;
  }
  r.pg = p.layer_base[l] + page * p.page_bytes + kv * (p.page_bytes >> 1);
  r.move = 1;
  r.full = nb == p.B;
  r.layer = l;
  r.kv = kv;
  r.page = (int)page;
  return r;
}

// Issue the global -> shared copies of one unit into `stage`.  stall: arm the
// stage's phase for bytes that no copy will bring (the host-side fault point
// "tma_wait"), so that the wait on it runs out with nothing in flight.
template <int DIR, int LAYOUT, bool TMAP>
__device__ __forceinline__ void issue_loads(const MoveParams& p, const TensorMaps* maps, const Unit& w,
                                            uint8_t* stage, uint64_t* bar, int lane, bool stall) {
  const uint32_t bytes = w.move ? (uint32_t)((TMAP && DIR == kPack && w.full ? p.B * p.H : w.nr) * p.R) : 0u;
  if (lane == 0) mbar_expect_tx(bar, stall ? max(bytes, 16u) : bytes);
  __syncwarp();
  if (!w.move || stall) return;
  if (DIR == kUnpack || LAYOUT == KVX_LAYOUT_NHD) {
    // chunk side (unpack) or an NHD page (pack): one contiguous run
    if (lane == 0) bulk_load(stage, DIR == kUnpack ? w.ck : w.pg, bytes, bar);
  } else if (TMAP && w.full) {
    if (lane == 0) box_load(stage, &maps->m[w.layer], w.kv, w.page, bar);
  } else {
    // HND page rows (h, s) land at the chunk's row r = s * H + h
    for (int r = lane; r < w.nr; r += 32) {
      const int s = r / p.H, h = r - s * p.H;
      bulk_load(stage + (int64_t)r * p.R, w.pg + ((int64_t)h * p.B + s) * p.R, (uint32_t)p.R, bar);
    }
  }
}

// Issue the shared -> global copies of one unit from `stage`.
template <int DIR, int LAYOUT, bool TMAP>
__device__ __forceinline__ void issue_stores(const MoveParams& p, const TensorMaps* maps, const Unit& w,
                                             const uint8_t* stage, int lane) {
  if (w.move) {
    const uint32_t bytes = (uint32_t)(w.nr * p.R);
    if (DIR == kPack || LAYOUT == KVX_LAYOUT_NHD) {
      if (lane == 0) bulk_store(DIR == kPack ? w.ck : w.pg, stage, bytes);
    } else if (TMAP && w.full) {
      if (lane == 0) box_store(&maps->m[w.layer], w.kv, w.page, stage);
    } else {
      for (int r = lane; r < w.nr; r += 32) {
        const int s = r / p.H, h = r - s * p.H;
        bulk_store(w.pg + ((int64_t)h * p.B + s) * p.R, stage + (int64_t)r * p.R, (uint32_t)p.R);
      }
    }
  }
  bulk_commit();
}

template <int DIR, int LAYOUT, bool TMAP>
__device__ __forceinline__ void tma_move_body(const MoveParams& p, const TensorMaps* maps, int stage_bytes,
                                              int stages, const TmaWait& wt) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t bars[kStagesMax];
  // 128-byte aligned stages (tensor copies need it)
  uint8_t* smem = smem_raw + ((128 - (smem_addr(smem_raw) & 127)) & 127);
  const int lane = threadIdx.x;
  if (lane == 0) {
    for (int k = 0; k < stages; ++k) mbar_init(&bars[k], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncwarp();
  const int64_t first = blockIdx.x, step = gridDim.x;
  const int64_t n = p.total_units > first ? (p.total_units - first + step - 1) / step : 0;
  int jl = 0, js = 0;  // decode cursors: loads run ahead of stores
  int64_t bl = 0, bs = 0;
  // Loads run `ahead` units ahead of stores: stages - 1 with a ring, and one
  // with a single stage (the next unit's load then waits for the store to
  // have read the stage).  Units [consumed, issued) have a load armed on
  // stage (unit % stages); at most one per stage.
  const int ahead = stages > 1 ? stages - 1 : 1;
  const int64_t pro = n < ahead ? n : ahead;
  for (int64_t it = 0; it < pro; ++it) {
    const int64_t u = first + it * step;
    const Unit w = decode<DIR>(p, u, jl, bl, lane);
    issue_loads<DIR, LAYOUT, TMAP>(p, maps, w, smem + it * stage_bytes, &bars[it], lane, u == wt.stall_unit);
  }
  int64_t issued = pro, failed_at = -1;
  for (int64_t it = 0; it < n; ++it) {
    const int k = (int)(it % stages);
    const Unit w = decode<DIR>(p, first + it * step, js, bs, -1);
    bool ok = true;
    if (lane == 0) ok = mbar_wait(&bars[k], (uint32_t)((it / stages) & 1), wt.cycles);
    ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
    if (!ok) {
      failed_at = it;
      break;
    }
    issue_stores<DIR, LAYOUT, TMAP>(p, maps, w, smem + (int64_t)k * stage_bytes, lane);
    const int64_t nxt = it + ahead;
    if (nxt < n) {
      // the store last issued from the next load's stage has read it: one turn
      // ago with a ring, just now with a single stage
      if (stages > 1)
        bulk_wait_read_1();
      else
        bulk_wait_read_0();
      __syncwarp();
      const int kn = (int)(nxt % stages);
      const int64_t un = first + nxt * step;
      const Unit wn = decode<DIR>(p, un, jl, bl, lane);
      issue_loads<DIR, LAYOUT, TMAP>(p, maps, wn, smem + (int64_t)kn * stage_bytes, &bars[kn], lane,
                                     un == wt.stall_unit);
      issued = nxt + 1;
    }
  }
  if (failed_at >= 0) {
    // No new loads; every load still armed gets another bounded wait, so that
    // none lands in this CTA's shared memory after it has left.
    if (lane == 0) {
      for (int64_t v = failed_at; v < issued; ++v)
        mbar_wait(&bars[v % stages], (uint32_t)((v / stages) & 1), wt.cycles);
      atomicExch(wt.timeout, 1);
    }
    __syncwarp();
  }
  bulk_wait_all();
}

template <int DIR, int LAYOUT>
__global__ void __launch_bounds__(32) tma_move_kernel(const __grid_constant__ MoveParams p, int stage_bytes,
                                                      int stages, const TmaWait wt) {
  tma_move_body<DIR, LAYOUT, false>(p, nullptr, stage_bytes, stages, wt);
}

template <int DIR>
__global__ void __launch_bounds__(32) tmap_move_kernel(const __grid_constant__ MoveParams p,
                                                       const __grid_constant__ TensorMaps maps, int stage_bytes,
                                                       int stages, const TmaWait wt) {
  tma_move_body<DIR, KVX_LAYOUT_HND, true>(p, &maps, stage_bytes, stages, wt);
}

// Largest dynamic shared memory a TMA launch uses: 96 KiB of stages (three of
// at most 32 KiB or two of at most 48 KiB) plus 128 bytes of alignment slack.
constexpr int kTmaSmemMax = (96 << 10) + 128;

template <typename K>
cudaError_t set_smem(K kernel) {
  return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kTmaSmemMax);
}

using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                              const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                              CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeFn encoder() {
  static EncodeFn fn = [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess) {
      cudaGetLastError();
      f = nullptr;
    }
    return (EncodeFn)f;
  }();
  return fn;
}

}  // namespace

bool encode_tensor_maps(const kvx_pool* P, int64_t row_bytes, void* out) {
  if (P->layout != KVX_LAYOUT_HND) return false;
  EncodeFn enc = encoder();
  if (!enc) return false;
  // element type: the widest of 1/2/4/8 bytes that keeps a row within a 256-element box dimension
  int esz = 1;
  while (esz < 8 && row_bytes / esz > 256) esz *= 2;
  if (row_bytes % esz != 0 || row_bytes / esz > 256 || P->num_heads > 256 || P->block_tokens > 256) return false;
  if (P->num_blocks > INT32_MAX) return false;
  const CUtensorMapDataType type = esz == 1   ? CU_TENSOR_MAP_DATA_TYPE_UINT8
                                   : esz == 2 ? CU_TENSOR_MAP_DATA_TYPE_UINT16
                                   : esz == 4 ? CU_TENSOR_MAP_DATA_TYPE_UINT32
                                              : CU_TENSOR_MAP_DATA_TYPE_INT64;
  const cuuint64_t R = (cuuint64_t)row_bytes, H = P->num_heads, B = P->block_tokens;
  // dimensions innermost first: row elements, head, token, K|V, page; head and
  // token carry each other's strides, so a box lands in [token][head][row] order
  const cuuint64_t dims[5] = {R / esz, H, B, 2, (cuuint64_t)P->num_blocks};
  const cuuint64_t strides[4] = {B * R, R, H * B * R, 2 * H * B * R};
  const cuuint32_t box[5] = {(cuuint32_t)(R / esz), (cuuint32_t)H, (cuuint32_t)B, 1, 1};
  const cuuint32_t elem_strides[5] = {1, 1, 1, 1, 1};
  CUtensorMap* maps = reinterpret_cast<CUtensorMap*>(out);
  for (int l = 0; l < P->num_layers; ++l) {
    if (enc(&maps[l], type, 5, P->layer_base[l], dims, strides, box, elem_strides, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_NONE,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return false;
  }
  return true;
}

// Raise the dynamic shared-memory limit of every TMA kernel once for the
// current device, when a context is created, so that the launch path makes no
// driver attribute calls.
cudaError_t prepare_tma_kernels() {
  cudaError_t e = cudaSuccess;
  for (cudaError_t r : {set_smem(tma_move_kernel<kPack, KVX_LAYOUT_HND>), set_smem(tma_move_kernel<kPack, KVX_LAYOUT_NHD>),
                        set_smem(tma_move_kernel<kUnpack, KVX_LAYOUT_HND>),
                        set_smem(tma_move_kernel<kUnpack, KVX_LAYOUT_NHD>), set_smem(tmap_move_kernel<kPack>),
                        set_smem(tmap_move_kernel<kUnpack>)})
    if (r != cudaSuccess && e == cudaSuccess) e = r;
  return e;
}

// Stage count and shared memory within what the kernels were prepared for.
bool stages_ok(int stage_bytes, int stages) {
  return stages >= 1 && stages <= kStagesMax && stage_bytes > 0 && stage_bytes % 128 == 0 &&
         (int64_t)stage_bytes * stages + 128 <= kTmaSmemMax;
}

cudaError_t launch_move_tma(int dir, int layout, const MoveParams& p, int grid, int stage_bytes, int stages,
                            const TmaWait& wt, cudaStream_t s) {
  if (!stages_ok(stage_bytes, stages) || wt.cycles < 1 || !wt.timeout) return cudaErrorInvalidValue;
  const size_t smem = (size_t)stage_bytes * stages + 128;
  auto go = [&](auto kernel) {
    kernel<<<grid, 32, smem, s>>>(p, stage_bytes, stages, wt);
    return cudaGetLastError();
  };
  if (dir == kPack)
    return layout == KVX_LAYOUT_HND ? go(tma_move_kernel<kPack, KVX_LAYOUT_HND>)
                                    : go(tma_move_kernel<kPack, KVX_LAYOUT_NHD>);
  return layout == KVX_LAYOUT_HND ? go(tma_move_kernel<kUnpack, KVX_LAYOUT_HND>)
                                  : go(tma_move_kernel<kUnpack, KVX_LAYOUT_NHD>);
}

cudaError_t launch_move_tmap(int dir, const MoveParams& p, const void* maps, int num_layers, int grid,
                             int stage_bytes, int stages, const TmaWait& wt, cudaStream_t s) {
  if (!stages_ok(stage_bytes, stages) || num_layers < 1 || num_layers > KVX_MAX_LAYERS || wt.cycles < 1 ||
      !wt.timeout)
    return cudaErrorInvalidValue;
  TensorMaps m;
  memcpy(m.m, maps, (size_t)num_layers * sizeof(CUtensorMap));
  const size_t smem = (size_t)stage_bytes * stages + 128;
  auto go = [&](auto kernel) {
    kernel<<<grid, 32, smem, s>>>(p, m, stage_bytes, stages, wt);
    return cudaGetLastError();
  };
  return dir == kPack ? go(tmap_move_kernel<kPack>) : go(tmap_move_kernel<kUnpack>);
}

}  // namespace kvx
