// tma_kernels.cu -- device-side pack / unpack with the Tensor Memory
// Accelerator's bulk copies (cp.async.bulk) staged through shared memory.
//
// Same work units and byte mapping as move_kernel (pack_kernels.cu): one
// (chunk, layer, page, K|V) unit at a time, here per CTA of one warp.  A unit
// is copied global -> shared by bulk copies that complete on an mbarrier, then
// shared -> global by bulk copies tracked as bulk groups.  The page side
// moves one 256-byte (row-sized) bulk copy per (head, token) row, landing in
// or leaving from shared memory in the chunk's [token][head] order; the chunk
// side moves as one contiguous bulk copy.  A ring of kStages shared-memory
// stages keeps the loads of the next units in flight while the current unit
// is stored.  Registers never hold the data.
//
// Only for chunks in device memory (kv_pack / kv_unpack / staged mode): the
// zero-copy path keeps the load/store kernel.  Every mbarrier wait is bounded
// by a clock limit; on expiry the kernel sets a timeout flag, drains its own
// bulk stores and returns instead of waiting forever.

#include "kvx_internal.h"

namespace kvx {
namespace {

constexpr int kStagesMax = 4;
constexpr long long kWaitCycles = 4000000000ll;  // about 2 s at the maximum SM clock

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
// Bounded wait on an mbarrier phase; false when the limit expired.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity))
    if (clock64() - t0 > kWaitCycles) return false;
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
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read_1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// One unit resolved to addresses.
struct Unit {
  uint8_t* pg;   // page side (K or V half of the page)
  uint8_t* ck;   // chunk side
  int nr;        // rows (tokens x heads)
  int move;      // 0: nothing to move (past a short chunk's end, or a bad page)
};

// Same decode as move_kernel; a bad table entry zero-fills the chunk rows
// (pack) with ordinary stores and reports the logical block.
template <int DIR>
__device__ __forceinline__ Unit decode(const MoveParams& p, int64_t u, int& j, int64_t& job_begin, int lane) {
  Unit r{nullptr, nullptr, 0, 0};
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
    // lane < 0: a second decode of the same unit (store side), which must not repeat these writes
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
  return r;
}

// Issue the global -> shared copies of one unit into `stage`.
template <int DIR, int LAYOUT>
__device__ __forceinline__ void issue_loads(const MoveParams& p, const Unit& w, uint8_t* stage, uint64_t* bar,
                                            int lane) {
  const uint32_t bytes = w.move ? (uint32_t)(w.nr * p.R) : 0u;
  if (lane == 0) mbar_expect_tx(bar, bytes);
  __syncwarp();
  if (!w.move) return;
  if (DIR == kUnpack || LAYOUT == KVX_LAYOUT_NHD) {
    // chunk side (unpack) or an NHD page (pack): one contiguous run
    if (lane == 0) bulk_load(stage, DIR == kUnpack ? w.ck : w.pg, bytes, bar);
  } else {
    // HND page rows (h, s) land at the chunk's row r = s * H + h
    for (int r = lane; r < w.nr; r += 32) {
      const int s = r / p.H, h = r - s * p.H;
      bulk_load(stage + (int64_t)r * p.R, w.pg + ((int64_t)h * p.B + s) * p.R, (uint32_t)p.R, bar);
    }
  }
}

// Issue the shared -> global copies of one unit from `stage`.
template <int DIR, int LAYOUT>
__device__ __forceinline__ void issue_stores(const MoveParams& p, const Unit& w, const uint8_t* stage, int lane) {
  if (w.move) {
    const uint32_t bytes = (uint32_t)(w.nr * p.R);
    if (DIR == kPack || LAYOUT == KVX_LAYOUT_NHD) {
      if (lane == 0) bulk_store(DIR == kPack ? w.ck : w.pg, stage, bytes);
    } else {
      for (int r = lane; r < w.nr; r += 32) {
        const int s = r / p.H, h = r - s * p.H;
        bulk_store(w.pg + ((int64_t)h * p.B + s) * p.R, stage + (int64_t)r * p.R, (uint32_t)p.R);
      }
    }
  }
  bulk_commit();
}

template <int DIR, int LAYOUT>
__global__ void __launch_bounds__(32) tma_move_kernel(const __grid_constant__ MoveParams p, int stage_bytes,
                                                      int stages, int* timeout) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ __align__(8) uint64_t bars[kStagesMax];
  const int lane = threadIdx.x;
  if (lane == 0) {
    for (int k = 0; k < stages; ++k) mbar_init(&bars[k], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncwarp();
  const int64_t first = blockIdx.x, step = gridDim.x;
  const int64_t n = p.total_units > first ? (p.total_units - first + step - 1) / step : 0;
  // decode cursors: one for loads (runs ahead), one for stores
  int jl = 0, js = 0;
  int64_t bl = 0, bs = 0;
  const int64_t pro = n < stages - 1 ? n : stages - 1;
  for (int64_t it = 0; it < pro; ++it) {
    const Unit w = decode<DIR>(p, first + it * step, jl, bl, lane);
    issue_loads<DIR, LAYOUT>(p, w, smem + it * stage_bytes, &bars[it], lane);
  }
  bool ok = true;
  for (int64_t it = 0; it < n && ok; ++it) {
    const int k = (int)(it % stages);
    const Unit w = decode<DIR>(p, first + it * step, js, bs, -1);  // lane -1: no side effects
    if (lane == 0) ok = mbar_wait(&bars[k], (uint32_t)((it / stages) & 1));
    ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
    if (!ok) break;
    issue_stores<DIR, LAYOUT>(p, w, smem + (int64_t)k * stage_bytes, lane);
    const int64_t nxt = it + stages - 1;
    if (nxt < n) {
      bulk_wait_read_1();  // the store issued from this stage one turn ago has read it
      __syncwarp();
      const int kn = (int)(nxt % stages);
      const Unit wn = decode<DIR>(p, first + nxt * step, jl, bl, lane);
      issue_loads<DIR, LAYOUT>(p, wn, smem + (int64_t)kn * stage_bytes, &bars[kn], lane);
    }
  }
  if (!ok && lane == 0) atomicExch(timeout, 1);
  bulk_wait_all();
}

}  // namespace

cudaError_t launch_move_tma(int dir, int layout, const MoveParams& p, int grid, int stage_bytes, int stages,
                            int* timeout, cudaStream_t s) {
  const size_t smem = (size_t)stage_bytes * stages;
  auto go = [&](auto kernel) {
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    kernel<<<grid, 32, smem, s>>>(p, stage_bytes, stages, timeout);
    return cudaGetLastError();
  };
  if (dir == kPack)
    return layout == KVX_LAYOUT_HND ? go(tma_move_kernel<kPack, KVX_LAYOUT_HND>)
                                    : go(tma_move_kernel<kPack, KVX_LAYOUT_NHD>);
  return layout == KVX_LAYOUT_HND ? go(tma_move_kernel<kUnpack, KVX_LAYOUT_HND>)
                                  : go(tma_move_kernel<kUnpack, KVX_LAYOUT_NHD>);
}

}  // namespace kvx
