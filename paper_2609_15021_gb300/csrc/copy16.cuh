// copy16.cuh -- 16-byte streaming copies shared by the move kernels
// (pack_kernels.cu) and the segment kernel (segment_kernels.cu); device code.
#pragma once

#include <stdint.h>

#include "kvx_internal.h"

namespace kvx {
namespace {

constexpr int kInflight = 8;  // 16-byte vectors per lane between loads and stores

// Streaming (evict-first) accesses: every byte is touched exactly once.
__device__ __forceinline__ uint4 ld16(const uint8_t* p) {
  return __ldcs(reinterpret_cast<const uint4*>(p));
}
__device__ __forceinline__ void st16(uint8_t* p, const uint4& v) {
  __stcs(reinterpret_cast<uint4*>(p), v);
}

// Move kInflight vectors: pack reads the page side, unpack reads the chunk side.
template <int DIR>
__device__ __forceinline__ void move_batch(uint8_t* pg, uint8_t* ck, const int64_t (&po)[kInflight],
                                           const int64_t (&co)[kInflight]) {
  uint4 v[kInflight];
  if (DIR == kPack) {
#pragma unroll
    for (int i = 0; i < kInflight; ++i) v[i] = ld16(pg + po[i]);
#pragma unroll
    for (int i = 0; i < kInflight; ++i) st16(ck + co[i], v[i]);
  } else {
#pragma unroll
    for (int i = 0; i < kInflight; ++i) v[i] = ld16(ck + co[i]);
#pragma unroll
    for (int i = 0; i < kInflight; ++i) st16(pg + po[i], v[i]);
  }
}

template <int DIR>
__device__ __forceinline__ void move_one(uint8_t* pg, uint8_t* ck, int64_t po, int64_t co) {
  if (DIR == kPack)
    st16(ck + co, ld16(pg + po));
  else
    st16(pg + po, ld16(ck + co));
}

// Same byte order on both sides (NHD pages, opaque segments): a flat copy of
// nbytes (a multiple of 16).
template <int DIR>
__device__ __forceinline__ void move_flat(uint8_t* pg, uint8_t* ck, int64_t nbytes, int lane) {
  int64_t off = (int64_t)lane * 16;
  constexpr int64_t kStep = 32 * 16;
  for (; off + (kInflight - 1) * kStep < nbytes; off += kInflight * kStep) {
    int64_t o[kInflight];
#pragma unroll
    for (int i = 0; i < kInflight; ++i) o[i] = off + i * kStep;
    move_batch<DIR>(pg, ck, o, o);
  }
  for (; off < nbytes; off += kStep) move_one<DIR>(pg, ck, off, off);
}

}  // namespace
}  // namespace kvx
