// tier.cpp -- the shared host tier: fixed-size chunk slots in one pinned pool,
// keyed by prefix-chained chunk keys, evicted least-recently-used.
//
// Paper Table 1: the shared tier is one pinned RAM pool holding fixed-token
// chunks with LRU eviction.  Sec. 3.2: a copy must be ordered on the current
// stream, and the related reports it cites concern asynchronous-copy buffers
// reused too early.  So an entry written by an asynchronous store becomes
// readable only through an event recorded on the writer's stream (a reader's
// stream waits on it), and a slot is never handed out again while work that
// reads or writes it may still be running: pinned entries, and entries whose
// release event has not completed, are not evicted.  Sec. 3.2 / Sec. 4.4: a
// cache salt forces a cold path and namespaces must not collide, so keys
// include a caller salt.

#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>

#include <mutex>
#include <new>
#include <unordered_map>
#include <vector>

#include "kvx_internal.h"

using namespace kvx;

namespace {

enum SlotState : int { kFree = 0, kWriting = 1, kReady = 2 };

struct Slot {
  uint64_t key = 0;
  int state = kFree;
  int64_t pins = 0;             // outstanding reserve/acquire without release
  uint64_t tick = 0;            // last use, for LRU
  cudaEvent_t ready = nullptr;  // recorded by commit on the writer's stream
  bool ready_recorded = false;
  cudaEvent_t done = nullptr;   // recorded by release on the user's stream
  bool done_recorded = false;
};

// SplitMix64 finaliser (Steele, Lea & Flood 2014) as the mixing step.
uint64_t mix64(uint64_t z) {
  z += 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

bool no_stream(kvx_stream_t s) { return s == KVX_NO_STREAM; }

kvx_status cuda_fail(cudaError_t e, const char* what) {
  set_last_cuda_error((int)e);
  set_error_text(what);
  cudaGetLastError();
  return KVX_ECUDA;
}

}  // namespace

struct kvx_tier {
  uint8_t* base = nullptr;
  bool owns = false;
  int64_t slot_bytes = 0;
  std::vector<Slot> slots;
  std::unordered_map<uint64_t, int64_t> index;  // key -> slot
  uint64_t clock = 0;
  int64_t hits = 0, misses = 0, evictions = 0;
  std::mutex mu;
};

namespace {

// An entry may be evicted when nothing pins it and the work that wrote it
// (commit event) and the work that last used it (release event) have
// completed on the GPU.
bool evictable(Slot& s) {
  if (s.pins > 0) return false;
  if (s.ready_recorded) {
    const cudaError_t q = cudaEventQuery(s.ready);
    if (q == cudaErrorNotReady) return false;
    cudaGetLastError();
  }
  if (s.done_recorded) {
    const cudaError_t q = cudaEventQuery(s.done);
    if (q == cudaErrorNotReady) return false;
    cudaGetLastError();
    s.done_recorded = false;
  }
  return true;
}

// Free slot, else the least recently used evictable one; -1 if none.
int64_t pick_slot(kvx_tier* t) {
  int64_t best = -1;
  for (int64_t i = 0; i < (int64_t)t->slots.size(); ++i) {
    Slot& s = t->slots[i];
    if (s.state == kFree) return i;
  }
  for (int64_t i = 0; i < (int64_t)t->slots.size(); ++i) {
    Slot& s = t->slots[i];
    if (!evictable(s)) continue;
    if (best < 0 || s.tick < t->slots[best].tick) best = i;
  }
  return best;
}

kvx_status ensure_event(cudaEvent_t* e) {
  if (*e) return KVX_OK;
  const cudaError_t r = cudaEventCreateWithFlags(e, cudaEventDisableTiming);
  if (r != cudaSuccess) {
    *e = nullptr;
    return cuda_fail(r, "cudaEventCreateWithFlags for a tier entry");
  }
  return KVX_OK;
}

void destroy_tier(kvx_tier* t) {
  if (!t) return;
  for (Slot& s : t->slots) {
    if (s.ready) cudaEventDestroy(s.ready);
    if (s.done) cudaEventDestroy(s.done);
  }
  cudaGetLastError();
  if (t->owns) kv_host_free(t->base);
  delete t;
}

}  // namespace

extern "C" {

kvx_status kv_chunk_keys(const int32_t* tokens, int64_t n_tokens, int32_t chunk_tokens, uint64_t salt,
                         uint64_t* keys, int64_t n_keys) {
  if (n_tokens < 0 || chunk_tokens < 1 || (n_tokens > 0 && (!tokens || !keys))) return KVX_EINVAL;
  const int64_t n = (n_tokens + chunk_tokens - 1) / chunk_tokens;
  if (n_keys < n) return KVX_ERANGE;
  uint64_t h = mix64(salt ^ 0x6B767866u);  // chain seed: the salt (namespace)
  for (int64_t c = 0; c < n; ++c) {
    const int64_t lo = c * chunk_tokens;
    const int64_t hi = lo + chunk_tokens < n_tokens ? lo + chunk_tokens : n_tokens;
    h = mix64(h ^ (uint64_t)(hi - lo));            // a short last chunk differs by length
    for (int64_t i = lo; i < hi; ++i) h = mix64(h ^ (uint32_t)tokens[i]);
    keys[c] = h;                                    // depends on every token before it
  }
  return KVX_OK;
}

kvx_status kv_tier_create_on(void* base, int64_t slot_bytes, int64_t n_slots, kvx_tier** out) {
  if (!out) return KVX_EINVAL;
  *out = nullptr;
  if (!base || slot_bytes < 16 || slot_bytes % 16 != 0 || n_slots < 1) return KVX_EINVAL;
  if ((uintptr_t)base & 15) return KVX_EALIGN;
  kvx_tier* t = new (std::nothrow) kvx_tier;
  if (!t) return KVX_ENOMEM;
  t->base = (uint8_t*)base;
  t->slot_bytes = slot_bytes;
  t->slots.resize((size_t)n_slots);
  *out = t;
  return KVX_OK;
}

kvx_status kv_tier_create(int64_t slot_bytes, int64_t n_slots, kvx_tier** out) {
  if (!out) return KVX_EINVAL;
  *out = nullptr;
  if (slot_bytes < 16 || slot_bytes % 16 != 0 || n_slots < 1) return KVX_EINVAL;
  if (n_slots > INT64_MAX / slot_bytes) return KVX_EINVAL;
  void* p = nullptr;
  kvx_status st = kv_host_alloc(slot_bytes * n_slots, &p);
  if (st != KVX_OK) return st;
  st = kv_tier_create_on(p, slot_bytes, n_slots, out);
  if (st != KVX_OK) {
    kv_host_free(p);
    return st;
  }
  (*out)->owns = true;
  return KVX_OK;
}

void kv_tier_destroy(kvx_tier* t) { destroy_tier(t); }

kvx_status kv_tier_reserve(kvx_tier* t, uint64_t key, void** slot) {
  if (!t || !slot) return KVX_EINVAL;
  std::lock_guard<std::mutex> lock(t->mu);
  auto it = t->index.find(key);
  int64_t i;
  if (it != t->index.end()) {
    i = it->second;
    Slot& s = t->slots[i];
    if (s.pins > 0 || !evictable(s)) return KVX_EBUSY;  // in use: cannot be rewritten now
  } else {
    i = pick_slot(t);
    if (i < 0) {
      set_error_text("every tier slot is pinned or still in use by the GPU");
      return KVX_ENOMEM;
    }
    Slot& s = t->slots[i];
    if (s.state != kFree) {
      t->index.erase(s.key);
      t->evictions++;
    }
    t->index[key] = i;
  }
  Slot& s = t->slots[i];
  s.key = key;
  s.state = kWriting;
  s.ready_recorded = false;
  s.pins = 1;
  s.tick = ++t->clock;
  *slot = t->base + i * t->slot_bytes;
  return KVX_OK;
}

kvx_status kv_tier_commit(kvx_tier* t, uint64_t key, kvx_stream_t stream) {
  if (!t) return KVX_EINVAL;
  std::lock_guard<std::mutex> lock(t->mu);
  auto it = t->index.find(key);
  if (it == t->index.end()) return KVX_ENOENT;
  Slot& s = t->slots[it->second];
  if (s.state != kWriting) return KVX_EINVAL;
  if (!no_stream(stream)) {
    kvx_status st = ensure_event(&s.ready);
    if (st != KVX_OK) return st;
    const cudaError_t e = cudaEventRecord(s.ready, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventRecord (tier commit)");
    s.ready_recorded = true;
  }
  s.state = kReady;
  s.pins = s.pins > 0 ? s.pins - 1 : 0;
  s.tick = ++t->clock;
  return KVX_OK;
}

kvx_status kv_tier_acquire(kvx_tier* t, uint64_t key, kvx_stream_t stream, void** slot) {
  if (!t || !slot) return KVX_EINVAL;
  std::lock_guard<std::mutex> lock(t->mu);
  auto it = t->index.find(key);
  if (it == t->index.end() || t->slots[it->second].state != kReady) {
    t->misses++;
    return KVX_ENOENT;
  }
  Slot& s = t->slots[it->second];
  if (s.ready_recorded && !no_stream(stream)) {
    const cudaError_t e = cudaStreamWaitEvent((cudaStream_t)stream, s.ready, 0);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamWaitEvent (tier acquire)");
  }
  s.pins++;
  s.tick = ++t->clock;
  t->hits++;
  *slot = t->base + it->second * t->slot_bytes;
  return KVX_OK;
}

kvx_status kv_tier_release(kvx_tier* t, uint64_t key, kvx_stream_t stream) {
  if (!t) return KVX_EINVAL;
  std::lock_guard<std::mutex> lock(t->mu);
  auto it = t->index.find(key);
  if (it == t->index.end()) return KVX_ENOENT;
  Slot& s = t->slots[it->second];
  if (s.pins < 1) return KVX_EINVAL;
  if (!no_stream(stream)) {
    kvx_status st = ensure_event(&s.done);
    if (st != KVX_OK) return st;
    const cudaError_t e = cudaEventRecord(s.done, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventRecord (tier release)");
    s.done_recorded = true;
  }
  s.pins--;
  return KVX_OK;
}

kvx_status kv_tier_prefix_hits(kvx_tier* t, const uint64_t* keys, int64_t n, int64_t* hits) {
  if (!t || !hits || n < 0 || (n > 0 && !keys)) return KVX_EINVAL;
  std::lock_guard<std::mutex> lock(t->mu);
  int64_t h = 0;
  while (h < n) {
    auto it = t->index.find(keys[h]);
    if (it == t->index.end() || t->slots[it->second].state != kReady) break;
    ++h;
  }
  *hits = h;
  return KVX_OK;
}

kvx_status kv_tier_stats(kvx_tier* t, kvx_tier_stats* out) {
  if (!t || !out) return KVX_EINVAL;
  std::lock_guard<std::mutex> lock(t->mu);
  out->slots = (int64_t)t->slots.size();
  out->slot_bytes = t->slot_bytes;
  int64_t used = 0, pinned = 0;
  for (const Slot& s : t->slots) {
    used += s.state != kFree;
    pinned += s.pins > 0;
  }
  out->entries = used;
  out->pinned = pinned;
  out->hits = t->hits;
  out->misses = t->misses;
  out->evictions = t->evictions;
  return KVX_OK;
}

}  // extern "C"
