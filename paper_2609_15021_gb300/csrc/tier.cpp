// tier.cpp -- the shared host tier: fixed-size chunk slots in one pinned pool,
// keyed by prefix-chained chunk keys, evicted least-recently-used.
//
// Paper Table 1 / Fig. 1: complete replicas share one pinned RAM pool holding
// fixed-token chunks with LRU eviction.  Sec. 3.2: a copy must be ordered on
// the current stream, and the related reports it cites concern asynchronous-
// copy buffers reused too early.  Sec. 3.2 / Sec. 4.4: a cache salt forces a
// cold path and namespaces must not collide, so keys include a caller salt.
//
// A tier is either private to one process or shared by several (POSIX shared
// memory holding the slot table, a process-shared robust mutex and the data,
// which every process registers as pinned, mapped memory).  Entry states:
//   WRITING    reserved by a writer, not readable
//   COMMITTING committed on the writer's stream, not yet published:
//              readable in the writer's process (the reader's stream waits on
//              the writer's event), invisible to other processes
//   READY      the data is complete: readable everywhere
// A commit on a stream enqueues, behind the writer's work, a publication of
// the commit's sequence number into the shared slot table (a system-scope
// release store by the GPU, tier_kernels.cu).  Any process that finds the
// number there turns COMMITTING into READY, so the entry becomes readable
// everywhere as soon as the GPU has passed the commit, with no further call
// of the writer's process; the writer's own event does the same in its
// process (and is the only path for a private tier).  This is the paper's
// completion-before-consumption rule applied across processes.
// Readers pin entries; a release on a stream keeps the pin until the work on
// that stream completes, so a slot in use by queued GPU work is never evicted.
// Pins are kept per process: when a process sharing the tier dies, its pins
// and the entries it was writing are reclaimed (kv_tier_reclaim, and by
// kv_tier_reserve when it finds no slot), so a crashed replica cannot hold
// slots forever.

#include <cuda_runtime.h>
#include <errno.h>
#include <fcntl.h>
#include <pthread.h>
#include <signal.h>
#include <stddef.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>
#include <sys/mman.h>
#include <sys/stat.h>
#include <time.h>
#include <unistd.h>

#include <algorithm>
#include <deque>
#include <mutex>
#include <new>
#include <unordered_map>
#include <vector>

#include "kvx_internal.h"

using namespace kvx;

namespace {

constexpr uint64_t kMagic = 0x3452454954584B56ull;  // "VKXTIER4"
constexpr int64_t kDataAlign = 2ll << 20;
constexpr int kHolders = 8;  // processes that may pin one entry at the same time

enum SlotState : int32_t { kFree = 0, kWriting = 1, kCommitting = 2, kReady = 3 };

struct Header {
  uint64_t magic;
  int64_t slot_bytes, n_slots, data_offset, total_bytes;
  int64_t index_size;  // entries of the key index: a power of two >= 2 * n_slots
  pthread_mutex_t mu;
  uint64_t clock;
  uint64_t seq;        // commits made on a stream, for their publication
  int64_t hits, misses, evictions;
  volatile int32_t initialised;
};

struct SlotMeta {
  uint64_t key;
  int32_t state;
  int32_t writer_pid;  // process whose event decides COMMITTING -> READY
  int64_t pins;        // outstanding acquires/reserves, and releases whose GPU work is pending
  uint64_t tick;       // last use, for LRU
  // the pins by process, so that a process that died can be dropped from them
  int32_t holder_pid[kHolders];
  int32_t holder_pins[kHolders];
  // A commit on a stream takes the next sequence number; the GPU writes it to
  // `published` once the stream has passed the commit (tier_kernels.cu).
  uint64_t commit_seq;
  uint64_t published;  // written by the GPU: read with acquire loads only
};

// Adds n (may be negative) to pid's pins of m; false if pid holds none and
// every holder place is taken.
bool add_pins(SlotMeta& m, int32_t pid, int32_t n) {
  int free_at = -1;
  for (int h = 0; h < kHolders; ++h) {
    if (m.holder_pins[h] > 0 && m.holder_pid[h] == pid) {
      const int32_t d = n < -m.holder_pins[h] ? -m.holder_pins[h] : n;
      m.holder_pins[h] += d;
      m.pins = m.pins + d > 0 ? m.pins + d : 0;
      return true;
    }
    if (m.holder_pins[h] <= 0 && free_at < 0) free_at = h;
  }
  if (n <= 0) return true;  // nothing held by pid: nothing to drop
  if (free_at < 0) return false;
  m.holder_pid[free_at] = pid;
  m.holder_pins[free_at] = n;
  m.pins += n;
  return true;
}

// A process that holds no pin on m can still get a holder place.
bool has_free_holder(const SlotMeta& m) {
  for (int h = 0; h < kHolders; ++h)
    if (m.holder_pins[h] <= 0) return true;
  return false;
}

void clear_pins(SlotMeta& m) {
  m.pins = 0;
  for (int h = 0; h < kHolders; ++h) m.holder_pins[h] = 0;
}

// A process of this host (pid namespace) that no longer exists.
bool process_gone(int32_t pid) {
  if (pid <= 0) return false;
  return kill(pid, 0) != 0 && errno == ESRCH;
}

// SplitMix64 finaliser (Steele, Lea & Flood 2014) as the mixing step.
uint64_t mix64(uint64_t z) {
  z += 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

bool no_stream(kvx_stream_t s) { return s == KVX_NO_STREAM; }

// Tier calls keep their bookkeeping on the host at call time; on a stream
// being captured into a graph, a replay would repeat their GPU work without it.
bool capturing(kvx_stream_t s) {
  if (no_stream(s)) return false;
  cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing((cudaStream_t)s, &st) != cudaSuccess) {
    cudaGetLastError();
    return false;  // an unusable stream fails at its first use below
  }
  if (st == cudaStreamCaptureStatusNone) return false;
  set_error_text("tier calls cannot be captured into a CUDA graph");
  return true;
}

kvx_status cuda_fail(cudaError_t e, const char* what) {
  set_last_cuda_error((int)e);
  set_error_text(what);
  cudaGetLastError();
  return KVX_ECUDA;
}

struct PendingEvent {
  int64_t slot;
  cudaEvent_t ev;
  uint64_t seq;   // commits: the commit's sequence number
  bool owns_ev;   // the event goes back to the spares with this entry (the last of its batch)
};

}  // namespace

struct kvx_tier {
  // the slot table, key index and counters: in shared memory for a shared tier
  Header* hdr = nullptr;
  SlotMeta* meta = nullptr;
  int64_t* index = nullptr;  // open addressing, linear probing: slot or -1 (empty)
  uint8_t* data = nullptr;
  uint8_t* meta_dev = nullptr;  // device address of meta (shared, registered tiers): publication target
  // ownership
  void* mapping = nullptr;   // shared: the whole mmap; private: the metadata allocation
  int64_t mapping_bytes = 0;
  bool shared = false;
  bool creator = false;
  bool registered = false;   // data registered with cudaHostRegister by this process
  bool owns_data = false;    // private tier whose pool came from kv_host_alloc
  char name[128] = "";
  int32_t pid = 0;
  // this process's pending GPU work on slots
  std::deque<PendingEvent> commits;    // COMMITTING entries written by this process, oldest first
  std::deque<PendingEvent> releases;   // pins held until queued work completes, oldest first
  std::unordered_map<int64_t, int32_t> queued;  // slot -> its releases in `releases`
  std::unordered_map<int64_t, cudaEvent_t> commit_event;  // slot -> event readers here may wait on
  std::vector<cudaEvent_t> spare;
  std::mutex local;          // guards the members above
};

namespace {

void rebuild_index_locked(kvx_tier* t);

// Takes the process-shared table lock.  It is robust: when its holder died,
// the next taker gets it, marks it consistent and rebuilds the key index from
// the slot table, since the holder may have died halfway through moving
// index entries.
void lock_table(kvx_tier* t) {
  if (pthread_mutex_lock(&t->hdr->mu) == EOWNERDEAD) {
    pthread_mutex_consistent(&t->hdr->mu);
    rebuild_index_locked(t);
  }
}

// The tier's own event queries and creations run in relaxed capture mode:
// a tier call made while the calling thread is capturing a graph on another
// stream (reserve, a lookup) then leaves that capture alone.
struct TierLock {
  kvx_tier* t;
  cudaStreamCaptureMode mode = cudaStreamCaptureModeRelaxed;
  bool swapped = false;
  explicit TierLock(kvx_tier* tier) : t(tier) {
    swapped = cudaThreadExchangeStreamCaptureMode(&mode) == cudaSuccess;
    if (!swapped) cudaGetLastError();
    t->local.lock();
    lock_table(t);
  }
  ~TierLock() {
    pthread_mutex_unlock(&t->hdr->mu);
    t->local.unlock();
    if (swapped && cudaThreadExchangeStreamCaptureMode(&mode) != cudaSuccess) cudaGetLastError();
  }
};

cudaEvent_t take_event(kvx_tier* t) {
  if (!t->spare.empty()) {
    cudaEvent_t e = t->spare.back();
    t->spare.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreateWithFlags(&e, cudaEventDisableTiming) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return e;
}

// COMMITTING -> READY once the GPU has published the commit (any process may
// do this: the acquire load pairs with the GPU's system-scope release, so the
// chunk's bytes are complete when the number is seen).
bool promote_published(SlotMeta& m) {
  if (m.state != kCommitting || m.commit_seq == 0) return false;
  if (__atomic_load_n(&m.published, __ATOMIC_ACQUIRE) != m.commit_seq) return false;
  m.state = kReady;
  return true;
}

// Settle this process's completed GPU work: COMMITTING -> READY, pins dropped.
// kFront settles completed work from the front of each queue up to the first
// that is still pending (O(1) amortised: every tier call does it, and work on
// one stream completes in order); kAll checks every entry; kWait waits for all.
enum PollMode { kFront, kAll, kWait };

void settle_commit(kvx_tier* t, const PendingEvent& p) {
  SlotMeta& m = t->meta[p.slot];
  if (m.state == kCommitting && m.writer_pid == t->pid && m.commit_seq == p.seq) m.state = kReady;
  auto it = t->commit_event.find(p.slot);
  if (it != t->commit_event.end() && it->second == p.ev) t->commit_event.erase(it);
  if (p.owns_ev) t->spare.push_back(p.ev);
}

void settle_release(kvx_tier* t, const PendingEvent& p) {
  add_pins(t->meta[p.slot], t->pid, -1);
  auto it = t->queued.find(p.slot);
  if (it != t->queued.end() && --it->second <= 0) t->queued.erase(it);
  if (p.owns_ev) t->spare.push_back(p.ev);
}

void poll_locked(kvx_tier* t, PollMode mode) {
  // The entries of one batch share an event and sit next to each other: the
  // event is asked once for all of them, so they settle together and the
  // last one returns the event only when the others are done with it.
  cudaEvent_t last = nullptr;
  bool last_done = false;
  auto done = [&](cudaEvent_t e) {
    if (e == last) return last_done;
    const cudaError_t q = mode == kWait ? cudaEventSynchronize(e) : cudaEventQuery(e);
    last = e;
    last_done = q != cudaErrorNotReady;
    if (last_done) cudaGetLastError();
    return last_done;
  };
  auto settle = [&](std::deque<PendingEvent>& q, void (*fn)(kvx_tier*, const PendingEvent&)) {
    if (mode == kFront) {
      while (!q.empty() && done(q.front().ev)) {
        fn(t, q.front());
        q.pop_front();
      }
      return;
    }
    std::deque<PendingEvent> pending;
    for (const PendingEvent& p : q) {
      if (done(p.ev))
        fn(t, p);
      else
        pending.push_back(p);
    }
    q.swap(pending);
  };
  settle(t->commits, settle_commit);
  settle(t->releases, settle_release);
  if (mode != kFront && t->meta_dev)  // commits of every process that the GPU has published
    for (int64_t i = 0; i < t->hdr->n_slots; ++i) promote_published(t->meta[i]);
}

// Key index: every slot that is not FREE has exactly one entry, at or after
// (cyclically) the home position of its key; lookups cost O(1) on average
// instead of a scan of every slot.
int64_t index_size_for(int64_t n_slots) {
  int64_t h = 2;
  while (h < 2 * n_slots) h <<= 1;
  return h;
}

int64_t index_home(const kvx_tier* t, uint64_t key) {
  return (int64_t)(mix64(key) & (uint64_t)(t->hdr->index_size - 1));
}

// Position of key in the index, or -1.
int64_t index_pos(const kvx_tier* t, uint64_t key) {
  const int64_t mask = t->hdr->index_size - 1;
  int64_t i = index_home(t, key);
  for (int64_t n = 0; n <= mask; ++n, i = (i + 1) & mask) {
    const int64_t s = t->index[i];
    if (s < 0) return -1;
    if (t->meta[s].key == key) return i;
  }
  return -1;
}

// The index has twice as many entries as slots, so a free entry always exists.
void index_insert(kvx_tier* t, uint64_t key, int64_t slot) {
  const int64_t mask = t->hdr->index_size - 1;
  int64_t i = index_home(t, key);
  while (t->index[i] >= 0) i = (i + 1) & mask;
  t->index[i] = slot;
}

// Removes the entry at position i, moving later entries of the same probe run
// back so that no lookup meets a hole before its key (deletion without
// tombstones for linear probing, Knuth TAOCP vol. 3, 6.4 Algorithm R).
void index_erase_at(kvx_tier* t, int64_t i) {
  const int64_t mask = t->hdr->index_size - 1;
  int64_t j = i;
  for (;;) {
    j = (j + 1) & mask;
    const int64_t s = t->index[j];
    if (s < 0) break;
    const int64_t k = index_home(t, t->meta[s].key);
    const bool stays = i <= j ? (i < k && k <= j) : (i < k || k <= j);
    if (stays) continue;
    t->index[i] = s;
    i = j;
  }
  t->index[i] = -1;
}

// Drops the index entry of a slot that becomes FREE or takes another key
// (called while the slot still holds its old key).
void index_erase(kvx_tier* t, uint64_t key) {
  const int64_t i = index_pos(t, key);
  if (i >= 0) index_erase_at(t, i);
}

// The slot table is the record and the index is derived from it.  The table
// itself is kept valid after every single store: a slot changes its key only
// while WRITING, so a process that dies mid-update leaves at worst a WRITING
// slot of a dead writer (freed by reclaim), never a readable entry under the
// wrong key.  Two live slots with one key cannot arise; should they, the newer
// is indexed and the other is evicted or reclaimed like any unindexed slot.
void rebuild_index_locked(kvx_tier* t) {
  memset(t->index, 0xFF, (size_t)t->hdr->index_size * 8);  // every entry -1: empty
  for (int64_t i = 0; i < t->hdr->n_slots; ++i) {
    const SlotMeta& m = t->meta[i];
    if (m.state == kFree) continue;
    const int64_t pos = index_pos(t, m.key);
    if (pos < 0)
      index_insert(t, m.key, i);
    else if (t->meta[t->index[pos]].tick < m.tick)
      t->index[pos] = i;
  }
}

int64_t find_slot(kvx_tier* t, uint64_t key) {
  const int64_t i = index_pos(t, key);
  if (i < 0) return -1;
  const int64_t s = t->index[i];
  promote_published(t->meta[s]);
  return t->meta[s].state != kFree ? s : -1;
}

// Free slot, else the least recently used slot that is READY and unpinned; -1 if none.
int64_t pick_slot(kvx_tier* t) {
  int64_t best = -1;
  for (int64_t i = 0; i < t->hdr->n_slots; ++i) {
    SlotMeta& m = t->meta[i];
    if (m.state == kFree) return i;
    promote_published(m);
    if (m.state != kReady || m.pins > 0) continue;
    if (best < 0 || m.tick < t->meta[best].tick) best = i;
  }
  return best;
}

// Pins of this process on `slot` whose release is queued behind GPU work.
int64_t queued_releases(const kvx_tier* t, int64_t slot) {
  auto it = t->queued.find(slot);
  return it == t->queued.end() ? 0 : it->second;
}

int32_t pins_of(const SlotMeta& m, int32_t pid) {
  for (int h = 0; h < kHolders; ++h)
    if (m.holder_pins[h] > 0 && m.holder_pid[h] == pid) return m.holder_pins[h];
  return 0;
}

// Shared tier: drop the pins of processes that no longer exist, and free the
// entries they were writing or committing (their bytes may be incomplete; the
// work of a process that died ended with it).  Returns the slots changed.
int64_t reclaim_locked(kvx_tier* t) {
  if (!t->shared) return 0;
  std::unordered_map<int32_t, bool> gone;  // liveness, once per process per scan
  auto is_gone = [&](int32_t pid) {
    auto it = gone.find(pid);
    if (it != gone.end()) return it->second;
    const bool g = pid != t->pid && process_gone(pid);
    gone[pid] = g;
    return g;
  };
  int64_t changed = 0;
  for (int64_t i = 0; i < t->hdr->n_slots; ++i) {
    SlotMeta& m = t->meta[i];
    if (m.state == kFree) continue;
    bool c = false;
    promote_published(m);  // a published commit is complete, whoever made it
    if ((m.state == kWriting || m.state == kCommitting) && is_gone(m.writer_pid)) {
      index_erase(t, m.key);
      m.state = kFree;
      clear_pins(m);
      c = true;
    }
    for (int h = 0; h < kHolders; ++h) {
      if (m.holder_pins[h] > 0 && is_gone(m.holder_pid[h])) {
        m.pins = m.pins > m.holder_pins[h] ? m.pins - m.holder_pins[h] : 0;
        m.holder_pins[h] = 0;
        c = true;
      }
    }
    changed += c;
  }
  return changed;
}

void destroy_tier(kvx_tier* t) {
  if (!t) return;
  {
    std::lock_guard<std::mutex> g(t->local);
    if (t->hdr) {
      lock_table(t);
      poll_locked(t, kWait);  // settle this process's pending work
      pthread_mutex_unlock(&t->hdr->mu);
    }
    for (cudaEvent_t e : t->spare) cudaEventDestroy(e);
    cudaGetLastError();
  }
  if (t->registered) {
    cudaHostUnregister(t->mapping);
    cudaGetLastError();
  }
  if (t->shared) {
    munmap(t->mapping, (size_t)t->mapping_bytes);
    if (t->creator) shm_unlink(t->name);
  } else {
    free(t->mapping);
    if (t->owns_data) kv_host_free(t->data);
  }
  delete t;
}

// Bytes of the header, the slot table and the key index of an n-slot tier.
int64_t metadata_bytes(int64_t n_slots) {
  return (int64_t)sizeof(Header) + n_slots * (int64_t)sizeof(SlotMeta) + index_size_for(n_slots) * 8;
}

// Points t's table and index into the metadata at m (the header already filled).
void attach_metadata(kvx_tier* t, void* m) {
  t->hdr = (Header*)m;
  t->meta = (SlotMeta*)((uint8_t*)m + sizeof(Header));
  t->index = (int64_t*)((uint8_t*)t->meta + t->hdr->n_slots * (int64_t)sizeof(SlotMeta));
}

kvx_status init_private(void* base, int64_t slot_bytes, int64_t n_slots, kvx_tier** out) {
  kvx_tier* t = new (std::nothrow) kvx_tier;
  if (!t) return KVX_ENOMEM;
  void* m = calloc(1, (size_t)metadata_bytes(n_slots));
  if (!m) {
    delete t;
    return KVX_ENOMEM;
  }
  t->mapping = m;
  Header* h = (Header*)m;
  h->magic = kMagic;
  h->slot_bytes = slot_bytes;
  h->n_slots = n_slots;
  h->index_size = index_size_for(n_slots);
  attach_metadata(t, m);
  memset(t->index, 0xFF, (size_t)h->index_size * 8);  // every entry -1: empty
  t->data = (uint8_t*)base;
  t->pid = (int32_t)getpid();
  pthread_mutex_init(&h->mu, nullptr);
  h->initialised = 1;
  *out = t;
  return KVX_OK;
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
  return guarded([&]() -> kvx_status {
    if (!out) return KVX_EINVAL;
    *out = nullptr;
    if (!base || slot_bytes < 16 || slot_bytes % 16 != 0 || n_slots < 1) return KVX_EINVAL;
    if ((uintptr_t)base & 15) return KVX_EALIGN;
    return init_private(base, slot_bytes, n_slots, out);
  });
}

kvx_status kv_tier_create(int64_t slot_bytes, int64_t n_slots, kvx_tier** out) {
  return guarded([&]() -> kvx_status {
    if (!out) return KVX_EINVAL;
    *out = nullptr;
    if (slot_bytes < 16 || slot_bytes % 16 != 0 || n_slots < 1) return KVX_EINVAL;
    if (n_slots > INT64_MAX / slot_bytes) return KVX_EINVAL;
    void* p = nullptr;
    kvx_status st = kv_host_alloc(slot_bytes * n_slots, &p);
    if (st != KVX_OK) return st;
    st = init_private(p, slot_bytes, n_slots, out);
    if (st != KVX_OK) {
      kv_host_free(p);
      return st;
    }
    (*out)->owns_data = true;
    return KVX_OK;
  });
}

kvx_status kv_tier_open_shared(const char* name, int64_t slot_bytes, int64_t n_slots, uint32_t flags,
                               kvx_tier** out) {
  return guarded([&]() -> kvx_status {
    if (!out || !name || name[0] != '/' || strlen(name) >= 120) return KVX_EINVAL;
    *out = nullptr;
    const bool create = (flags & KVX_TIER_CREATE) != 0;
    if (create && (slot_bytes < 16 || slot_bytes % 16 != 0 || n_slots < 1)) return KVX_EINVAL;
    const int fd = shm_open(name, create ? (O_CREAT | O_EXCL | O_RDWR) : O_RDWR, 0600);
    if (fd < 0) {
      set_error_text(create ? "shm_open: the name exists or cannot be created" : "shm_open: no such tier");
      return create ? KVX_EINVAL : KVX_ENOENT;
    }
    int64_t total = 0, data_offset = 0;
    if (create) {
      const int64_t meta_bytes = metadata_bytes(n_slots);
      data_offset = (meta_bytes + kDataAlign - 1) / kDataAlign * kDataAlign;
      if (n_slots > (INT64_MAX - data_offset) / slot_bytes) {
        close(fd);
        shm_unlink(name);
        return KVX_EINVAL;
      }
      total = data_offset + slot_bytes * n_slots;
      if (ftruncate(fd, (off_t)total) != 0) {
        close(fd);
        shm_unlink(name);
        set_error_text("ftruncate of the shared tier failed");
        return KVX_ENOMEM;
      }
      // Reserve the pages now: a shared-memory file system without room for
      // them would otherwise end the process with SIGBUS at first touch.
      const int fr = posix_fallocate(fd, 0, (off_t)total);
      if (fr != 0 && fr != EOPNOTSUPP && fr != EINVAL) {
        close(fd);
        shm_unlink(name);
        set_error_text("the shared-memory file system has no room for the tier");
        return KVX_ENOMEM;
      }
    } else {
      struct stat sb;
      // wait (bounded) for the creator to size and initialise the region
      for (int i = 0; i < 5000; ++i) {
        if (fstat(fd, &sb) == 0 && sb.st_size >= (off_t)sizeof(Header)) break;
        usleep(1000);
      }
      if (fstat(fd, &sb) != 0 || sb.st_size < (off_t)sizeof(Header)) {
        close(fd);
        return KVX_ENOENT;
      }
      total = (int64_t)sb.st_size;
    }
    void* map = mmap(nullptr, (size_t)total, PROT_READ | PROT_WRITE, MAP_SHARED, fd, 0);
    close(fd);
    if (map == MAP_FAILED) {
      if (create) shm_unlink(name);
      return KVX_ENOMEM;
    }
    kvx_tier* t = new (std::nothrow) kvx_tier;
    if (!t) {
      munmap(map, (size_t)total);
      if (create) shm_unlink(name);
      return KVX_ENOMEM;
    }
    t->shared = true;
    t->creator = create;
    t->mapping = map;
    t->mapping_bytes = total;
    t->pid = (int32_t)getpid();
    snprintf(t->name, sizeof(t->name), "%s", name);
    Header* h = (Header*)map;
    t->hdr = h;
    if (create) {
      h->magic = kMagic;
      h->slot_bytes = slot_bytes;
      h->n_slots = n_slots;
      h->data_offset = data_offset;
      h->total_bytes = total;
      h->index_size = index_size_for(n_slots);
      attach_metadata(t, map);
      memset(t->index, 0xFF, (size_t)h->index_size * 8);  // every entry -1: empty
      pthread_mutexattr_t a;
      pthread_mutexattr_init(&a);
      pthread_mutexattr_setpshared(&a, PTHREAD_PROCESS_SHARED);
      pthread_mutexattr_setrobust(&a, PTHREAD_MUTEX_ROBUST);
      pthread_mutex_init(&h->mu, &a);
      pthread_mutexattr_destroy(&a);
      __atomic_store_n(&h->initialised, 1, __ATOMIC_RELEASE);
    } else {
      int i = 0;
      while (__atomic_load_n(&h->initialised, __ATOMIC_ACQUIRE) != 1 && i++ < 5000) usleep(1000);
      if (h->initialised != 1 || h->magic != kMagic || h->total_bytes != total ||
          h->index_size != index_size_for(h->n_slots) || metadata_bytes(h->n_slots) > h->data_offset) {
        munmap(map, (size_t)total);
        delete t;
        set_error_text("the shared tier is not initialised or does not match");
        return KVX_EINVAL;
      }
      attach_metadata(t, map);
    }
    t->data = (uint8_t*)map + h->data_offset;
    // Shared memory is kept on base pages: the SMs' zero-copy accesses run at the
    // link peak on them, and a mixture of page sizes slowed zero-copy on GB300
    // to a third.  (The copy engines are slow on base pages: with a shared tier,
    // zero-copy, the default mode, is the one to use.)
    madvise(t->data, (size_t)(h->slot_bytes * h->n_slots), MADV_NOHUGEPAGE);
    if (!(flags & KVX_TIER_NO_PIN)) {
      // The whole region, slot table included: the GPU publishes commits into it.
      const cudaError_t e = cudaHostRegister(map, (size_t)total, cudaHostRegisterPortable | cudaHostRegisterMapped);
      if (e != cudaSuccess) {
        kvx_status st = cuda_fail(e, "cudaHostRegister of the shared tier");
        t->creator = create;
        destroy_tier(t);
        return st;
      }
      t->registered = true;
      void* dmap = nullptr;
      if (cudaHostGetDevicePointer(&dmap, map, 0) == cudaSuccess && dmap && prepare_tier_kernels() == cudaSuccess)
        t->meta_dev = (uint8_t*)dmap + ((uint8_t*)t->meta - (uint8_t*)map);
      cudaGetLastError();  // without publication, commits turn READY through the writer's events only
    }
    *out = t;
    return KVX_OK;
  });
}

void kv_tier_destroy(kvx_tier* t) { destroy_tier(t); }

kvx_status kv_tier_poll(kvx_tier* t) {
  return guarded([&]() -> kvx_status {
    if (!t) return KVX_EINVAL;
    TierLock lock(t);
    poll_locked(t, kAll);
    return KVX_OK;
  });
}

}  // extern "C"

namespace {

// kv_tier_reserve under the lock, after the caller's poll.
kvx_status reserve_locked(kvx_tier* t, uint64_t key, void** slot) {
  int64_t i = -1;
  // a second pass after reclaiming what processes that died left behind
  for (int pass = 0; pass < 2; ++pass) {
    if (pass == 1) {
      poll_locked(t, kAll);  // completed work behind a pending one frees slots too
      if (reclaim_locked(t) == 0 && pick_slot(t) < 0 && find_slot(t, key) < 0) break;
    }
    i = find_slot(t, key);
    if (i >= 0) {
      const SlotMeta& m = t->meta[i];
      if (m.pins == 0 && m.state == kReady) break;
      i = -2;  // in use: cannot be rewritten now
      continue;
    }
    i = pick_slot(t);
    if (i >= 0) {
      SlotMeta& m = t->meta[i];
      if (m.state != kFree) {
        index_erase(t, m.key);
        t->hdr->evictions++;
      }
      // WRITING before the key changes: were this process to die from here
      // on, the slot is a dead writer's reservation, never old bytes
      // readable under the new key.
      m.writer_pid = t->pid;
      m.state = kWriting;
      m.key = key;
      index_insert(t, key, i);
      if (fault_point("tier_exit")) _exit(3);  // test hook: die holding the lock, mid-reserve
      break;
    }
  }
  if (i == -2) {
    set_error_text("the entry is pinned, being written, or still in use by the GPU");
    return KVX_EBUSY;
  }
  if (i < 0) {
    set_error_text("every tier slot is pinned, being written, or still in use by the GPU");
    return KVX_ENOMEM;
  }
  SlotMeta& m = t->meta[i];
  m.writer_pid = t->pid;
  m.state = kWriting;
  clear_pins(m);
  add_pins(m, t->pid, 1);
  m.tick = ++t->hdr->clock;
  *slot = t->data + i * t->hdr->slot_bytes;
  return KVX_OK;
}

}  // namespace

extern "C" {

kvx_status kv_tier_reserve(kvx_tier* t, uint64_t key, void** slot) {
  return guarded([&]() -> kvx_status {
    if (!t || !slot) return KVX_EINVAL;
    TierLock lock(t);
    poll_locked(t, kFront);
    return reserve_locked(t, key, slot);
  });
}

kvx_status kv_tier_reserve_many(kvx_tier* t, const uint64_t* keys, int64_t n, void** slots, int64_t* n_reserved) {
  return guarded([&]() -> kvx_status {
    if (n_reserved) *n_reserved = 0;
    if (!t || n < 0 || (n > 0 && (!keys || !slots))) return KVX_EINVAL;
    if (n == 0) return KVX_OK;
    TierLock lock(t);
    poll_locked(t, kFront);
    for (int64_t j = 0; j < n; ++j) {
      const kvx_status st = reserve_locked(t, keys[j], &slots[j]);
      if (st != KVX_OK) {
        if (n_reserved) *n_reserved = j;
        return st;
      }
    }
    if (n_reserved) *n_reserved = n;
    return KVX_OK;
  });
}

kvx_status kv_tier_commit(kvx_tier* t, uint64_t key, kvx_stream_t stream) {
  return kv_tier_commit_many(t, &key, 1, stream);
}

kvx_status kv_tier_commit_many(kvx_tier* t, const uint64_t* keys, int64_t n, kvx_stream_t stream) {
  return guarded([&]() -> kvx_status {
    if (!t || n < 0 || (n > 0 && !keys) || capturing(stream)) return KVX_EINVAL;
    if (n == 0) return KVX_OK;
    TierLock lock(t);
    poll_locked(t, kFront);
    std::vector<int64_t> slots((size_t)n);
    std::unordered_map<int64_t, bool> seen;
    for (int64_t j = 0; j < n; ++j) {  // every key first: on an error nothing is committed
      const int64_t i = find_slot(t, keys[j]);
      if (i < 0) return KVX_ENOENT;
      const SlotMeta& m = t->meta[i];
      if (m.state != kWriting || m.writer_pid != t->pid) return KVX_EINVAL;
      if (!seen.emplace(i, true).second) {
        set_error_text("a key is listed twice");
        return KVX_EINVAL;
      }
      slots[(size_t)j] = i;
    }
    if (no_stream(stream)) {
      for (int64_t i : slots) {
        SlotMeta& m = t->meta[i];
        m.state = kReady;
        add_pins(m, t->pid, -1);
        m.tick = ++t->hdr->clock;
      }
      return KVX_OK;
    }
    // The sequence numbers are these commits' alone; a publication that lands
    // after a failure below matches no commit.
    const uint64_t seq0 = t->hdr->seq + 1;
    t->hdr->seq += (uint64_t)n;
    if (t->meta_dev) {
      TierPublish b;
      b.meta = t->meta_dev;
      b.stride = (int64_t)sizeof(SlotMeta);
      b.offset = (int64_t)offsetof(SlotMeta, published);
      for (int64_t j0 = 0; j0 < n; j0 += kMaxPublish) {
        b.n = (int32_t)std::min<int64_t>(kMaxPublish, n - j0);
        b.seq0 = seq0 + (uint64_t)j0;
        for (int32_t j = 0; j < b.n; ++j) b.slot[j] = (int32_t)slots[(size_t)(j0 + j)];
        const cudaError_t r = fault_point("launch") ? cudaErrorUnknown : launch_tier_publish(b, (cudaStream_t)stream);
        if (r != cudaSuccess) return cuda_fail(r, "publication kernel launch (tier commit)");
      }
    }
    cudaEvent_t e = take_event(t);
    if (!e) return cuda_fail(cudaErrorMemoryAllocation, "cudaEventCreate (tier commit)");
    const cudaError_t r = cudaEventRecord(e, (cudaStream_t)stream);
    if (r != cudaSuccess) {
      t->spare.push_back(e);
      return cuda_fail(r, "cudaEventRecord (tier commit)");
    }
    for (int64_t j = 0; j < n; ++j) {
      const int64_t i = slots[(size_t)j];
      SlotMeta& m = t->meta[i];
      m.commit_seq = seq0 + (uint64_t)j;
      m.state = kCommitting;
      // one event for the batch: the last entry gives it back
      t->commits.push_back({i, e, m.commit_seq, j == n - 1});
      t->commit_event[i] = e;
      add_pins(m, t->pid, -1);
      m.tick = ++t->hdr->clock;
    }
    return KVX_OK;
  });
}

kvx_status kv_tier_acquire(kvx_tier* t, uint64_t key, kvx_stream_t stream, void** slot) {
  if (!slot) return KVX_EINVAL;
  return kv_tier_acquire_many(t, &key, 1, stream, slot);
}

kvx_status kv_tier_acquire_many(kvx_tier* t, const uint64_t* keys, int64_t n, kvx_stream_t stream,
                                void** slots) {
  return guarded([&]() -> kvx_status {
    if (!t || n < 0 || (n > 0 && (!keys || !slots)) || capturing(stream)) return KVX_EINVAL;
    if (n == 0) return KVX_OK;
    TierLock lock(t);
    poll_locked(t, kFront);
    std::vector<int64_t> idx((size_t)n);
    std::vector<cudaEvent_t> waits;  // this process's commit events the readers must follow, once each
    for (int64_t j = 0; j < n; ++j) {  // every key first: on an error nothing is pinned
      const int64_t i = find_slot(t, keys[j]);
      bool ok = i >= 0 && t->meta[i].state == kReady;
      if (i >= 0 && t->meta[i].state == kCommitting && t->meta[i].writer_pid == t->pid) {
        auto it = t->commit_event.find(i);  // written here: order the reader on the writer's event
        if (it != t->commit_event.end()) {
          if (std::find(waits.begin(), waits.end(), it->second) == waits.end()) waits.push_back(it->second);
          ok = true;
        }
      }
      if (!ok) {
        t->hdr->misses++;
        return KVX_ENOENT;
      }
      if (pins_of(t->meta[i], t->pid) == 0 && !has_free_holder(t->meta[i])) {
        set_error_text("the entry is pinned by as many processes as it can track");
        return KVX_EBUSY;
      }
      idx[(size_t)j] = i;
    }
    for (cudaEvent_t e : waits) {
      const cudaError_t r = no_stream(stream) ? cudaEventSynchronize(e) : cudaStreamWaitEvent((cudaStream_t)stream, e, 0);
      if (r != cudaSuccess) return cuda_fail(r, no_stream(stream) ? "cudaEventSynchronize (tier acquire)"
                                                                   : "cudaStreamWaitEvent (tier acquire)");
    }
    for (int64_t j = 0; j < n; ++j) {
      const int64_t i = idx[(size_t)j];
      SlotMeta& m = t->meta[i];
      add_pins(m, t->pid, 1);  // cannot fail: a holder place was checked above
      m.tick = ++t->hdr->clock;
      t->hdr->hits++;
      slots[j] = t->data + i * t->hdr->slot_bytes;
    }
    return KVX_OK;
  });
}

kvx_status kv_tier_release(kvx_tier* t, uint64_t key, kvx_stream_t stream) {
  return kv_tier_release_many(t, &key, 1, stream);
}

kvx_status kv_tier_release_many(kvx_tier* t, const uint64_t* keys, int64_t n, kvx_stream_t stream) {
  return guarded([&]() -> kvx_status {
    if (!t || n < 0 || (n > 0 && !keys) || capturing(stream)) return KVX_EINVAL;
    if (n == 0) return KVX_OK;
    TierLock lock(t);
    poll_locked(t, kFront);
    std::vector<int64_t> idx((size_t)n);
    std::unordered_map<int64_t, int64_t> asked;  // releases of each slot in this call
    for (int64_t j = 0; j < n; ++j) {  // every key first: on an error nothing is released
      const int64_t i = find_slot(t, keys[j]);
      if (i < 0) return KVX_ENOENT;
      idx[(size_t)j] = i;
      if (pins_of(t->meta[i], t->pid) - queued_releases(t, i) < ++asked[i]) {
        set_error_text("this process holds no pin on the entry");
        return KVX_EINVAL;
      }
    }
    if (no_stream(stream)) {
      for (int64_t i : idx) {
        SlotMeta& m = t->meta[i];
        add_pins(m, t->pid, -1);
        if (m.state == kWriting && m.pins == 0) {  // a writer giving up its reservation
          index_erase(t, m.key);
          m.state = kFree;
        }
      }
      return KVX_OK;
    }
    cudaEvent_t e = take_event(t);
    if (!e) return cuda_fail(cudaErrorMemoryAllocation, "cudaEventCreate (tier release)");
    const cudaError_t r = cudaEventRecord(e, (cudaStream_t)stream);
    if (r != cudaSuccess) {
      t->spare.push_back(e);
      return cuda_fail(r, "cudaEventRecord (tier release)");
    }
    for (int64_t j = 0; j < n; ++j) {  // the pins stay until the queued work completes; one event for all
      const int64_t i = idx[(size_t)j];
      t->releases.push_back({i, e, 0, j == n - 1});
      t->queued[i]++;
    }
    return KVX_OK;
  });
}

kvx_status kv_tier_reclaim(kvx_tier* t, int64_t* reclaimed) {
  return guarded([&]() -> kvx_status {
    if (!t) return KVX_EINVAL;
    TierLock lock(t);
    poll_locked(t, kFront);
    const int64_t n = reclaim_locked(t);
    if (reclaimed) *reclaimed = n;
    return KVX_OK;
  });
}

kvx_status kv_tier_prefix_hits(kvx_tier* t, const uint64_t* keys, int64_t n, int64_t* hits) {
  return guarded([&]() -> kvx_status {
    if (!t || !hits || n < 0 || (n > 0 && !keys)) return KVX_EINVAL;
    TierLock lock(t);
    poll_locked(t, kFront);
    int64_t h = 0;
    while (h < n) {
      const int64_t i = find_slot(t, keys[h]);
      if (i < 0) break;
      const SlotMeta& m = t->meta[i];
      const bool visible = m.state == kReady || (m.state == kCommitting && m.writer_pid == t->pid);
      if (!visible) break;
      ++h;
    }
    *hits = h;
    return KVX_OK;
  });
}

kvx_status kv_tier_wait(kvx_tier* t, const uint64_t* keys, int64_t n, int64_t timeout_ns, int64_t* hits) {
  return guarded([&]() -> kvx_status {
    if (!t || n < 0 || (n > 0 && !keys) || timeout_ns < 0) return KVX_EINVAL;
    auto now = [] {
      timespec ts;
      clock_gettime(CLOCK_MONOTONIC, &ts);
      return (int64_t)ts.tv_sec * 1000000000ll + ts.tv_nsec;
    };
    const int64_t deadline = now() + timeout_ns;
    int64_t pause_ns = 20000, h = 0;
    for (;;) {
      {
        TierLock lock(t);
        poll_locked(t, kFront);
        // Entries become readable in any order, and one can be evicted again
        // before it is pinned: count the readable prefix from the start each
        // time, a lookup per key.
        h = 0;
        while (h < n) {
          const int64_t i = find_slot(t, keys[h]);
          if (i < 0) break;
          const SlotMeta& m = t->meta[i];
          if (!(m.state == kReady || (m.state == kCommitting && m.writer_pid == t->pid))) break;
          ++h;
        }
      }
      if (h == n || now() >= deadline) break;
      const int64_t left = deadline - now();
      const int64_t d = std::max<int64_t>(0, std::min(pause_ns, left));
      timespec ts{(time_t)(d / 1000000000ll), (long)(d % 1000000000ll)};
      nanosleep(&ts, nullptr);
      pause_ns = std::min<int64_t>(pause_ns * 2, 1000000);
    }
    if (hits) *hits = h;
    if (h == n) return KVX_OK;
    set_error_text("tier entries did not become readable before the wait's limit");
    return KVX_ETIMEOUT;
  });
}

kvx_status kv_tier_stats(kvx_tier* t, kvx_tier_stats* out) {
  return guarded([&]() -> kvx_status {
    if (!t || !out) return KVX_EINVAL;
    TierLock lock(t);
    poll_locked(t, kFront);
    out->slots = t->hdr->n_slots;
    out->slot_bytes = t->hdr->slot_bytes;
    int64_t used = 0, pinned = 0;
    for (int64_t i = 0; i < t->hdr->n_slots; ++i) {
      used += t->meta[i].state != kFree;
      pinned += t->meta[i].pins > 0;
    }
    out->entries = used;
    out->pinned = pinned;
    out->hits = t->hdr->hits;
    out->misses = t->hdr->misses;
    out->evictions = t->hdr->evictions;
    return KVX_OK;
  });
}

}  // extern "C"
