// host_alloc.cpp -- page-locked host pools for the shared tier (kv_host_alloc,
// kv_host_alloc_numa, kv_host_alloc_ex, kv_host_free).
//
// Sec. 3.3: the shared tier is one exact-size pinned pool, and a request that
// silently fell back to pageable memory was one of the paper's failures.  A
// pool here comes from the driver's pinned allocator (cudaHostAlloc, portable
// and mapped) unless huge pages or a NUMA placement are asked for; then the
// library maps anonymous memory itself, backs it with transparent huge pages
// where it is large enough, places it, and registers it page-locked,
// portable and mapped.
//
// Why (measured on GB300 with a Grace host and 64 KiB base pages):
// * The SMs' zero-copy accesses (the default transfer mode) ran at the link
//   peak from both kinds of pool in a quiet process.  In the benchmark, whose
//   process also pins and frees other buffers and starts a subprocess,
//   cudaHostAlloc pools held the peak in every run of an interleaved A/B on
//   one machine (200.5-201.8 GB/s), while the library's huge-page pools fell to
//   146-194 GB/s in the same runs: their zero-copy accesses stalled for
//   hundreds of milliseconds after memory-management events in the process.
// * The copy engines (cudaMemcpyAsync, KVX_MODE_STAGED) moved 6-18 GB/s from a
//   pool of base pages, 84 GB/s on average (172-422 ms per 33 GB, from step to
//   step) from cudaHostAlloc memory, and 192 GB/s, the link peak, steadily
//   from a pool fully backed by huge pages.  A pool only partly backed (31.1
//   of 33.3 GB) ran staged at 97 GB/s.
// So the default is the driver's allocator, and KVX_HOST_HUGE asks for the
// huge-page mapping for copy-engine use.  That mapping is huge-page aligned,
// asked for huge pages, faulted in at once (MADV_POPULATE_WRITE), and any
// range still on base pages is collapsed into huge pages (MADV_COLLAPSE)
// before the pages are pinned; a pool that huge pages do not back wholly is
// never handed out.
//
// NUMA: on a host with several memory nodes the pool belongs on the node next
// to the GPU that uses it; mbind with a preferred-node policy places it there
// without risking an out-of-memory kill when the node fills up.  The system
// calls and madvise values are the kernel ABI numbers.

#include <cuda_runtime.h>
#include <errno.h>
#include <stdint.h>
#include <stdio.h>
#include <string.h>
#include <sys/mman.h>
#include <sys/syscall.h>
#include <unistd.h>

#include <mutex>
#include <unordered_map>

#include "kvx_internal.h"

using namespace kvx;

namespace {

constexpr int kMpolPreferred = 1;    // linux/mempolicy.h: MPOL_PREFERRED
constexpr int kMaxNodes = 1024;      // nodes a node mask below can name
constexpr int kMadvPopulateWrite = 23;
constexpr int kMadvCollapse = 25;

// A pool made here.  Mapped pools sit between two inaccessible guard pages,
// so the kernel never merges their mapping with a neighbour's and
// /proc/self/smaps describes exactly the pool.
struct Pool {
  size_t len = 0;           // mapped length; 0 for the driver's allocator
  int64_t bytes = 0;        // requested
  int64_t huge_bytes = 0;   // backed by huge pages when pinned
  int32_t node = -1;        // NUMA node of the first page, or -1
  int32_t source = KVX_HOST_SOURCE_DRIVER;
};
std::mutex g_mu;
std::unordered_map<void*, Pool> g_pools;

bool node_exists(int node) {
  char path[64];
  snprintf(path, sizeof(path), "/sys/devices/system/node/node%d", node);
  return access(path, F_OK) == 0;
}

// Free memory of a node in bytes (its meminfo "MemFree"), or -1 if unknown.
int64_t node_free_bytes(int node) {
  char path[80];
  snprintf(path, sizeof(path), "/sys/devices/system/node/node%d/meminfo", node);
  FILE* f = fopen(path, "r");
  if (!f) return -1;
  char line[256];
  long long kb = -1;
  while (fgets(line, sizeof(line), f)) {
    const char* p = strstr(line, "MemFree:");
    if (p && sscanf(p + 8, "%lld", &kb) == 1) break;
  }
  fclose(f);
  return kb < 0 ? -1 : (int64_t)kb * 1024;
}

// Size of a transparent huge page (PMD), or 0 if the kernel does not say.
size_t huge_page_bytes() {
  FILE* f = fopen("/sys/kernel/mm/transparent_hugepage/hpage_pmd_size", "r");
  if (!f) return 0;
  unsigned long v = 0;
  if (fscanf(f, "%lu", &v) != 1) v = 0;
  fclose(f);
  return (size_t)v;
}

// Node of the page holding `addr` (move_pages query form), or -1.
int page_node(void* addr) {
  void* pages[1] = {addr};
  int status[1] = {-1};
  if (syscall(SYS_move_pages, 0, 1, pages, nullptr, status, 0) != 0) return -1;
  return status[0] >= 0 ? status[0] : -1;
}

// Transparent huge pages can be had for a mapping that asks (not "never").
bool thp_available() {
  FILE* f = fopen("/sys/kernel/mm/transparent_hugepage/enabled", "r");
  if (!f) return false;
  char line[128] = "";
  const bool ok = fgets(line, sizeof(line), f) != nullptr && strstr(line, "[never]") == nullptr;
  fclose(f);
  return ok;
}

// The driver's pinned allocator (cudaHostAlloc, portable and mapped).
kvx_status driver_pool(int64_t bytes, void** out) {
  void* p = nullptr;
  const cudaError_t e = cudaHostAlloc(&p, (size_t)bytes, cudaHostAllocPortable | cudaHostAllocMapped);
  if (e != cudaSuccess) {
    set_last_cuda_error((int)e);
    set_error_text("cudaHostAlloc of the host pool");
    cudaGetLastError();
    return e == cudaErrorMemoryAllocation ? KVX_ENOMEM : KVX_ECUDA;
  }
  Pool rec;
  rec.bytes = bytes;
  rec.node = page_node(p);  // -1 where the kernel does not say for the driver's mapping
  {
    std::lock_guard<std::mutex> g(g_mu);
    g_pools[p] = rec;
  }
  *out = p;
  return KVX_OK;
}

// Bytes of [p, p + len) backed by transparent huge pages (AnonHugePages of the
// mappings inside that range in /proc/self/smaps), or -1 if unreadable.
int64_t huge_backed_bytes(const void* p, size_t len) {
  FILE* f = fopen("/proc/self/smaps", "r");
  if (!f) return -1;
  const uintptr_t a = (uintptr_t)p, b = a + len;
  char line[512];
  bool inside = false;
  long long total_kb = 0;
  while (fgets(line, sizeof(line), f)) {
    unsigned long lo = 0, hi = 0;
    long long kb = 0;
    if (sscanf(line, "%lx-%lx ", &lo, &hi) == 2 && strchr(line, ':') != nullptr && line[0] != ' ' &&
        strncmp(line, "AnonHugePages", 13) != 0) {
      inside = lo >= a && hi <= b;
    } else if (inside && sscanf(line, "AnonHugePages: %lld kB", &kb) == 1) {
      total_kb += kb;
    }
  }
  fclose(f);
  return (int64_t)total_kb * 1024;
}

// Maps a pool of at least `bytes` between two guard pages, places it on
// `node` (>= 0), backs it with huge pages (huge) or explicitly with base
// pages, faults it in and pins it.  KVX_EAGAIN-like outcome: returns
// KVX_ENOMEM with *partial set when huge pages were asked but did not back
// the whole pool; the mapping is then already released.
kvx_status map_pool(int node, int64_t bytes, bool huge_pages, void** out, bool* partial) {
  *partial = false;
  const size_t page = (size_t)sysconf(_SC_PAGESIZE);
  const size_t huge = huge_page_bytes();
  const size_t unit = huge_pages ? huge : page;
  const size_t len = ((size_t)bytes + unit - 1) / unit * unit;
  const size_t span = len + 2 * unit;  // room to align the start and keep a guard page on each side
  uint8_t* raw = (uint8_t*)mmap(nullptr, span, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS, -1, 0);
  if (raw == (uint8_t*)MAP_FAILED) {
    set_error_text("mmap of the host pool failed");
    return KVX_ENOMEM;
  }
  uint8_t* p = (uint8_t*)(((uintptr_t)raw + page + unit - 1) / unit * unit);  // >= one page in
  uint8_t* lo = p - page;
  uint8_t* hi = p + len + page;
  if (lo > raw) munmap(raw, (size_t)(lo - raw));
  if (raw + span > hi) munmap(hi, (size_t)(raw + span - hi));
  mprotect(lo, page, PROT_NONE);
  mprotect(p + len, page, PROT_NONE);
  auto release = [&] { munmap(lo, (size_t)(hi - lo)); };
  if (node >= 0) {
    unsigned long mask[kMaxNodes / (8 * sizeof(unsigned long))] = {};
    mask[node / (8 * sizeof(unsigned long))] |= 1ul << (node % (8 * sizeof(unsigned long)));
    // maxnode counts one more than the bits the kernel reads from the mask
    if (syscall(SYS_mbind, p, len, kMpolPreferred, mask, (unsigned long)kMaxNodes + 1, 0u) != 0) {
      release();
      set_error_text("mbind of the host pool failed");
      return KVX_EINVAL;
    }
  }
  int64_t huge_bytes = 0;
  if (huge_pages) {
    madvise(p, len, MADV_HUGEPAGE);
    madvise(p, len, kMadvPopulateWrite);  // fault in now, as huge pages where the kernel can
    for (int attempt = 0; attempt < 3; ++attempt) {
      huge_bytes = huge_backed_bytes(p, len);
      if (huge_bytes >= (int64_t)len) break;
      madvise(p, len, kMadvCollapse);     // collapse what is still on base pages
    }
    huge_bytes = huge_backed_bytes(p, len);
    if (huge_bytes < (int64_t)len) {
      // Measured on GB300: a pool partly on huge pages zero-copied at 76 GB/s
      // where one wholly on either kind ran at 202 GB/s.  Never hand one out.
      release();
      *partial = true;
      set_error_text("huge pages could not back the whole host pool");
      return KVX_ENOMEM;
    }
  } else {
    madvise(p, len, MADV_NOHUGEPAGE);    // all base pages: no mixture either
    madvise(p, len, kMadvPopulateWrite);
  }
  // Not inherited by child processes.  Measured on GB300: a fork (a
  // subprocess started by the process that owns the pool) made the next
  // zero-copy store through a pinned private pool take 2.4 s instead of 43 ms
  // and split its huge-page mappings, and khugepaged collapsing them again
  // 12 s later cost another 0.9 s store; with the pool kept out of the child,
  // neither happened.
  if (madvise(p, len, MADV_DONTFORK) != 0) {
    release();
    set_error_text("madvise(MADV_DONTFORK) of the host pool failed");
    return KVX_ENOMEM;
  }
  const cudaError_t e = cudaHostRegister(p, len, cudaHostRegisterPortable | cudaHostRegisterMapped);
  if (e != cudaSuccess) {
    set_last_cuda_error((int)e);
    set_error_text("cudaHostRegister of the host pool");
    cudaGetLastError();
    release();
    return e == cudaErrorMemoryAllocation ? KVX_ENOMEM : KVX_ECUDA;
  }
  Pool rec;
  rec.len = len;
  rec.bytes = bytes;
  rec.huge_bytes = huge_bytes;
  rec.node = page_node(p);
  rec.source = KVX_HOST_SOURCE_MAPPED;
  {
    std::lock_guard<std::mutex> g(g_mu);
    g_pools[p] = rec;
  }
  *out = p;
  return KVX_OK;
}

}  // namespace

extern "C" {

kvx_status kv_host_alloc_ex(int64_t bytes, int32_t numa_node, uint32_t flags, void** out, int32_t* numa_out) {
  return guarded([&]() -> kvx_status {
    if (!out) return KVX_EINVAL;
    *out = nullptr;
    if (numa_out) *numa_out = -1;
    if (bytes <= 0 || numa_node < KVX_NUMA_ANY || numa_node >= kMaxNodes ||
        (flags & ~(KVX_HOST_DRIVER | KVX_HOST_HUGE)))
      return KVX_EINVAL;
    if ((flags & KVX_HOST_DRIVER) && (numa_node != KVX_NUMA_ANY || (flags & KVX_HOST_HUGE))) return KVX_EINVAL;
    if (fault_point("host_alloc")) {
      set_last_cuda_error((int)cudaErrorMemoryAllocation);
      set_error_text("pinning of the host pool (injected fault)");
      return KVX_ENOMEM;
    }
    // Without a placement, the driver's allocator unless huge pages are asked
    // for (and can be had); a placement needs the library's own mapping.
    // Huge pages where rounding the pool up to whole huge pages wastes at most
    // an eighth of it.
    const size_t huge = thp_available() ? huge_page_bytes() : 0;
    const size_t rounded = huge ? ((size_t)bytes + huge - 1) / huge * huge : 0;
    const bool huge_fits = huge != 0 && (rounded - (size_t)bytes) * 8 <= (size_t)bytes;
    if (numa_node == KVX_NUMA_ANY && (!(flags & KVX_HOST_HUGE) || !huge_fits)) return driver_pool(bytes, out);
    int node = numa_node;
    if (node == KVX_NUMA_ANY) {
      node = -1;
    } else if (node == KVX_NUMA_NEAREST) {
      int dev = 0, id = -1;
      if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&id, cudaDevAttrHostNumaId, dev) != cudaSuccess)
        id = -1;
      cudaGetLastError();
      node = id >= 0 && id < kMaxNodes && node_exists(id) ? id : -1;  // -1: no placement asked
    } else if (!node_exists(node)) {
      set_error_text("no such host NUMA node");
      return KVX_EINVAL;
    }
    if (node >= 0) {
      const int64_t avail = node_free_bytes(node);
      if (avail >= 0 && avail < bytes) {
        set_error_text("the NUMA node has less free memory than requested");
        return KVX_ENOMEM;
      }
    }
    // If huge pages cannot back all of it: the driver's allocator (no placement
    // asked) or base pages (placement asked).
    bool partial = false;
    kvx_status st = KVX_ENOMEM;
    if (huge_fits) {
      st = map_pool(node, bytes, true, out, &partial);
      if (st != KVX_OK && !partial) return st;
    }
    if (st != KVX_OK) {
      if (numa_node == KVX_NUMA_ANY) return driver_pool(bytes, out);
      st = map_pool(node, bytes, false, out, &partial);
    }
    if (st == KVX_OK && numa_out) *numa_out = page_node(*out);
    return st;
  });
}

kvx_status kv_host_pool_info(const void* host, kvx_host_pool_info* info) {
  if (!host || !info) return KVX_EINVAL;
  std::lock_guard<std::mutex> g(g_mu);
  auto it = g_pools.find(const_cast<void*>(host));
  if (it == g_pools.end()) return KVX_ENOENT;
  const Pool& r = it->second;
  info->bytes = r.bytes;
  info->mapped_bytes = r.len ? (int64_t)r.len : r.bytes;
  info->huge_page_bytes = r.huge_bytes;
  info->numa_node = r.node;
  info->source = r.source;
  return KVX_OK;
}

kvx_status kv_host_alloc(int64_t bytes, void** out) {
  return kv_host_alloc_ex(bytes, KVX_NUMA_ANY, 0, out, nullptr);
}

kvx_status kv_host_alloc_numa(int32_t numa_node, int64_t bytes, void** out, int32_t* numa_out) {
  if (numa_node < KVX_NUMA_NEAREST) {
    if (out) *out = nullptr;
    return KVX_EINVAL;
  }
  return kv_host_alloc_ex(bytes, numa_node, 0, out, numa_out);
}

void kv_host_free(void* p) {
  if (!p) return;
  Pool rec;
  {
    std::lock_guard<std::mutex> g(g_mu);
    auto it = g_pools.find(p);
    if (it == g_pools.end()) return;  // not a pool of this library
    rec = it->second;
    g_pools.erase(it);
  }
  if (rec.source == KVX_HOST_SOURCE_DRIVER) {
    cudaFreeHost(p);
  } else {
    cudaHostUnregister(p);
    cudaGetLastError();
    const size_t page = (size_t)sysconf(_SC_PAGESIZE);
    munmap((uint8_t*)p - page, rec.len + 2 * page);  // the pool and its two guard pages
  }
  cudaGetLastError();
}

}  // extern "C"
