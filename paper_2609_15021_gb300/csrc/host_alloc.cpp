// host_alloc.cpp -- page-locked host pools for the shared tier (kv_host_alloc,
// kv_host_alloc_numa, kv_host_alloc_ex, kv_host_free).
//
// Sec. 3.3: the shared tier is one exact-size pinned pool, and a request that
// silently fell back to pageable memory was one of the paper's failures.  A
// pool here is anonymous memory mapped by the library, backed by transparent
// huge pages where it is large enough, optionally placed on one NUMA node,
// and registered page-locked, portable and mapped.
//
// Why huge pages (measured on GB300 with a Grace host and 64 KiB base pages):
// the SMs' zero-copy accesses run at the link peak whatever backs the pool,
// but the copy engines (cudaMemcpyAsync, the staged mode) moved 6-18 GB/s
// from a pool of base pages, 84 GB/s on average (172-422 ms per 33 GB, from
// step to step) from cudaHostAlloc memory, and 192 GB/s, the link peak,
// steadily from a pool fully backed by huge pages.  A pool only partly backed
// (31.1 of 33.3 GB) ran staged at 97 GB/s.  So the mapping is huge-page
// aligned, asked for huge pages, faulted in at once (MADV_POPULATE_WRITE),
// and any range still on base pages is collapsed into huge pages
// (MADV_COLLAPSE) before the pages are pinned; both are advice, so the pool
// is still created if the kernel cannot comply.  Where no huge page can back
// the pool (smaller than one, or a host without transparent huge pages) and
// no placement is asked, the driver's allocator serves instead, as it does on
// request (KVX_HOST_DRIVER).
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

std::mutex g_mu;
std::unordered_map<void*, size_t> g_mappings;  // pools made here: base -> mapped length

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
  {
    std::lock_guard<std::mutex> g(g_mu);
    g_mappings[p] = 0;  // length 0: freed with cudaFreeHost
  }
  *out = p;
  return KVX_OK;
}

// Maps, places (node >= 0), backs with huge pages where possible and pins a
// pool of at least `bytes`.  On success *out is the pool and *len_out the
// mapped length.
kvx_status map_pool(int node, int64_t bytes, void** out, size_t* len_out) {
  const size_t page = (size_t)sysconf(_SC_PAGESIZE);
  const size_t huge = thp_available() ? huge_page_bytes() : 0;
  const bool use_huge = huge >= page && (size_t)bytes >= huge;
  const size_t unit = use_huge ? huge : page;
  const size_t len = ((size_t)bytes + unit - 1) / unit * unit;
  const size_t span = use_huge ? len + huge : len;  // room to align the start
  uint8_t* raw = (uint8_t*)mmap(nullptr, span, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS, -1, 0);
  if (raw == (uint8_t*)MAP_FAILED) {
    set_error_text("mmap of the host pool failed");
    return KVX_ENOMEM;
  }
  uint8_t* p = raw;
  if (use_huge) {
    p = (uint8_t*)(((uintptr_t)raw + huge - 1) / huge * huge);
    if (p > raw) munmap(raw, (size_t)(p - raw));
    const size_t tail = (size_t)(raw + span - (p + len));
    if (tail) munmap(p + len, tail);
  }
  if (node >= 0) {
    unsigned long mask[kMaxNodes / (8 * sizeof(unsigned long))] = {};
    mask[node / (8 * sizeof(unsigned long))] |= 1ul << (node % (8 * sizeof(unsigned long)));
    // maxnode counts one more than the bits the kernel reads from the mask
    if (syscall(SYS_mbind, p, len, kMpolPreferred, mask, (unsigned long)kMaxNodes + 1, 0u) != 0) {
      munmap(p, len);
      set_error_text("mbind of the host pool failed");
      return KVX_EINVAL;
    }
  }
  if (use_huge) {
    madvise(p, len, MADV_HUGEPAGE);
    madvise(p, len, kMadvPopulateWrite);  // fault in now, as huge pages where the kernel can
    madvise(p, len, kMadvCollapse);       // and collapse what it could not
  }
  const cudaError_t e = cudaHostRegister(p, len, cudaHostRegisterPortable | cudaHostRegisterMapped);
  if (e != cudaSuccess) {
    set_last_cuda_error((int)e);
    set_error_text("cudaHostRegister of the host pool");
    cudaGetLastError();
    munmap(p, len);
    return e == cudaErrorMemoryAllocation ? KVX_ENOMEM : KVX_ECUDA;
  }
  {
    std::lock_guard<std::mutex> g(g_mu);
    g_mappings[p] = len;
  }
  *out = p;
  *len_out = len;
  return KVX_OK;
}

}  // namespace

extern "C" {

kvx_status kv_host_alloc_ex(int64_t bytes, int32_t numa_node, uint32_t flags, void** out, int32_t* numa_out) {
  if (!out) return KVX_EINVAL;
  *out = nullptr;
  if (numa_out) *numa_out = -1;
  if (bytes <= 0 || numa_node < KVX_NUMA_ANY || numa_node >= kMaxNodes || (flags & ~KVX_HOST_DRIVER))
    return KVX_EINVAL;
  if ((flags & KVX_HOST_DRIVER) && numa_node != KVX_NUMA_ANY) return KVX_EINVAL;
  if (fault_point("host_alloc")) {
    set_last_cuda_error((int)cudaErrorMemoryAllocation);
    set_error_text("pinning of the host pool (injected fault)");
    return KVX_ENOMEM;
  }
  // The driver's allocator where asked, and where the library's mapping would
  // get no huge pages and no placement anyway (a small pool, or no
  // transparent huge pages): its memory serves the copy engines better than
  // base pages do.
  const size_t huge = thp_available() ? huge_page_bytes() : 0;
  if ((flags & KVX_HOST_DRIVER) || (numa_node == KVX_NUMA_ANY && (huge == 0 || (size_t)bytes < huge)))
    return driver_pool(bytes, out);
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
  size_t len = 0;
  const kvx_status st = map_pool(node, bytes, out, &len);
  if (st == KVX_OK && numa_out) *numa_out = page_node(*out);
  return st;
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
  size_t len = 0;
  {
    std::lock_guard<std::mutex> g(g_mu);
    auto it = g_mappings.find(p);
    if (it == g_mappings.end()) return;  // not a pool of this library
    len = it->second;
    g_mappings.erase(it);
  }
  if (len == 0) {
    cudaFreeHost(p);
  } else {
    cudaHostUnregister(p);
    cudaGetLastError();
    munmap(p, len);
  }
  cudaGetLastError();
}

}  // extern "C"
