// numa_alloc.cpp -- page-locked host pools placed on one host NUMA node.
//
// Sec. 3.3: the shared tier is one full-size pinned pool.  On a host with
// several memory nodes, that pool belongs on the node next to the GPU that
// reads and writes it; otherwise every zero-copy access also crosses the
// link between sockets.  kv_host_alloc_numa maps anonymous memory, asks the
// kernel to place it on the node (mbind, MPOL_PREFERRED: no out-of-memory
// kill if the node fills up), registers it page-locked, portable and mapped
// (which faults every page in under that policy), and reports where the
// pages landed.  The mbind and move_pages system calls are used directly;
// their constants are the kernel ABI values.

#include <cuda_runtime.h>
#include <errno.h>
#include <stdio.h>
#include <stdint.h>
#include <string.h>
#include <sys/mman.h>
#include <sys/syscall.h>
#include <unistd.h>

#include <mutex>
#include <unordered_map>

#include "kvx_internal.h"

using namespace kvx;

namespace {

constexpr int kMpolPreferred = 1;      // linux/mempolicy.h: MPOL_PREFERRED
constexpr int kMaxNodes = 1024;        // nodes a node mask below can name

std::mutex g_mu;
std::unordered_map<void*, size_t> g_mappings;  // kv_host_alloc_numa allocations: base -> mapped length

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
  int64_t kb = -1;
  while (fgets(line, sizeof(line), f)) {
    const char* p = strstr(line, "MemFree:");
    if (p && sscanf(p + 8, "%ld", &kb) == 1) break;
  }
  fclose(f);
  return kb < 0 ? -1 : kb * 1024;
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

}  // namespace

namespace kvx {
// kv_host_free's hook: true if p came from kv_host_alloc_numa (then it is freed here).
bool free_numa_allocation(void* p) {
  size_t len = 0;
  {
    std::lock_guard<std::mutex> g(g_mu);
    auto it = g_mappings.find(p);
    if (it == g_mappings.end()) return false;
    len = it->second;
    g_mappings.erase(it);
  }
  cudaHostUnregister(p);
  cudaGetLastError();
  munmap(p, len);
  return true;
}
}  // namespace kvx

extern "C" kvx_status kv_host_alloc_numa(int32_t numa_node, int64_t bytes, void** out, int32_t* numa_out) {
  if (!out) return KVX_EINVAL;
  *out = nullptr;
  if (numa_out) *numa_out = -1;
  if (bytes <= 0 || numa_node < KVX_NUMA_NEAREST || numa_node >= kMaxNodes) return KVX_EINVAL;
  int node = numa_node;
  if (node == KVX_NUMA_NEAREST) {
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
  // Pools of at least one huge page are mapped huge-page aligned and sized and
  // asked for transparent huge pages.  Measured on GB300 with a 33 GB pool:
  // mapped as the kernel chose, zero-copy store + restore ran at 95 GB/s;
  // aligned with huge pages, at 202 GB/s, the same as cudaHostAlloc memory.
  const size_t page = (size_t)sysconf(_SC_PAGESIZE);
  const size_t huge = huge_page_bytes();
  const bool use_huge = huge >= page && (size_t)bytes >= huge;
  const size_t unit = use_huge ? huge : page;
  const size_t len = ((size_t)bytes + unit - 1) / unit * unit;
  const size_t span = use_huge ? len + huge : len;  // room to align the start
  uint8_t* raw = (uint8_t*)mmap(nullptr, span, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS, -1, 0);
  if (raw == (uint8_t*)MAP_FAILED) return KVX_ENOMEM;
  void* p = raw;
  if (use_huge) {
    uint8_t* start = (uint8_t*)(((uintptr_t)raw + huge - 1) / huge * huge);
    if (start > raw) munmap(raw, (size_t)(start - raw));
    const size_t tail = (size_t)(raw + span - (start + len));
    if (tail) munmap(start + len, tail);
    p = start;
    madvise(p, len, MADV_HUGEPAGE);  // advice only: base pages if none are available
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
  if (numa_out) *numa_out = page_node(p);
  *out = p;
  return KVX_OK;
}
