// host_touch.cpp -- reading the host pages of pinned chunks before a transfer
// after idle time (kv_store / kv_load) or on request (kv_host_touch).

#include <cuda_runtime.h>
#include <unistd.h>

#include <algorithm>
#include <atomic>
#include <chrono>
#include <condition_variable>
#include <deque>
#include <memory>
#include <mutex>
#include <thread>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "kvx_internal.h"

using namespace kvx;

namespace {

// On GB300 a transfer through pinned host memory that had sat untouched for
// seconds ran at half speed or less until the CPU had read the pages (one byte
// per page, 13.8 ms on one thread for 33 GB, then the restore ran at the link
// peak).  The reads run on a process-wide pool of persistent threads, started
// once, so no call creates threads.  A transfer call hands the pages to the
// pool and enqueues, ahead of its transfer on the caller's stream, a host
// function that waits until the pool has read them: the calling thread does
// not wait, the GPU moves the chunks only after their pages were read, and the
// stream cannot complete (so the caller cannot free the chunks) while the pool
// still reads them.  The reads are volatile and their values unused.

constexpr int64_t kTouchBlock = 256;                 // pages handed out at a time
constexpr int64_t kTouchBoundNs = 5000000000ll;      // a waiter gives up after 5 s

struct TouchJob {
  struct Range {
    const volatile uint8_t* p;
    int64_t bytes;
  };
  std::vector<Range> ranges;
  std::vector<int64_t> first_page;  // first page index of each range
  int64_t pages = 0, page = 4096;
  std::atomic<int64_t> next{0};     // next page index to hand out
  std::atomic<bool> cancel{false};
  std::mutex mu;
  std::condition_variable cv;
  int active = 0;                   // threads inside touch_some, under mu
};

int64_t host_page_bytes() { return std::max<int64_t>(4096, (int64_t)sysconf(_SC_PAGESIZE)); }

std::shared_ptr<TouchJob> make_touch_job(void* const* ptrs, const int64_t* bytes, int64_t n) {
  auto j = std::make_shared<TouchJob>();
  j->page = host_page_bytes();
  j->ranges.reserve((size_t)n);
  j->first_page.reserve((size_t)n);
  for (int64_t i = 0; i < n; ++i) {
    if (bytes[i] <= 0) continue;
    j->ranges.push_back({(const volatile uint8_t*)ptrs[i], bytes[i]});
    j->first_page.push_back(j->pages);
    j->pages += (bytes[i] + j->page - 1) / j->page;
  }
  return j;
}

// Reads pages of the job until none are left to hand out (or it is cancelled).
void touch_some(TouchJob& j) {
  {
    std::lock_guard<std::mutex> l(j.mu);
    ++j.active;
  }
  uint8_t sink = 0;
  for (;;) {
    if (j.cancel.load()) break;
    const int64_t b = j.next.fetch_add(kTouchBlock);
    if (b >= j.pages) break;
    const int64_t e = std::min(b + kTouchBlock, j.pages);
    size_t r = (size_t)(std::upper_bound(j.first_page.begin(), j.first_page.end(), b) - j.first_page.begin()) - 1;
    for (int64_t pg = b; pg < e; ++pg) {
      while (r + 1 < j.ranges.size() && pg >= j.first_page[r + 1]) ++r;
      sink ^= j.ranges[r].p[(pg - j.first_page[r]) * j.page];
    }
  }
  (void)sink;
  std::lock_guard<std::mutex> l(j.mu);
  if (--j.active == 0) j.cv.notify_all();
}

// Waits until every page has been read, or, after kTouchBoundNs, cancels the
// rest and waits until no thread is still reading; either way no page of the
// job is read after it returns.
void wait_touch(TouchJob& j) {
  std::unique_lock<std::mutex> l(j.mu);
  const auto finished = [&] { return j.active == 0 && (j.next.load() >= j.pages || j.cancel.load()); };
  if (!j.cv.wait_for(l, std::chrono::nanoseconds(kTouchBoundNs), finished)) {
    j.cancel.store(true);
    j.cv.wait(l, [&] { return j.active == 0; });
  }
}

// The persistent threads.  Made once per process, by the first kv_ctx_create
// (or the first kv_host_touch); a forked child (which inherits no threads)
// touches on its calling thread.
struct TouchPool {
  std::mutex mu;
  std::condition_variable cv;
  std::deque<std::shared_ptr<TouchJob>> queue;
  int threads = 0;
};
std::atomic<pid_t> g_touch_pid{0};  // process owning g_touch_pool's threads
TouchPool* g_touch_pool = nullptr;  // never freed: its threads run until exit
std::once_flag g_touch_once;

void touch_worker(TouchPool* pool) {
  for (;;) {
    std::shared_ptr<TouchJob> j;
    {
      std::unique_lock<std::mutex> l(pool->mu);
      pool->cv.wait(l, [&] { return !pool->queue.empty(); });
      j = pool->queue.front();
    }
    touch_some(*j);
    std::lock_guard<std::mutex> l(pool->mu);
    if (!pool->queue.empty() && pool->queue.front() == j) pool->queue.pop_front();  // handed out or cancelled
  }
}

TouchPool* touch_pool() {
  std::call_once(g_touch_once, [] {
    try {
      auto* pool = new TouchPool;
      const unsigned hw = std::thread::hardware_concurrency();
      const int want = (int)std::min<unsigned>(16, hw > 1 ? hw - 1 : 1);
      for (int t = 0; t < want; ++t) {
        try {
          std::thread(touch_worker, pool).detach();
          pool->threads++;
        } catch (...) {
          break;  // no more threads to be had
        }
      }
      g_touch_pool = pool;
      g_touch_pid.store(getpid());
    } catch (...) {
      g_touch_pool = nullptr;
    }
  });
  return (g_touch_pool && g_touch_pool->threads > 0 && g_touch_pid.load() == getpid()) ? g_touch_pool : nullptr;
}

// Hands the job to the pool; false if there is no pool in this process.
bool submit_touch(const std::shared_ptr<TouchJob>& j) {
  TouchPool* pool = touch_pool();
  if (!pool) return false;
  {
    std::lock_guard<std::mutex> l(pool->mu);
    pool->queue.push_back(j);
  }
  pool->cv.notify_all();
  return true;
}

// Host function on the caller's stream: the transfer behind it waits for the touch.
void CUDART_CB touch_gate(void* arg) {
  auto* j = static_cast<std::shared_ptr<TouchJob>*>(arg);
  wait_touch(**j);
  delete j;
}

bool stream_capturing(cudaStream_t s) {
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &cap) != cudaSuccess) {
    cudaGetLastError();
    return true;  // unknown: take it as capturing, so nothing is added to the stream
  }
  return cap != cudaStreamCaptureStatusNone;
}

}  // namespace

namespace kvx {

void start_touch_threads() { touch_pool(); }

void touch_before_transfer(void* const* chunks, const std::vector<int32_t>& tokens, const kvx_pool* P,
                           const Geometry& g, cudaStream_t stream) {
  if (stream_capturing(stream)) return;  // a replayed host function would wait on a job long gone
  try {
    std::vector<int64_t> bytes(tokens.size());
    for (size_t i = 0; i < tokens.size(); ++i) bytes[i] = chunk_bytes(P, g, tokens[i]);
    std::shared_ptr<TouchJob> j = make_touch_job(chunks, bytes.data(), (int64_t)bytes.size());
    if (submit_touch(j)) {
      auto* arg = new std::shared_ptr<TouchJob>(j);
      if (cudaLaunchHostFunc(stream, touch_gate, arg) == cudaSuccess) return;
      cudaGetLastError();
      delete arg;
    }
    touch_some(*j);
    wait_touch(*j);
  } catch (...) {
  }
}

}  // namespace kvx

extern "C" kvx_status kv_host_touch(void* const* ptrs, const int64_t* bytes, int64_t n) {
  return guarded([&]() -> kvx_status {
    nvtxRangePushA("kv_host_touch");
    struct Pop {
      ~Pop() { nvtxRangePop(); }
    } pop;
    if (n < 0 || (n > 0 && (!ptrs || !bytes))) return KVX_EINVAL;
    for (int64_t i = 0; i < n; ++i)
      if (bytes[i] < 0 || (bytes[i] > 0 && !ptrs[i])) return KVX_EINVAL;
    std::shared_ptr<TouchJob> j = make_touch_job(ptrs, bytes, n);
    if (j->pages == 0) return KVX_OK;
    submit_touch(j);  // the pool's threads and this one share the pages
    touch_some(*j);
    wait_touch(*j);
    return KVX_OK;
  });
}
