// bf_capi.cu -- the C ABI declared in include/bf.h: scenario validation, the
// device-format tables, launches and bounded waits (the tree search's host
// side is in bf_capi_tree.cu).  All search arithmetic runs in the kernels
// (bf_kernels.cu, bf_sim.cuh, bf_tree.cu); this file only marshals.
#include <cuda.h>
#include <cuda_runtime.h>
#include <unistd.h>

#include <atomic>
#include <chrono>
#include <cstdarg>
#include <cstddef>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <algorithm>
#include <condition_variable>
#include <mutex>
#include <string>
#include <thread>
#include <vector>

#include "bf_capi_internal.h"

namespace bfcapi {

using bfk::host::build_tables;
using bfk::host::make_plan;
using bfk::host::pow3;
using bfk::host::split_and_window;
using bfk::host::split_and_window_pruned;
using bfk::host::kSearchTasks;
using bfk::host::whole_space_tables;
using bfk::host::lanetree_record;

thread_local std::string g_error;
std::atomic<uint32_t> g_wait_timeout_ms{600000};

int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_error = buf;
  return code;
}

int cuda_fail(cudaError_t e, const char* what) {
  cudaGetLastError();  // clear a sticky-free error so later calls start clean
  const int code = (e == cudaErrorMemoryAllocation) ? BF_ENOMEM : BF_ECUDA;
  return fail(code, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

// Allocation-failure injection for host-side fault tests: BF_FAIL_ALLOC=<n>
// makes the n-th library allocation of the process (1-based) fail.
bool inject_alloc_failure() {
  static std::atomic<int> countdown{[] {
    const char* s = std::getenv("BF_FAIL_ALLOC");
    return s ? std::atoi(s) : 0;
  }()};
  if (countdown.load(std::memory_order_relaxed) <= 0) return false;
  return countdown.fetch_sub(1) == 1;
}

cudaError_t lib_malloc(void** p, size_t bytes) {
  if (inject_alloc_failure()) return cudaErrorMemoryAllocation;
  return cudaMalloc(p, bytes);
}

cudaError_t lib_malloc_host(void** p, size_t bytes) {
  if (inject_alloc_failure()) return cudaErrorMemoryAllocation;
  return cudaMallocHost(p, bytes);
}

// Stream-ordered device memory from the device's default pool: no device-wide
// synchronisation on free (cudaFree has one), and a free enqueued after a
// call's kernels waits for them even when the host stopped waiting.
cudaError_t lib_malloc_async(void** p, size_t bytes, cudaStream_t st) {
  if (inject_alloc_failure()) return cudaErrorMemoryAllocation;
  return cudaMallocAsync(p, bytes, st);
}

int validate(const bf_scenario_desc* d, const char* who) {
  if (!d) return fail(BF_EINVAL, "%s: desc is NULL", who);
  const uint32_t n = d->n;
  if (n < 1 || n > BF_MAX_TOOLS) return fail(BF_EINVAL, "%s: n=%u outside 1..%d", who, n, BF_MAX_TOOLS);
  for (uint32_t v = 0; v < n; ++v) {
    const uint32_t below = (v == 0) ? 0u : ((1u << v) - 1u);
    if (d->pred_mask[v] & ~below)
      return fail(BF_EINVAL, "%s: pred_mask[%u]=0x%x has an edge u->%u with u >= %u (tools must be topologically numbered)",
                  who, v, d->pred_mask[v], v, v);
    if (d->cpu_us[v] < 1) return fail(BF_EINVAL, "%s: cpu_us[%u] must be >= 1", who, v);
    if (d->gpu_us[v] < 1) return fail(BF_EINVAL, "%s: gpu_us[%u] must be >= 1", who, v);
    const uint64_t w = (uint64_t)d->load_us[v] + d->gpu_us[v] + d->xfer_us[v];
    if (w >= (1ull << 22))
      return fail(BF_EINVAL, "%s: load_us+gpu_us+xfer_us of tool %u is %llu, must be < 2^22", who, v,
                  (unsigned long long)w);
    if (d->vram_mib[v] > (1u << 27)) return fail(BF_EINVAL, "%s: vram_mib[%u] > 2^27", who, v);
  }
  if (d->vram_budget_mib > (1u << 31)) return fail(BF_EINVAL, "%s: vram_budget_mib > 2^31", who);
  if (d->slowdown_q10[1] != 1024) return fail(BF_EINVAL, "%s: slowdown_q10[1] must be 1024", who);
  for (uint32_t k = 2; k <= n; ++k) {
    if (d->slowdown_q10[k] < d->slowdown_q10[k - 1])
      return fail(BF_EINVAL, "%s: slowdown_q10 decreases at k=%u", who, k);
    if (d->slowdown_q10[k] > 65536) return fail(BF_EINVAL, "%s: slowdown_q10[%u] > 65536", who, k);
  }
  // Every tool runs at most max(c, floor((l+g+x) f[n] / 1024) + n + 1) us,
  // and at every instant before the end some tool runs, so the sum bounds
  // every makespan.
  uint64_t bound = 0;
  for (uint32_t v = 0; v < n; ++v) {
    const uint64_t w = (uint64_t)d->load_us[v] + d->gpu_us[v] + d->xfer_us[v];
    const uint64_t gpu_bound = w * d->slowdown_q10[n] / 1024 + n + 1;
    bound += d->cpu_us[v] > gpu_bound ? d->cpu_us[v] : gpu_bound;
  }
  if (bound > 0xFFFFFFFDull)
    return fail(BF_EINVAL, "%s: makespan bound %llu does not fit in 32 bits", who, (unsigned long long)bound);
  return BF_OK;
}

uint32_t wait_limit_ms() { return g_wait_timeout_ms.load(std::memory_order_relaxed); }

int wait_stream(cudaStream_t st, const char* who) {
  const auto t0 = std::chrono::steady_clock::now();
  for (uint32_t polls = 0;; ++polls) {
    const cudaError_t e = cudaStreamQuery(st);
    if (e == cudaSuccess) return BF_OK;
    if (e != cudaErrorNotReady) return cuda_fail(e, who);
    const auto us = std::chrono::duration_cast<std::chrono::microseconds>(std::chrono::steady_clock::now() - t0).count();
    const uint32_t limit = g_wait_timeout_ms.load(std::memory_order_relaxed);
    if (limit && us > 1000LL * limit) return fail(BF_ETIMEOUT, "%s: GPU work not finished after %u ms", who, limit);
    // The first 5 ms are polled without sleeping: a sleep of 20 us lasts about
    // 75 us on Linux, which would add up to that much to every search of a
    // millisecond or two.  Longer waits sleep 20 us between polls.
    if (us > 5000) std::this_thread::sleep_for(std::chrono::microseconds(20));
  }
}

// A handle's scratch lives on the device that was current at creation; its
// calls must run there.
int check_device(const bf_scenario* scn, const char* who) {
  int dev = -1;
  const cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, who);
  if (dev != scn->device)
    return fail(BF_EINVAL, "%s: the scenario was created on device %d but device %d is current", who, scn->device,
                dev);
  return BF_OK;
}

// The entry points that enumerate index ranges hold indices in 32 bits.
int require_enum(const bf_scenario_desc& d, const char* who) {
  if (d.n > BF_MAX_TOOLS_ENUM)
    return fail(BF_EINVAL, "%s: n=%u; full enumeration takes n <= %d (3^n < 2^32)", who, d.n, BF_MAX_TOOLS_ENUM);
  return BF_OK;
}

void fill_result(unsigned long long key, uint32_t n, uint64_t first, bf_result* out) {
  std::memset(out, 0, sizeof *out);
  const uint32_t ms = (uint32_t)(key >> 32);
  if (key == ~0ull || ms == 0xFFFFFFFFu) {
    out->index = first;
    out->makespan_us = 0xFFFFFFFFu;
    out->feasible = 0;
    return;
  }
  out->index = key & 0xFFFFFFFFull;
  out->makespan_us = ms;
  out->feasible = 1;
  uint64_t idx = out->index;
  for (uint32_t i = 0; i < n; ++i) {
    out->mode[i] = (uint8_t)(idx % 3);
    idx /= 3;
  }
}

// One case per compiled window width (BF_FOR_EACH_BUCKET); CALL(NW) is a
// macro defined at the use site.  Every bucket_for value has a case.
#define BF_DISPATCH_CASE(NW) \
  case NW: {                 \
    e = bfk::CALL(NW);       \
  } break;
#define BF_DISPATCH(NT_VAL, CALL)                  \
  switch (NT_VAL) {                                \
    BF_FOR_EACH_BUCKET(BF_DISPATCH_CASE)           \
    default: { e = cudaErrorInvalidValue; } break; \
  }

// Worker threads for the host-side preparation of batches, started on first
// use and kept for the life of the process: starting 16 threads on every
// call cost more than the work itself (1.3 of 1.4 ms for 4096 scenarios on a
// 16-core Grace).  One job at a time; a caller that finds the pool busy does
// its job on its own thread.  A job returns only after every worker has
// finished with it, so no worker still holds it afterwards.
class HostPool {
 public:
  static HostPool* get() {
    static HostPool* pool = [] {
      HostPool* p = new (std::nothrow) HostPool;  // never destroyed: its threads live until exit
      if (p && p->workers_ == 0) {
        delete p;
        p = nullptr;
      }
      return p;
    }();
    return pool;
  }

  // Run job(part) for every part in [0, nparts) on the workers and the
  // calling thread.  False (nothing run) if another job holds the pool.
  template <typename Job>
  bool try_run(uint32_t nparts, Job& job) {
    if (getpid() != pid_) return false;  // a forked child has no workers
    std::unique_lock<std::mutex> one(run_mu_, std::try_to_lock);
    if (!one.owns_lock()) return false;
    struct Thunk {
      static void call(void* j, uint32_t part) { (*static_cast<Job*>(j))(part); }
    };
    {
      std::lock_guard<std::mutex> lk(mu_);
      job_ = &job;
      call_ = &Thunk::call;
      nparts_ = nparts;
      next_.store(0, std::memory_order_relaxed);
      finished_ = 0;
      ++generation_;
    }
    cv_.notify_all();
    for (uint32_t part; (part = next_.fetch_add(1)) < nparts;) job(part);
    std::unique_lock<std::mutex> lk(mu_);
    done_cv_.wait(lk, [&] { return finished_ == workers_; });
    return true;
  }

 private:
  HostPool() : pid_(getpid()) {
    unsigned hw = std::thread::hardware_concurrency();
    const unsigned want = hw > 1 ? (hw - 1 < 15 ? hw - 1 : 15) : 0;
    for (unsigned t = 0; t < want; ++t) {
      try {
        std::thread(&HostPool::work, this).detach();
        ++workers_;
      } catch (const std::exception&) {
        break;
      }
    }
  }

  void work() {
    uint64_t seen = 0;
    for (;;) {
      std::unique_lock<std::mutex> lk(mu_);
      cv_.wait(lk, [&] { return generation_ != seen; });
      seen = generation_;
      void* job = job_;
      void (*call)(void*, uint32_t) = call_;
      const uint32_t nparts = nparts_;
      lk.unlock();
      for (uint32_t part; (part = next_.fetch_add(1)) < nparts;) call(job, part);
      lk.lock();
      if (++finished_ == workers_) done_cv_.notify_one();
    }
  }

  const pid_t pid_;    // the process whose threads these are
  std::mutex run_mu_;  // held by the caller of the current job
  std::mutex mu_;
  std::condition_variable cv_, done_cv_;
  uint64_t generation_ = 0;
  void* job_ = nullptr;
  void (*call_)(void*, uint32_t) = nullptr;
  uint32_t nparts_ = 0;
  std::atomic<uint32_t> next_{0};
  uint32_t workers_ = 0, finished_ = 0;
};

// Run work(lo, hi, &parts[t]) over [0, count) in up to 16 parts (one per 32
// scenarios or more: a record takes about 2 us on the Arm host, a dispatch to
// the pool some tens of us) on the host pool; parts gets one entry per part.
template <typename Part, typename Work>
void parallel_parts(uint32_t count, std::vector<Part>& parts, Work work) {
  uint32_t nparts = count / 32u;
  if (nparts > 16u) nparts = 16u;
  parts.assign(nparts > 1 ? nparts : 1, Part{});
  if (nparts > 1) {
    auto job = [&](uint32_t t) {
      work((uint32_t)((uint64_t)count * t / nparts), (uint32_t)((uint64_t)count * (t + 1) / nparts), &parts[t]);
    };
    HostPool* pool = HostPool::get();
    if (pool && pool->try_run(nparts, job)) return;
    parts.assign(1, Part{});
  }
  work(0u, count, &parts[0]);
}

// The lowest position in descs[0, count) whose desc a batch cannot search
// (invalid, or n > BF_MAX_TOOLS_ENUM), checked on the host pool; 0xFFFFFFFF
// if none.  A failed check on a pool thread writes that thread's error text
// only: the caller checks that desc again to report it.
uint32_t first_invalid(const bf_scenario_desc* descs, uint32_t count) {
  struct Part {
    uint32_t bad = 0xFFFFFFFFu;
  };
  std::vector<Part> parts;
  parallel_parts(count, parts, [&](uint32_t lo, uint32_t hi, Part* part) {
    for (uint32_t i = lo; i < hi && part->bad == 0xFFFFFFFFu; ++i) {
      bool ok = false;
      try {  // a failed check formats its message, which may allocate; no exception leaves a pool thread
        ok = validate(descs + i, "bf_search_batch") == BF_OK && require_enum(descs[i], "bf_search_batch") == BF_OK;
      } catch (...) {
      }
      if (!ok) part->bad = i;
    }
  });
  uint32_t bad = 0xFFFFFFFFu;
  for (const Part& p : parts) bad = p.bad < bad ? p.bad : bad;
  return bad;
}

// Lane-tree records of descs[ids[j]], j < count.
void build_lanetree_records(const bf_scenario_desc* descs, const uint32_t* ids, uint32_t count,
                            bfk::LaneTreeRecord* recs) {
  struct Part {};
  std::vector<Part> parts;
  parallel_parts(count, parts, [&](uint32_t lo, uint32_t hi, Part*) {
    for (uint32_t j = lo; j < hi; ++j) lanetree_record(descs + ids[j], recs + j);
  });
}

inline size_t align256(size_t x) { return (x + 255) / 256 * 256; }

// Index-list evaluation: the 20-slot kernels up to 20 tools, the 32-slot one above.
cudaError_t launch_list(const bf_scenario* scn, const uint64_t* idx, uint64_t count, uint32_t* ms, uint8_t* fe,
                        int grid, cudaStream_t st) {
  const uint32_t n = scn->desc.n;
  const uint64_t total = pow3(n);
  if (n > BF_MAX_TOOLS_ENUM) return bfk::launch_wide_list(scn->wide, total, idx, count, ms, fe, grid, st);
  cudaError_t e = cudaSuccess;
#define CALL(NW) launch_list_nw##NW(scn->tables, total, idx, count, ms, fe, grid, st)
  BF_DISPATCH(bfk::bucket_for(n), CALL)
#undef CALL
  return e;
}

// One launch of the search kernel -- or, for the whole space of a scenario
// with a lane-tree record, of the lane-tree kernel; its last block writes
// the best key into the host mirror (scn->h_scratch->search.key) and resets
// the launch state.
int run_search(const bf_scenario* scn, uint64_t first, uint64_t count, bf_result* out,
               cudaStream_t st, const char* who) {
  if (count == 0) {
    fill_result(~0ull, scn->desc.n, first, out);
    return BF_OK;
  }
  // The whole space runs on the renumbered tables; a part of it keeps the
  // scenario's numbering, in which an index range is a box of the split.
  const bool whole = first == 0 && count == pow3(scn->desc.n);
  if (whole && scn->lanetree) {
    const cudaError_t e = bfk::launch_lanetree_single(&scn->d_scratch->lt, scn->desc.n, scn->lt_x, scn->lt_blocks,
                                                      &scn->d_scratch->search, scn->d_host_search_key, st);
    if (e != cudaSuccess) return cuda_fail(e, who);
    const int rc = wait_stream(st, who);
    if (rc != BF_OK) return rc;
    fill_result(*static_cast<volatile unsigned long long*>(&scn->h_scratch->search.key), scn->desc.n, first, out);
    return BF_OK;
  }
  const bfk::Tables& tb = whole ? scn->rtables : scn->tables;
  const bfk::Tables& tw = whole ? scn->rwindow : scn->window;
  const bfk::Plan plan = make_plan(whole ? scn->rplan : scn->plan, first, count, kSearchTasks);
  cudaError_t e = cudaSuccess;
#define CALL(NW) launch_search_nw##NW(tb, tw, plan, &scn->d_scratch->search, scn->d_host_search_key, st)
  BF_DISPATCH(bfk::bucket_for(tw.n), CALL)
#undef CALL
  if (e != cudaSuccess) return cuda_fail(e, who);
  const int rc = wait_stream(st, who);
  if (rc != BF_OK) return rc;
  fill_result(*static_cast<volatile unsigned long long*>(&scn->h_scratch->search.key), scn->desc.n, first, out);
  return BF_OK;
}

}  // namespace bfcapi

using namespace bfcapi;

extern "C" {

int bf_validate_desc(const bf_scenario_desc* desc) { return validate(desc, "bf_validate_desc"); }

int bf_create_scenario(const bf_scenario_desc* desc, bf_scenario** out) {
  if (!out) return fail(BF_EINVAL, "bf_create_scenario: out is NULL");
  const int rc = validate(desc, "bf_create_scenario");
  if (rc != BF_OK) return rc;
  bf_scenario* s = new (std::nothrow) bf_scenario;
  if (!s) return fail(BF_ENOMEM, "bf_create_scenario: host allocation failed");
  std::memset(s, 0, sizeof *s);
  s->desc = *desc;
  build_tables(desc, &s->wide);
  if (desc->n <= BF_MAX_TOOLS_ENUM) {
    build_tables(desc, &s->tables);
    split_and_window(s->tables, &s->plan, &s->window);
    whole_space_tables(s->tables, s->plan, s->window, split_and_window, &s->rtables, &s->rplan, &s->rwindow);
    split_and_window_pruned(s->rtables, &s->pplan, &s->pwindow);
  }
  cudaError_t e = cudaGetDevice(&s->device);
  bfk::LaneTreeRecord ltrec;
  if (e == cudaSuccess && desc->n >= bfk::kLtSingleMinTools && desc->n <= bfk::kLtMaxTools) {
    // Optional: if the lane-tree kernel's launch shape cannot be had, the
    // search kernel runs every search of this handle.
    if (bfk::lanetree_single_blocks(desc->n, &s->lt_blocks) != cudaSuccess) {
      cudaGetLastError();
    } else {
      double lt_events = 0.0;
      bfk::host::lanetree_record(desc, &ltrec,
                                 (uint64_t)s->lt_blocks * bfk::kLtLaunchThreads * bfk::kLtSingleRootsPerLane,
                                 &lt_events);
      s->lanetree = bfk::host::lanetree_preferred(s->rtables, s->rplan, s->rwindow, ltrec, lt_events);
      if (s->lanetree)
        bfk::host::lanetree_sampled_levels(ltrec, (uint64_t)s->lt_blocks * bfk::kLtLaunchThreads *
                                                      bfk::kLtSingleRootsPerLane,
                                           &ltrec.x, &ltrec.y);
      s->lt_x = ltrec.x;
    }
  }
  if (e == cudaSuccess) e = lib_malloc(reinterpret_cast<void**>(&s->d_scratch), sizeof(bf_scratch));
  if (e == cudaSuccess) e = lib_malloc_host(reinterpret_cast<void**>(&s->h_scratch), sizeof(bf_scratch));
  if (e != cudaSuccess) {
    const int code = cuda_fail(e, "bf_create_scenario");
    if (s->d_scratch) cudaFree(s->d_scratch);
    delete s;
    return code;
  }
  s->d_key = &s->d_scratch->key;
  s->h_key = &s->h_scratch->key;
  // The search kernel's launch state starts as (~0, 0, 0) and every launch
  // leaves it so; its result goes to the pinned host mirror, which the
  // device addresses directly.
  void* mirror = nullptr;
  e = cudaMemset(&s->d_scratch->search, 0, sizeof(bfk::SearchSync));
  if (e == cudaSuccess) e = cudaMemset(&s->d_scratch->search.key, 0xFF, sizeof(unsigned long long));
  if (e == cudaSuccess && s->lanetree)
    e = cudaMemcpy(&s->d_scratch->lt, &ltrec, sizeof ltrec, cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaHostGetDevicePointer(&mirror, s->h_scratch, 0);
  if (e != cudaSuccess) {
    const int code = cuda_fail(e, "bf_create_scenario");
    cudaFree(s->d_scratch);
    cudaFreeHost(s->h_scratch);
    delete s;
    return code;
  }
  s->d_host_search_key = &static_cast<bf_scratch*>(mirror)->search.key;
  *out = s;
  return BF_OK;
}

int bf_destroy_scenario(bf_scenario* scn) {
  if (!scn) return BF_OK;
  if (scn->d_survivors) cudaFree(scn->d_survivors);
  if (scn->d_levels) cudaFree(scn->d_levels);
  cudaError_t e1 = scn->d_scratch ? cudaFree(scn->d_scratch) : cudaSuccess;
  cudaError_t e2 = scn->h_scratch ? cudaFreeHost(scn->h_scratch) : cudaSuccess;
  delete scn;
  if (e1 != cudaSuccess) return cuda_fail(e1, "bf_destroy_scenario");
  if (e2 != cudaSuccess) return cuda_fail(e2, "bf_destroy_scenario");
  return BF_OK;
}

int bf_eval_mappings(const bf_scenario* scn, uint64_t first, uint64_t count, uint32_t* d_makespan,
                     uint8_t* d_feasible, void* cuda_stream) {
  if (!scn) return fail(BF_EINVAL, "bf_eval_mappings: scenario is NULL");
  if (require_enum(scn->desc, "bf_eval_mappings") != BF_OK) return BF_EINVAL;
  if (const int rc = check_device(scn, "bf_eval_mappings")) return rc;
  const uint64_t total = pow3(scn->desc.n);
  if (first > total || count > total - first)
    return fail(BF_ERANGE, "bf_eval_mappings: [%llu, %llu+%llu) is outside [0, 3^%u)",
                (unsigned long long)first, (unsigned long long)first, (unsigned long long)count, scn->desc.n);
  if (count == 0) return BF_OK;
  if (!d_makespan || !d_feasible) return fail(BF_EINVAL, "bf_eval_mappings: NULL output buffer");
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const bfk::Plan plan = make_plan(scn->plan, first, count, kSearchTasks);
  cudaError_t e = cudaSuccess;
#define CALL(NW) launch_eval_nw##NW(scn->tables, scn->window, plan, d_makespan, d_feasible, st)
  BF_DISPATCH(bfk::bucket_for(scn->window.n), CALL)
#undef CALL
  if (e != cudaSuccess) return cuda_fail(e, "bf_eval_mappings");
  return BF_OK;
}

int bf_search_best(const bf_scenario* scn, bf_result* out, void* cuda_stream) {
  if (!scn || !out) return fail(BF_EINVAL, "bf_search_best: NULL argument");
  if (require_enum(scn->desc, "bf_search_best") != BF_OK) return BF_EINVAL;
  if (const int rc = check_device(scn, "bf_search_best")) return rc;
  return run_search(scn, 0, pow3(scn->desc.n), out, static_cast<cudaStream_t>(cuda_stream), "bf_search_best");
}

int bf_search_range(const bf_scenario* scn, uint64_t first, uint64_t count, bf_result* out,
                    void* cuda_stream) {
  if (!scn || !out) return fail(BF_EINVAL, "bf_search_range: NULL argument");
  if (require_enum(scn->desc, "bf_search_range") != BF_OK) return BF_EINVAL;
  if (const int rc = check_device(scn, "bf_search_range")) return rc;
  const uint64_t total = pow3(scn->desc.n);
  if (first > total || count > total - first)
    return fail(BF_ERANGE, "bf_search_range: [%llu, %llu+%llu) is outside [0, 3^%u)",
                (unsigned long long)first, (unsigned long long)first, (unsigned long long)count, scn->desc.n);
  return run_search(scn, first, count, out, static_cast<cudaStream_t>(cuda_stream), "bf_search_range");
}

int bf_eval_indices(const bf_scenario* scn, const uint64_t* d_indices, uint64_t count, uint32_t* d_makespan,
                    uint8_t* d_feasible, void* cuda_stream) {
  if (!scn) return fail(BF_EINVAL, "bf_eval_indices: scenario is NULL");
  if (count == 0) return BF_OK;
  if (!d_indices || !d_makespan || !d_feasible) return fail(BF_EINVAL, "bf_eval_indices: NULL buffer");
  if (const int rc = check_device(scn, "bf_eval_indices")) return rc;
  int sms = 0;
  cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, scn->device);
  if (e != cudaSuccess) return cuda_fail(e, "bf_eval_indices");
  const uint64_t need = (count + bfk::kThreads - 1) / bfk::kThreads, cap = (uint64_t)sms * 16;
  const int grid = (int)(need < cap ? need : cap);
  e = launch_list(scn, d_indices, count, d_makespan, d_feasible, grid, static_cast<cudaStream_t>(cuda_stream));
  if (e != cudaSuccess) return cuda_fail(e, "bf_eval_indices");
  return BF_OK;
}

int bf_whatif(const bf_scenario* scn, uint64_t base_index, bf_probe* out, uint32_t capacity, uint32_t* count,
              void* cuda_stream) {
  const char* who = "bf_whatif";
  if (!scn || !out || !count) return fail(BF_EINVAL, "%s: NULL argument", who);
  if (const int rc = check_device(scn, who)) return rc;
  const uint32_t n = scn->desc.n;
  const uint64_t total = pow3(n);
  if (base_index >= total)
    return fail(BF_ERANGE, "%s: base index %llu is outside [0, 3^%u)", who, (unsigned long long)base_index, n);
  uint32_t d[BF_MAX_TOOLS];
  uint64_t p3[BF_MAX_TOOLS];
  {
    uint64_t v = base_index, p = 1;
    for (uint32_t i = 0; i < n; ++i, p *= 3) {
      d[i] = (uint32_t)(v % 3);
      v /= 3;
      p3[i] = p;
    }
  }
  // Candidates: every single-tool reprobe, then every swap that Algorithm 1
  // could run (i not on gpu_now, j on gpu_now); which swaps it runs depends on
  // the single reprobes' outcomes, so all are scored in the same launch.
  bf_scratch* h = scn->h_scratch;
  uint32_t nc = 0;
  for (uint32_t i = 0; i < n; ++i)
    for (uint32_t a = 0; a < 3; ++a)
      if (a != d[i]) h->idx[nc++] = base_index - d[i] * p3[i] + a * p3[i];
  const uint32_t n_single = nc;
  for (uint32_t i = 0; i < n; ++i) {
    if (d[i] == BF_MODE_GPU_NOW) continue;
    for (uint32_t j = 0; j < n; ++j)
      if (d[j] == BF_MODE_GPU_NOW)
        h->idx[nc++] = base_index - d[i] * p3[i] + BF_MODE_GPU_NOW * p3[i] + (BF_MODE_GPU_QUEUE - BF_MODE_GPU_NOW) * p3[j];
  }
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  bf_scratch* dv = scn->d_scratch;
  cudaError_t e = cudaMemcpyAsync(dv->idx, h->idx, sizeof(uint64_t) * nc, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = launch_list(scn, dv->idx, nc, dv->ms, dv->fe, 1 + (int)(nc / bfk::kThreads), st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(h->ms, dv->ms, sizeof(uint32_t) * nc, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(h->fe, dv->fe, nc, cudaMemcpyDeviceToHost, st);
  if (e != cudaSuccess) return cuda_fail(e, who);
  const int rc = wait_stream(st, who);
  if (rc != BF_OK) return rc;
  // Assemble in Algorithm 1's order.
  uint32_t k = 0, c = 0, sw = n_single;
  bf_probe probes[BF_MAX_PROBES];
  for (uint32_t i = 0; i < n; ++i) {
    const uint32_t first_swap = sw;
    uint32_t n_now = 0;
    for (uint32_t j = 0; j < n; ++j) n_now += (d[j] == BF_MODE_GPU_NOW);
    if (d[i] != BF_MODE_GPU_NOW) sw += n_now;
    for (uint32_t a = 0; a < 3; ++a) {
      if (a == d[i]) continue;
      bf_probe& pr = probes[k++];
      pr.index = h->idx[c];
      pr.makespan_us = h->ms[c];
      pr.feasible = h->fe[c] == 1;
      pr.kind = 0;
      pr.tool = (uint8_t)i;
      pr.mode = (uint8_t)a;
      pr.other = 0xFF;
      const bool exceed = h->fe[c] != 1;
      ++c;
      if (exceed && a == BF_MODE_GPU_NOW) {
        uint32_t s = first_swap;
        for (uint32_t j = 0; j < n; ++j) {
          if (d[j] != BF_MODE_GPU_NOW) continue;
          bf_probe& q = probes[k++];
          q.index = h->idx[s];
          q.makespan_us = h->ms[s];
          q.feasible = h->fe[s] == 1;
          q.kind = 1;
          q.tool = (uint8_t)i;
          q.mode = BF_MODE_GPU_NOW;
          q.other = (uint8_t)j;
          ++s;
        }
      }
    }
  }
  if (k > capacity) return fail(BF_EINVAL, "%s: %u probes do not fit in capacity %u", who, k, capacity);
  std::memcpy(out, probes, sizeof(bf_probe) * k);
  *count = k;
  return BF_OK;
}

int bf_search_pruned(const bf_scenario* scn_const, uint64_t hint_index, bf_result* out, void* cuda_stream) {
  const char* who = "bf_search_pruned";
  if (!scn_const || !out) return fail(BF_EINVAL, "%s: NULL argument", who);
  if (require_enum(scn_const->desc, who) != BF_OK) return BF_EINVAL;
  if (const int rc = check_device(scn_const, who)) return rc;
  // The handle's lazily allocated survivor buffer is scratch, not state.
  bf_scenario* scn = const_cast<bf_scenario*>(scn_const);
  const uint32_t n = scn->desc.n;
  const uint64_t total = pow3(n);
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  cudaError_t e = cudaSuccess;

  // 1. Incumbent: the best feasible of a few mappings (the hint, all-cpu,
  //    all-gpu_now, all-gpu_queue, each tool on its isolated-faster device).
  bf_scratch* h = scn->h_scratch;
  bf_scratch* dv = scn->d_scratch;
  uint32_t nc = 0;
  if (hint_index < total) h->idx[nc++] = hint_index;
  {
    uint64_t now = 0, que = 0, fast = 0, p = 1;
    for (uint32_t i = 0; i < n; ++i, p *= 3) {
      now += p;
      que += 2 * p;
      if (scn->tables.wnow[i] / 1024u < scn->tables.cpu[i]) fast += p;
    }
    h->idx[nc++] = 0;
    h->idx[nc++] = now;
    h->idx[nc++] = que;
    h->idx[nc++] = fast;
  }
  if (!scn->d_survivors) {
    e = lib_malloc(reinterpret_cast<void**>(&scn->d_survivors), sizeof(uint32_t) * scn->pplan.pow3P);
    if (e != cudaSuccess) return cuda_fail(e, who);
  }
  e = cudaMemcpyAsync(dv->idx, h->idx, sizeof(uint64_t) * nc, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = launch_list(scn, dv->idx, nc, dv->ms, dv->fe, 1, st);

  // 2. Keep the prefixes whose checkpoint bound does not exceed the incumbent;
  //    the filter kernel takes the incumbent from the list kernel's output and
  //    hands it back with the survivor count (one host round trip for both).
  bfk::Plan plan = make_plan(scn->pplan, 0, total, kSearchTasks);
  if (e == cudaSuccess) e = cudaMemsetAsync(&dv->survivors, 0, sizeof(uint32_t), st);
  if (e == cudaSuccess) {
#define CALL(NW)                                                                                          \
  launch_prefix_filter_nw##NW(scn->rtables, plan, dv->ms, dv->fe, nc, scn->d_survivors, &dv->survivors, \
                              &dv->pruned_bound, st)
    BF_DISPATCH(bfk::bucket_for(scn->pwindow.n), CALL)
#undef CALL
  }
  static_assert(offsetof(bf_scratch, pruned_bound) == offsetof(bf_scratch, survivors) + sizeof(uint32_t),
                "survivors and pruned_bound are copied together");
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(&h->survivors, &dv->survivors, 2 * sizeof(uint32_t), cudaMemcpyDeviceToHost, st);
  if (e != cudaSuccess) return cuda_fail(e, who);
  int rc = wait_stream(st, who);
  if (rc != BF_OK) return rc;
  plan.bound = h->pruned_bound;
  const uint32_t nsurv = h->survivors;
  // A weak prefix bound (no cut points in the DAG) keeps most prefixes; the
  // tree search, whose expansions bound every node with the forward
  // earliest-finish pass, then finds the same optimum faster.
  if ((uint64_t)nsurv * 64u > plan.pow3P) return bf_search_tree(scn, BF_SPACE_FULL, 0u, hint_index, out, nullptr, cuda_stream);

  // 3. Full enumeration of the survivors' mappings, bound applied again at the
  //    inner checkpoint; tasks of at least 16 mid combinations, about
  //    kSearchTasks of them.
  plan.groups = (nsurv + 31u) / 32u;
  e = cudaMemsetAsync(scn->d_key, 0xFF, sizeof(unsigned long long), st);
  if (e == cudaSuccess && nsurv) {
    const uint64_t num_m = (uint64_t)plan.m_hi - plan.m_lo + 1;
    uint64_t parts = (kSearchTasks + plan.groups - 1) / plan.groups;
    const uint64_t min_chunk = num_m < 16 ? num_m : 16;
    const uint64_t max_parts = (num_m + min_chunk - 1) / min_chunk;
    if (parts > max_parts) parts = max_parts;
    if (parts < 1) parts = 1;
    plan.m_chunk = (uint32_t)((num_m + parts - 1) / parts);
    plan.m_parts = (uint32_t)((num_m + plan.m_chunk - 1) / plan.m_chunk);
#define CALL(NW) launch_pruned_search_nw##NW(scn->rtables, scn->pwindow, plan, scn->d_survivors, nsurv, scn->d_key, st)
    BF_DISPATCH(bfk::bucket_for(scn->pwindow.n), CALL)
#undef CALL
  }
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(scn->h_key, scn->d_key, sizeof(unsigned long long), cudaMemcpyDeviceToHost, st);
  if (e != cudaSuccess) return cuda_fail(e, who);
  rc = wait_stream(st, who);
  if (rc != BF_OK) return rc;
  fill_result(*scn->h_key, n, 0, out);
  return BF_OK;
}

// A batch runs on the lane-tree batch kernel in up to three groups, one per
// table form: up to kLtBatchTools tools, up to kLtNarrowTools, up to
// kLtMaxTools (a 14-tool layered batch scenario ran on the prefix/mid/inner
// batch kernel before; the no-alloc entry point still takes that kernel above
// kLtBatchTools).  Batches of at least kBatchPipelineMin scenarios of the
// first group are pipelined: the first eighth of that group is built, copied
// and launched on the caller's stream, and the rest of the batch is built
// while that kernel runs and launched on a second stream (created for the
// call) that waits only for the key reset, so that the kernels overlap; the
// caller's stream waits for the second before the keys come back.  4096 x
// 3^10: the kernel otherwise waits about 0.5 ms for the records.
constexpr uint32_t kBatchPipelineMin = 1024;
constexpr uint32_t kBatchGroups = 3;

inline uint32_t batch_group(uint32_t n) {
  return n <= bfk::kLtBatchTools ? 0u : (n <= bfk::kLtNarrowTools ? 1u : 2u);
}

static int search_batch_impl(const bf_scenario_desc* descs, uint32_t count, bf_result* out, void* cuda_stream) {
  if (count == 0) return BF_OK;
  if (!descs || !out) return fail(BF_EINVAL, "bf_search_batch: NULL argument");
  const uint32_t bad = first_invalid(descs, count);
  if (bad != 0xFFFFFFFFu) {
    int rc = validate(descs + bad, "bf_search_batch");
    if (rc == BF_OK) rc = require_enum(descs[bad], "bf_search_batch");
    return fail(rc == BF_OK ? BF_EINVAL : rc, "bf_search_batch: descs[%u]: %s", bad, g_error.c_str());
  }
  // Positions ordered by group, each group in the batch's order; key j and
  // record j belong to position ids[j].
  uint32_t gcount[kBatchGroups] = {}, gnmax[kBatchGroups] = {};
  for (uint32_t i = 0; i < count; ++i) ++gcount[batch_group(descs[i].n)];
  std::vector<uint32_t> ids(count);
  uint32_t fill[kBatchGroups] = {0u, gcount[0], gcount[0] + gcount[1]};
  for (uint32_t i = 0; i < count; ++i) {
    const uint32_t g = batch_group(descs[i].n);
    ids[fill[g]++] = i;
    gnmax[g] = descs[i].n > gnmax[g] ? descs[i].n : gnmax[g];
  }
  const bool pipe = gcount[0] >= kBatchPipelineMin;
  const uint32_t k1 = pipe ? gcount[0] / 8u : gcount[0];
  // Launch l covers positions [lb[l], lb[l + 1]): the first part of group 0,
  // the rest of it, group 1, group 2; its first-block array has
  // lb[l + 1] - lb[l] + 1 entries at fb[lb[l] + l].
  const uint32_t lb[5] = {0u, k1, gcount[0], gcount[0] + gcount[1], count};
  const uint32_t lnmax[4] = {gnmax[0], gnmax[0], gnmax[1], gnmax[2]};
  // Record buffers of the calling thread, grown as needed and reused: a
  // fresh 2.8 MB array (4096 scenarios) cost about 0.4 ms of zeroing and page
  // faults per call.  Every record is written whole before it is copied; a
  // copy from pageable memory has read it by the time cudaMemcpyAsync
  // returns, so the next call may reuse the buffers even after a timeout.
  thread_local std::vector<bfk::LaneTreeRecord> lt;
  if (lt.size() < count) lt.resize(count);
  std::vector<uint32_t> fb(count + 4, 0u);
  auto build = [&](uint32_t l0, uint32_t l1) {  // records and first blocks of launches [l0, l1)
    build_lanetree_records(descs, ids.data() + lb[l0], lb[l1] - lb[l0], lt.data() + lb[l0]);
    for (uint32_t l = l0; l < l1; ++l) {
      uint32_t* f = fb.data() + lb[l] + l;
      for (uint32_t j = lb[l]; j < lb[l + 1]; ++j) f[j - lb[l] + 1] = f[j - lb[l]] + lt[j].nblocks;
    }
  };
  build(0, 1);

  // One device allocation: records, first-block arrays, keys.
  const size_t lt_bytes = sizeof(bfk::LaneTreeRecord) * count, fb_bytes = sizeof(uint32_t) * fb.size();
  const size_t kbytes = sizeof(unsigned long long) * count;
  const size_t off_fb = align256(lt_bytes), off_keys = off_fb + align256(fb_bytes);
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  cudaStream_t rest = st;  // stream of the later launches
  cudaEvent_t reset_done = nullptr, rest_done = nullptr;
  unsigned char* d_base = nullptr;
  std::vector<unsigned long long> keys(count);
  cudaError_t e = lib_malloc_async(reinterpret_cast<void**>(&d_base), off_keys + kbytes, st);
  auto* d_lt = reinterpret_cast<bfk::LaneTreeRecord*>(d_base);
  auto* d_fb = reinterpret_cast<uint32_t*>(d_base + off_fb);
  auto* d_keys = reinterpret_cast<unsigned long long*>(d_base + off_keys);
  auto launch = [&](uint32_t l, cudaStream_t s) {
    const uint32_t c = lb[l + 1] - lb[l];
    if (c == 0) return cudaSuccess;
    const uint32_t* f = fb.data() + lb[l] + l;
    return bfk::launch_lanetree(d_lt + lb[l], d_fb + lb[l] + l, c, f[c], lnmax[l], d_keys + lb[l], s);
  };
  if (e == cudaSuccess && pipe) {
    e = cudaStreamCreateWithFlags(&rest, cudaStreamNonBlocking);
    if (e != cudaSuccess) rest = st;
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&reset_done, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&rest_done, cudaEventDisableTiming);
  }
  if (e == cudaSuccess && k1) e = cudaMemcpyAsync(d_lt, lt.data(), sizeof(bfk::LaneTreeRecord) * k1, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess && k1) e = cudaMemcpyAsync(d_fb, fb.data(), sizeof(uint32_t) * (k1 + 1), cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(d_keys, 0xFF, kbytes, st);
  if (e == cudaSuccess && rest != st) e = cudaEventRecord(reset_done, st);
  if (e == cudaSuccess) e = launch(0, st);
  bool rest_used = false;  // work enqueued on `rest` that the caller's stream must wait for
  if (e == cudaSuccess && count > k1) {
    build(1, 4);  // the other records, built while the first launch runs
    if (rest != st) {
      e = cudaStreamWaitEvent(rest, reset_done, 0);
      rest_used = e == cudaSuccess;
    }
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(d_lt + k1, lt.data() + k1, sizeof(bfk::LaneTreeRecord) * (count - k1),
                          cudaMemcpyHostToDevice, rest);
    if (e == cudaSuccess)  // first blocks of launches 1 to 3
      e = cudaMemcpyAsync(d_fb + k1 + 1, fb.data() + k1 + 1, sizeof(uint32_t) * (fb.size() - k1 - 1),
                          cudaMemcpyHostToDevice, rest);
    for (uint32_t l = 1; l < 4 && e == cudaSuccess; ++l) e = launch(l, rest);
  }
  // The caller's stream waits for the later launches (also after an error,
  // before the scratch is freed there); if that cannot be enqueued, the host
  // waits for them.
  if (rest_used) {
    cudaError_t ew = cudaEventRecord(rest_done, rest);
    if (ew == cudaSuccess) ew = cudaStreamWaitEvent(st, rest_done, 0);
    if (ew != cudaSuccess) {
      cudaStreamSynchronize(rest);
      if (e == cudaSuccess) e = ew;
    }
  }
  int rc = BF_OK;
  if (e != cudaSuccess) rc = cuda_fail(e, "bf_search_batch");
  // Bounded wait first: a copy into pageable memory would block without limit.
  if (rc == BF_OK) rc = wait_stream(st, "bf_search_batch");
  if (rc == BF_OK) e = cudaMemcpyAsync(keys.data(), d_keys, kbytes, cudaMemcpyDeviceToHost, st);
  // Ordered after the kernels and the copy, also when the wait timed out.
  if (d_base) {
    const cudaError_t ef = cudaFreeAsync(d_base, st);
    if (e == cudaSuccess) e = ef;
  }
  if (rc == BF_OK) {
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) rc = cuda_fail(e, "bf_search_batch");
  }
  // Released once their work is done (destroying a stream or an event with
  // work pending does not wait).
  if (rest != st) cudaStreamDestroy(rest);
  if (reset_done) cudaEventDestroy(reset_done);
  if (rest_done) cudaEventDestroy(rest_done);
  if (rc != BF_OK) return rc;
  for (uint32_t j = 0; j < count; ++j) fill_result(keys[j], descs[ids[j]].n, 0, out + ids[j]);
  return BF_OK;
}

// ---------------------------------------------------------------------------
// bf_search_batch_noalloc: the batched search with no allocation at all.
//
// Its scratch (the packed per-scenario records and one result key per
// scenario) lives in the file-scope device array below instead of memory
// obtained from cudaMalloc.  The array is part of this library's module, so
// every GPU that loads the library holds it until the process exits.
// ---------------------------------------------------------------------------
}  // extern "C"

namespace {

// Regions of the array: lane-tree records, the first-block arrays of the
// groups' launches (one entry more per group), keys; each sized for
// BF_NOALLOC_MAX_SCENARIOS scenarios.
constexpr size_t kNoAllocFirstBlockOffset =
    (sizeof(bfk::LaneTreeRecord) * BF_NOALLOC_MAX_SCENARIOS + 255) / 256 * 256;
constexpr size_t kNoAllocKeyOffset =
    kNoAllocFirstBlockOffset + (sizeof(uint32_t) * (BF_NOALLOC_MAX_SCENARIOS + kBatchGroups) + 255) / 256 * 256;
constexpr size_t kNoAllocBytes = kNoAllocKeyOffset + sizeof(unsigned long long) * BF_NOALLOC_MAX_SCENARIOS;

}  // namespace

static __device__ __align__(256) unsigned char bf_noalloc_scratch[kNoAllocBytes];

namespace {

constexpr int kNoAllocMaxDevices = 64;

// Per-device bookkeeping of the array.  `base` is its device address, resolved
// with that device current in the context whose ID is `ctx_id` (a device reset
// destroys the context and the module with it, so a new context resolves the
// address again).  `pending` is set when a call returned BF_ETIMEOUT: its
// kernel may still be reading the array on `pending_stream`, so the next call
// waits for that stream before reusing the array.  `mu` serialises the calls
// on one device: they all share the one array.
struct NoAllocDevice {
  std::mutex mu;
  unsigned long long ctx_id = 0;
  unsigned char* base = nullptr;
  bool pending = false;
  cudaStream_t pending_stream = nullptr;
};
NoAllocDevice g_noalloc[kNoAllocMaxDevices];

// The driver's cuCtxGetCurrent and cuCtxGetId, looked up through the runtime
// (the library links no driver library).
using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);
struct CtxFns {
  CtxGetCurrentFn get_current = nullptr;
  CtxGetIdFn get_id = nullptr;
};

const CtxFns& ctx_fns() {
  static const CtxFns fns = [] {
    CtxFns f;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      f.get_current = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      f.get_id = reinterpret_cast<CtxGetIdFn>(p);
    return f;
  }();
  return fns;
}

// ID of the current context, 0 when none is current yet.
int current_ctx_id(unsigned long long* id, const char* who) {
  const CtxFns& f = ctx_fns();
  if (!f.get_current || !f.get_id) return fail(BF_ECUDA, "%s: cuCtxGetCurrent/cuCtxGetId not available", who);
  CUcontext ctx = nullptr;
  if (f.get_current(&ctx) != CUDA_SUCCESS) return fail(BF_ECUDA, "%s: cuCtxGetCurrent failed", who);
  *id = 0;
  if (ctx && f.get_id(ctx, id) != CUDA_SUCCESS) return fail(BF_ECUDA, "%s: cuCtxGetId failed", who);
  return BF_OK;
}

// Set-up of the current device, done by the first call on it (and again in a
// new context after a device reset): the device address of bf_noalloc_scratch.
// In host code the array's name only stands in for it.  Called with the
// device's lock held.
int noalloc_setup(NoAllocDevice& d, const char* who) {
  unsigned long long id = 0;
  int rc = current_ctx_id(&id, who);
  if (rc != BF_OK) return rc;
  if (id != 0 && id == d.ctx_id) return BF_OK;
  void* addr = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&addr, bf_noalloc_scratch);  // creates the context if needed
  if (e != cudaSuccess) return cuda_fail(e, who);
  rc = current_ctx_id(&id, who);
  if (rc != BF_OK) return rc;
  d.base = static_cast<unsigned char*>(addr);
  d.ctx_id = id;
  d.pending = false;  // work of an earlier context ended with it
  return BF_OK;
}

int search_batch_noalloc_locked(NoAllocDevice& dv, const bf_scenario_desc* descs, uint32_t count, bf_result* out,
                                cudaStream_t st, const char* who) {
  int rc = noalloc_setup(dv, who);
  if (rc != BF_OK) return rc;
  if (dv.pending) {  // a timed-out call's kernel may still read the array
    rc = wait_stream(dv.pending_stream, who);
    if (rc == BF_ETIMEOUT)
      return fail(BF_ETIMEOUT, "%s: the kernel of an earlier call that timed out is still using the fixed scratch",
                  who);
    if (rc != BF_OK) return rc;
    dv.pending = false;
  }
  auto* d_lt = reinterpret_cast<bfk::LaneTreeRecord*>(dv.base);
  auto* d_fb = reinterpret_cast<uint32_t*>(dv.base + kNoAllocFirstBlockOffset);
  auto* d_keys = reinterpret_cast<unsigned long long*>(dv.base + kNoAllocKeyOffset);
  // Positions ordered by group (as bf_search_batch): key j and record j
  // belong to position ids[j]; group g's first-block array has gcount[g] + 1
  // entries at fb[gbeg[g] + g].
  uint32_t ids[BF_NOALLOC_MAX_SCENARIOS], fb[BF_NOALLOC_MAX_SCENARIOS + kBatchGroups];
  uint32_t gcount[kBatchGroups] = {}, gnmax[kBatchGroups] = {};
  for (uint32_t i = 0; i < count; ++i) ++gcount[batch_group(descs[i].n)];
  const uint32_t gbeg[kBatchGroups + 1] = {0u, gcount[0], gcount[0] + gcount[1], count};
  uint32_t fill[kBatchGroups] = {gbeg[0], gbeg[1], gbeg[2]};
  for (uint32_t i = 0; i < count; ++i) {
    const uint32_t g = batch_group(descs[i].n);
    ids[fill[g]++] = i;
    gnmax[g] = descs[i].n > gnmax[g] ? descs[i].n : gnmax[g];
  }

  // Pack the records a few at a time through stack buffers (a copy from
  // pageable memory has left the buffer when cudaMemcpyAsync returns).
  constexpr uint32_t kChunk = 8;
  cudaError_t e = cudaSuccess;
  {
    bfk::LaneTreeRecord chunk[kChunk];
    for (uint32_t g = 0; g < kBatchGroups; ++g) {
      uint32_t* f = fb + gbeg[g] + g;
      f[0] = 0u;
      for (uint32_t j0 = gbeg[g]; j0 < gbeg[g + 1] && e == cudaSuccess; j0 += kChunk) {
        const uint32_t nrec = (gbeg[g + 1] - j0 < kChunk) ? (gbeg[g + 1] - j0) : kChunk;
        for (uint32_t j = 0; j < nrec; ++j) {
          lanetree_record(descs + ids[j0 + j], chunk + j);
          f[j0 + j - gbeg[g] + 1] = f[j0 + j - gbeg[g]] + chunk[j].nblocks;
        }
        e = cudaMemcpyAsync(d_lt + j0, chunk, sizeof(bfk::LaneTreeRecord) * nrec, cudaMemcpyHostToDevice, st);
      }
    }
  }
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(d_fb, fb, sizeof(uint32_t) * (count + kBatchGroups), cudaMemcpyHostToDevice, st);
  // The keys keep the previous call's values: reset them to "nothing found".
  if (e == cudaSuccess) e = cudaMemsetAsync(d_keys, 0xFF, sizeof(unsigned long long) * count, st);
  for (uint32_t g = 0; g < kBatchGroups && e == cudaSuccess; ++g) {
    const uint32_t c = gbeg[g + 1] - gbeg[g];
    if (c == 0) continue;
    const uint32_t* f = fb + gbeg[g] + g;
    e = bfk::launch_lanetree(d_lt + gbeg[g], d_fb + gbeg[g] + g, c, f[c], gnmax[g], d_keys + gbeg[g], st);
  }
  if (e != cudaSuccess) return cuda_fail(e, who);
  rc = wait_stream(st, who);
  if (rc == BF_ETIMEOUT) {
    dv.pending = true;
    dv.pending_stream = st;
  }
  if (rc != BF_OK) return rc;
  constexpr uint32_t kKeyChunk = 256;
  unsigned long long keys[kKeyChunk];
  for (uint32_t i0 = 0; i0 < count; i0 += kKeyChunk) {
    const uint32_t nk = (count - i0 < kKeyChunk) ? (count - i0) : kKeyChunk;
    e = cudaMemcpyAsync(keys, d_keys + i0, sizeof(unsigned long long) * nk, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(e, who);
    for (uint32_t j = 0; j < nk; ++j) {
      const uint32_t i = ids[i0 + j];
      fill_result(keys[j], descs[i].n, 0, out + i);
    }
  }
  return BF_OK;
}

}  // namespace

extern "C" {

int bf_search_batch_noalloc(const bf_scenario_desc* descs, uint32_t count, bf_result* out, void* cuda_stream) {
  const char* who = "bf_search_batch_noalloc";
  if (count == 0) return BF_OK;
  if (!descs || !out) return fail(BF_EINVAL, "%s: NULL argument", who);
  if (count > BF_NOALLOC_MAX_SCENARIOS)
    return fail(BF_EINVAL, "%s: %u scenarios exceed this entry point's fixed scratch of %d scenarios; split the "
                "batch or use bf_search_batch", who, count, BF_NOALLOC_MAX_SCENARIOS);
  for (uint32_t i = 0; i < count; ++i) {
    int rc = validate(descs + i, who);
    if (rc == BF_OK) rc = require_enum(descs[i], who);
    if (rc != BF_OK) return fail(rc, "%s: descs[%u]: %s", who, i, g_error.c_str());
  }
  int dev = 0;
  const cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, who);
  if (dev < 0 || dev >= kNoAllocMaxDevices)
    return fail(BF_EINVAL, "%s: device %d is beyond the %d devices this entry point supports", who, dev,
                kNoAllocMaxDevices);
  NoAllocDevice& dv = g_noalloc[dev];
  std::lock_guard<std::mutex> lock(dv.mu);
  return search_batch_noalloc_locked(dv, descs, count, out, static_cast<cudaStream_t>(cuda_stream), who);
}

// Entry points that allocate host memory keep C++ exceptions inside the library.
int bf_search_batch(const bf_scenario_desc* descs, uint32_t count, bf_result* out, void* cuda_stream) {
  try {
    return search_batch_impl(descs, count, out, cuda_stream);
  } catch (const std::bad_alloc&) {
    return fail(BF_ENOMEM, "bf_search_batch: host allocation failed");
  } catch (const std::exception& ex) {
    return fail(BF_EINVAL, "bf_search_batch: %s", ex.what());
  }
}

void bf_set_wait_timeout_ms(uint32_t ms) { g_wait_timeout_ms.store(ms, std::memory_order_relaxed); }

const char* bf_last_error(void) { return g_error.c_str(); }

const char* bf_version(void) { return "bf 1.0 (model v1)"; }

}  // extern "C"
