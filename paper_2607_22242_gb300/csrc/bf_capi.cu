// bf_capi.cu -- the C ABI declared in include/bf.h: scenario validation, the
// device-format tables, launches and bounded waits.  All search arithmetic
// runs in the kernels (bf_kernels.cu, bf_sim.cuh); this file only marshals.
#include <cuda_runtime.h>

#include <chrono>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <thread>
#include <vector>

#include "../../include/bf.h"
#include "bf_launch.h"

struct bf_scenario {
  bf_scenario_desc desc;
  bfk::Tables tables;
  int device;
  unsigned long long* d_key;  // device scratch: one packed search key
  unsigned long long* h_key;  // pinned host copy of it
};

namespace {

thread_local std::string g_error;
uint32_t g_wait_timeout_ms = 600000;

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
  static int countdown = [] {
    const char* s = std::getenv("BF_FAIL_ALLOC");
    return s ? std::atoi(s) : 0;
  }();
  if (countdown <= 0) return false;
  return --countdown == 0;
}

cudaError_t lib_malloc(void** p, size_t bytes) {
  if (inject_alloc_failure()) return cudaErrorMemoryAllocation;
  return cudaMalloc(p, bytes);
}

cudaError_t lib_malloc_host(void** p, size_t bytes) {
  if (inject_alloc_failure()) return cudaErrorMemoryAllocation;
  return cudaMallocHost(p, bytes);
}

uint64_t pow3(uint32_t n) {
  uint64_t p = 1;
  for (uint32_t i = 0; i < n; ++i) p *= 3;
  return p;
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

void build_tables(const bf_scenario_desc* d, bfk::Tables* t) {
  std::memset(t, 0, sizeof *t);
  const uint32_t n = d->n;
  t->n = n;
  t->budget = d->vram_budget_mib;
  t->all_mask = (n == 32) ? ~0u : ((1u << n) - 1u);
  for (uint32_t v = 0; v < n; ++v) {
    t->pred[v] = d->pred_mask[v];
    for (uint32_t u = 0; u < v; ++u)
      if (d->pred_mask[v] & (1u << u)) t->succ[u] |= 1u << v;
    t->cpu[v] = d->cpu_us[v];
    t->wnow[v] = (d->gpu_us[v] + d->xfer_us[v]) * 1024u;
    t->wq[v] = (d->load_us[v] + d->gpu_us[v] + d->xfer_us[v]) * 1024u;
    t->vram[v] = d->vram_mib[v];
    if (d->vram_mib[v] > d->vram_budget_mib) t->big_mask |= 1u << v;
  }
  for (uint32_t k = 1; k <= BF_MAX_TOOLS; ++k) {
    // Entries above n are never used; fill them with f[n] so every k is defined.
    const uint32_t f = d->slowdown_q10[k <= n ? k : n];
    uint32_t l = 0;
    while ((1u << l) < f) ++l;  // ceil(log2 f)
    if (l < 12) l = 12;
    const unsigned __int128 num = (unsigned __int128)1 << (52 + l);
    t->f[k] = f;
    t->fshift[k] = l - 12;
    t->fmagic[k] = (uint64_t)((num + f - 1) / f);
  }
  t->f[0] = 1024;
  t->fmagic[0] = 1ull << 54;
}

int wait_stream(cudaStream_t st, const char* who) {
  const auto t0 = std::chrono::steady_clock::now();
  for (;;) {
    const cudaError_t e = cudaStreamQuery(st);
    if (e == cudaSuccess) return BF_OK;
    if (e != cudaErrorNotReady) return cuda_fail(e, who);
    if (g_wait_timeout_ms) {
      const auto ms = std::chrono::duration_cast<std::chrono::milliseconds>(
                          std::chrono::steady_clock::now() - t0).count();
      if (ms > (long long)g_wait_timeout_ms)
        return fail(BF_ETIMEOUT, "%s: GPU work not finished after %u ms", who, g_wait_timeout_ms);
    }
    std::this_thread::sleep_for(std::chrono::microseconds(20));
  }
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

// Consecutive mappings per thread in the search kernels: enough to amortise
// the decode and the reductions, small enough to fill every SM for mid-size N.
uint32_t search_chunk(uint64_t count) {
  if (count >= (1ull << 26)) return 64;
  if (count >= (1ull << 20)) return 16;
  return 4;
}

#define BF_DISPATCH(NT_VAL, CALL)                         \
  switch (NT_VAL) {                                       \
    case 4: { e = bfk::CALL(4); } break;                  \
    case 6: { e = bfk::CALL(6); } break;                  \
    case 8: { e = bfk::CALL(8); } break;                  \
    case 10: { e = bfk::CALL(10); } break;                \
    case 12: { e = bfk::CALL(12); } break;                \
    case 14: { e = bfk::CALL(14); } break;                \
    case 16: { e = bfk::CALL(16); } break;                \
    case 18: { e = bfk::CALL(18); } break;                \
    case 19: { e = bfk::CALL(19); } break;                \
    default: { e = bfk::CALL(20); } break;                \
  }

int run_search(const bf_scenario* scn, uint64_t first, uint64_t count, bf_result* out,
               cudaStream_t st, const char* who) {
  cudaError_t e = cudaMemsetAsync(scn->d_key, 0xFF, sizeof(unsigned long long), st);
  if (e != cudaSuccess) return cuda_fail(e, who);
  if (count) {
    const uint32_t per_thread = search_chunk(count);
#define CALL(NT) launch_search_nt##NT(scn->tables, (uint32_t)first, count, per_thread, scn->d_key, st)
    BF_DISPATCH(bfk::bucket_for(scn->desc.n), CALL)
#undef CALL
    if (e != cudaSuccess) return cuda_fail(e, who);
  }
  e = cudaMemcpyAsync(scn->h_key, scn->d_key, sizeof(unsigned long long), cudaMemcpyDeviceToHost, st);
  if (e != cudaSuccess) return cuda_fail(e, who);
  const int rc = wait_stream(st, who);
  if (rc != BF_OK) return rc;
  fill_result(*scn->h_key, scn->desc.n, first, out);
  return BF_OK;
}

}  // namespace

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
  build_tables(desc, &s->tables);
  cudaError_t e = cudaGetDevice(&s->device);
  if (e == cudaSuccess) e = lib_malloc(reinterpret_cast<void**>(&s->d_key), sizeof(unsigned long long));
  if (e == cudaSuccess) e = lib_malloc_host(reinterpret_cast<void**>(&s->h_key), sizeof(unsigned long long));
  if (e != cudaSuccess) {
    const int code = cuda_fail(e, "bf_create_scenario");
    if (s->d_key) cudaFree(s->d_key);
    delete s;
    return code;
  }
  *out = s;
  return BF_OK;
}

int bf_destroy_scenario(bf_scenario* scn) {
  if (!scn) return BF_OK;
  cudaError_t e1 = scn->d_key ? cudaFree(scn->d_key) : cudaSuccess;
  cudaError_t e2 = scn->h_key ? cudaFreeHost(scn->h_key) : cudaSuccess;
  delete scn;
  if (e1 != cudaSuccess) return cuda_fail(e1, "bf_destroy_scenario");
  if (e2 != cudaSuccess) return cuda_fail(e2, "bf_destroy_scenario");
  return BF_OK;
}

int bf_eval_mappings(const bf_scenario* scn, uint64_t first, uint64_t count, uint32_t* d_makespan,
                     uint8_t* d_feasible, void* cuda_stream) {
  if (!scn) return fail(BF_EINVAL, "bf_eval_mappings: scenario is NULL");
  const uint64_t total = pow3(scn->desc.n);
  if (first > total || count > total - first)
    return fail(BF_ERANGE, "bf_eval_mappings: [%llu, %llu+%llu) is outside [0, 3^%u)",
                (unsigned long long)first, (unsigned long long)first, (unsigned long long)count, scn->desc.n);
  if (count == 0) return BF_OK;
  if (!d_makespan || !d_feasible) return fail(BF_EINVAL, "bf_eval_mappings: NULL output buffer");
  int sms = 0;
  cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, scn->device);
  if (e != cudaSuccess) return cuda_fail(e, "bf_eval_mappings");
  const uint64_t blocks_needed = (count + bfk::kThreads - 1) / bfk::kThreads;
  const uint64_t cap = (uint64_t)sms * 16;
  const int grid = (int)(blocks_needed < cap ? blocks_needed : cap);
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
#define CALL(NT) launch_eval_nt##NT(scn->tables, (uint32_t)first, count, d_makespan, d_feasible, grid, st)
  BF_DISPATCH(bfk::bucket_for(scn->desc.n), CALL)
#undef CALL
  if (e != cudaSuccess) return cuda_fail(e, "bf_eval_mappings");
  return BF_OK;
}

int bf_search_best(const bf_scenario* scn, bf_result* out, void* cuda_stream) {
  if (!scn || !out) return fail(BF_EINVAL, "bf_search_best: NULL argument");
  return run_search(scn, 0, pow3(scn->desc.n), out, static_cast<cudaStream_t>(cuda_stream), "bf_search_best");
}

int bf_search_range(const bf_scenario* scn, uint64_t first, uint64_t count, bf_result* out,
                    void* cuda_stream) {
  if (!scn || !out) return fail(BF_EINVAL, "bf_search_range: NULL argument");
  const uint64_t total = pow3(scn->desc.n);
  if (first > total || count > total - first)
    return fail(BF_ERANGE, "bf_search_range: [%llu, %llu+%llu) is outside [0, 3^%u)",
                (unsigned long long)first, (unsigned long long)first, (unsigned long long)count, scn->desc.n);
  return run_search(scn, first, count, out, static_cast<cudaStream_t>(cuda_stream), "bf_search_range");
}

int bf_search_batch(const bf_scenario_desc* descs, uint32_t count, bf_result* out, void* cuda_stream) {
  if (count == 0) return BF_OK;
  if (!descs || !out) return fail(BF_EINVAL, "bf_search_batch: NULL argument");
  uint32_t nmax = 0;
  for (uint32_t i = 0; i < count; ++i) {
    const int rc = validate(descs + i, "bf_search_batch");
    if (rc != BF_OK) return fail(rc, "bf_search_batch: descs[%u]: %s", i, g_error.c_str());
    if (descs[i].n > nmax) nmax = descs[i].n;
  }
  std::vector<bfk::Tables> tables(count);
  for (uint32_t i = 0; i < count; ++i) build_tables(descs + i, &tables[i]);
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  bfk::Tables* d_tables = nullptr;
  unsigned long long* d_keys = nullptr;
  std::vector<unsigned long long> keys(count);
  const size_t tbytes = sizeof(bfk::Tables) * count, kbytes = sizeof(unsigned long long) * count;
  cudaError_t e = lib_malloc(reinterpret_cast<void**>(&d_tables), tbytes);
  if (e == cudaSuccess) e = lib_malloc(reinterpret_cast<void**>(&d_keys), kbytes);
  if (e == cudaSuccess) e = cudaMemcpyAsync(d_tables, tables.data(), tbytes, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(d_keys, 0xFF, kbytes, st);
  int rc = BF_OK;
  if (e == cudaSuccess) {
    const uint64_t per_scn = pow3(nmax);
    const uint32_t per_thread = per_scn >= 8192 ? 32 : 4;
    const uint64_t threads = (per_scn + per_thread - 1) / per_thread;
    const uint32_t bps = (uint32_t)((threads + bfk::kThreads - 1) / bfk::kThreads);
#define CALL(NT) launch_batch_nt##NT(d_tables, count, per_thread, bps, d_keys, st)
    BF_DISPATCH(bfk::bucket_for(nmax), CALL)
#undef CALL
  }
  if (e == cudaSuccess) e = cudaMemcpyAsync(keys.data(), d_keys, kbytes, cudaMemcpyDeviceToHost, st);
  if (e != cudaSuccess) rc = cuda_fail(e, "bf_search_batch");
  if (rc == BF_OK) rc = wait_stream(st, "bf_search_batch");
  if (rc != BF_ETIMEOUT) {  // on timeout the kernel may still use the scratch: leak it rather than free in-use memory
    if (d_tables) cudaFree(d_tables);
    if (d_keys) cudaFree(d_keys);
  }
  if (rc != BF_OK) return rc;
  for (uint32_t i = 0; i < count; ++i) fill_result(keys[i], descs[i].n, 0, out + i);
  return BF_OK;
}

void bf_set_wait_timeout_ms(uint32_t ms) { g_wait_timeout_ms = ms; }

const char* bf_last_error(void) { return g_error.c_str(); }

const char* bf_version(void) { return "bf 1.0 (model v1)"; }

}  // extern "C"
