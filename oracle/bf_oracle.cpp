// bf_oracle.cpp -- TEST INFRASTRUCTURE: the CPU oracle for the brute-force
// device-mapping search.  Only the tests, the smoke check and the benchmark's
// CPU-baseline leg may load this library.  It shares no code, header, table or
// helper with the CUDA search; it is written for obviousness, not speed.
//
// What it computes.  §2.1 states the problem: a DAG of N tool invocations, each
// mapped to one of {cpu, gpu_now, gpu_queue}; a mapping is feasible only if the
// VRAM of the GPU tools running at any instant stays within the budget M; its
// end-to-end latency is the largest completion time over the sinks; the
// brute-force oracle of §2.3 / §4.1 is the feasible mapping of lowest latency
// over all 3^N mappings.  The paper measures latencies on hardware; this oracle
// evaluates them under a fixed integer model ("bf latency model, version 1"):
//
//   * Integer microseconds for real time T; a virtual GPU-work clock V in
//     1/1024 isolated-microsecond units.  A GPU tool that starts at clock V
//     with isolated time w finishes when V reaches V + 1024*w.
//   * Factor A (§2.3, GPU utilisation contention): while k GPU tools run, each
//     progresses at 1024/f[k] of its isolated speed (processor sharing);
//     CPU tools are unaffected and CPU cores are unlimited.
//   * gpu_now (§2.1): starts as soon as its predecessors are done and holds
//     its VRAM while running; a start that takes live VRAM above M is
//     infeasible (the out-of-memory failure of Factor B, §2.3).  Work = g + x
//     (Table 1's GPU time includes the PCIe transfer).
//   * gpu_queue (§2.1, Factor B): waits in one serialised FIFO queue without
//     holding VRAM; the head starts when no queued tool is running and live
//     VRAM + its footprint <= M; work = l + g + x (Table 1's gpu_queue column
//     prices a queued run as GPU + Load).  A queued tool with m > M can never
//     start: infeasible.
//   * cpu: runs for c on its own core.
//
// The simulation below follows the model's steps in order:
//   admission at T=0; then repeat { next CPU completion; next GPU completion
//   under the current slowdown (rounded up to a whole microsecond); advance T
//   and V to the earlier one (V advanced by the floor of the elapsed work when
//   a CPU tool ends first); retire every tool that ends at that instant;
//   admission at the new T } until every tool is done.  The makespan is T at
//   the last retirement; an infeasible mapping has makespan 0xFFFFFFFF.
//
// Mapping index: idx = sum_i a_i * 3^i with a_i in {0=cpu, 1=gpu_now,
// 2=gpu_queue}; tool 0 is the least-significant digit.  The argmin compares
// (makespan, idx) lexicographically over feasible mappings, so ties go to the
// lowest index.
//
// The binary decision space (§4.1: every scenario of S1-S10 chooses between
// CPU and GPU only, 2^N mappings): mappings whose digits are all 0 or 1.  The
// b-th of them (b = sum_i b_i 2^i) is the mapping with a_i = b_i; its index
// is sum_i b_i 3^i.  The binary search below enumerates b and compares
// (makespan, idx) as above.

#include <cstdint>
#include <cstring>
#include <thread>
#include <vector>

namespace {

const int kMaxTools = 32;
const uint64_t kInfinity = UINT64_MAX;
const uint64_t kInfeasibleMakespan = 0xFFFFFFFFull;
const uint64_t kStalled = 0xFFFFFFFFFFFFFFFEull;  // never produced by a correct model

enum Mode { kCpu = 0, kGpuNow = 1, kGpuQueue = 2 };
enum Status { kPending, kWaitingInQueue, kRunning, kDone };

// The oracle's own scenario record, unpacked from a flat uint32 array:
//   [0] n, [1] M, then 32 words each of pred, c, g, x, l, m, then 33 words f.
struct OracleScenario {
  int n;
  uint64_t budget;
  uint32_t pred[kMaxTools];
  uint64_t cpu[kMaxTools], gpu[kMaxTools], xfer[kMaxTools], load[kMaxTools], vram[kMaxTools];
  uint64_t slowdown[kMaxTools + 1];
};

const int kFlatWords = 2 + 6 * kMaxTools + (kMaxTools + 1);

OracleScenario unpack(const uint32_t* w) {
  OracleScenario s;
  s.n = (int)w[0];
  s.budget = w[1];
  const uint32_t* p = w + 2;
  for (int i = 0; i < kMaxTools; ++i) s.pred[i] = p[0 * kMaxTools + i];
  for (int i = 0; i < kMaxTools; ++i) s.cpu[i] = p[1 * kMaxTools + i];
  for (int i = 0; i < kMaxTools; ++i) s.gpu[i] = p[2 * kMaxTools + i];
  for (int i = 0; i < kMaxTools; ++i) s.xfer[i] = p[3 * kMaxTools + i];
  for (int i = 0; i < kMaxTools; ++i) s.load[i] = p[4 * kMaxTools + i];
  for (int i = 0; i < kMaxTools; ++i) s.vram[i] = p[5 * kMaxTools + i];
  for (int k = 0; k <= kMaxTools; ++k) s.slowdown[k] = p[6 * kMaxTools + k];
  return s;
}

void decode_mapping(uint64_t idx, int n, int* mode) {
  for (int i = 0; i < n; ++i) {
    mode[i] = (int)(idx % 3);
    idx /= 3;
  }
}

uint64_t ceil_div(uint64_t a, uint64_t b) { return (a + b - 1) / b; }

struct Simulation {
  const OracleScenario& s;
  const int* mode;

  uint64_t T = 0;          // real time, microseconds
  uint64_t V = 0;          // virtual GPU work clock, 1/1024 isolated microseconds
  uint64_t live_vram = 0;  // MiB held by running GPU tools
  int running_gpu = 0;     // k
  bool queue_busy = false; // a queued tool is running
  bool infeasible = false;

  Status status[kMaxTools];
  uint64_t ready_time[kMaxTools];
  uint64_t cpu_end[kMaxTools];   // real end time of a running cpu tool
  uint64_t gpu_vend[kMaxTools];  // virtual end of a running GPU tool

  Simulation(const OracleScenario& sc, const int* m) : s(sc), mode(m) {
    for (int i = 0; i < kMaxTools; ++i) {
      status[i] = kPending;
      ready_time[i] = cpu_end[i] = gpu_vend[i] = 0;
    }
  }

  bool predecessors_done(int v) const {
    for (int u = 0; u < s.n; ++u)
      if (((s.pred[v] >> u) & 1u) && status[u] != kDone) return false;
    return true;
  }

  bool all_done() const {
    for (int v = 0; v < s.n; ++v)
      if (status[v] != kDone) return false;
    return true;
  }

  void start_on_gpu(int v, uint64_t isolated_us) {
    status[v] = kRunning;
    live_vram += s.vram[v];
    gpu_vend[v] = V + isolated_us * 1024;
    running_gpu += 1;
  }

  // Admission procedure at the current T.
  void admission() {
    // 1. Tools whose predecessors are all done become ready, in index order.
    for (int v = 0; v < s.n; ++v) {
      if (status[v] != kPending || !predecessors_done(v)) continue;
      ready_time[v] = T;
      if (mode[v] == kCpu) {
        status[v] = kRunning;
        cpu_end[v] = T + s.cpu[v];
      } else if (mode[v] == kGpuNow) {
        start_on_gpu(v, s.gpu[v] + s.xfer[v]);
        if (live_vram > s.budget) {  // out of memory at start
          infeasible = true;
          return;
        }
      } else {
        status[v] = kWaitingInQueue;
      }
    }
    // 2. The queue head: earliest ready time, ties to the lower index.
    int head = -1;
    for (int v = 0; v < s.n; ++v) {
      if (status[v] != kWaitingInQueue) continue;
      if (head < 0 || ready_time[v] < ready_time[head]) head = v;
    }
    if (head < 0) return;
    if (s.vram[head] > s.budget) {  // can never be admitted
      infeasible = true;
      return;
    }
    if (!queue_busy && live_vram + s.vram[head] <= s.budget) {
      start_on_gpu(head, s.load[head] + s.gpu[head] + s.xfer[head]);
      queue_busy = true;
    }
    // Otherwise the head keeps waiting (no bypass).
  }

  // Returns the makespan, or kInfeasibleMakespan.
  uint64_t run() {
    admission();
    if (infeasible) return kInfeasibleMakespan;
    while (!all_done()) {
      // 1. Next CPU completion.
      uint64_t t_cpu = kInfinity;
      for (int v = 0; v < s.n; ++v)
        if (status[v] == kRunning && mode[v] == kCpu && cpu_end[v] < t_cpu) t_cpu = cpu_end[v];
      // 2. Next GPU completion under the current slowdown f[k].
      uint64_t t_gpu = kInfinity, v_min = kInfinity;
      if (running_gpu > 0) {
        for (int v = 0; v < s.n; ++v)
          if (status[v] == kRunning && mode[v] != kCpu && gpu_vend[v] < v_min) v_min = gpu_vend[v];
        t_gpu = T + ceil_div((v_min - V) * s.slowdown[running_gpu], 1ull << 20);
      }
      // Under the model something is always running here; a stalled state
      // would mean a broken simulation, reported rather than looped on.
      if (t_cpu == kInfinity && t_gpu == kInfinity) return kStalled;
      // 3. Advance to the earlier event.
      if (t_gpu <= t_cpu) {
        T = t_gpu;
        V = v_min;
      } else {
        if (running_gpu > 0) V += ((t_cpu - T) << 20) / s.slowdown[running_gpu];
        T = t_cpu;
      }
      // 4. Retire every tool that ends now.
      for (int v = 0; v < s.n; ++v) {
        if (status[v] != kRunning) continue;
        if (mode[v] == kCpu) {
          if (cpu_end[v] == T) status[v] = kDone;
        } else if (gpu_vend[v] == V) {
          status[v] = kDone;
          live_vram -= s.vram[v];
          running_gpu -= 1;
          if (mode[v] == kGpuQueue) queue_busy = false;
        }
      }
      // 5. Admission at the new T.
      admission();
      if (infeasible) return kInfeasibleMakespan;
    }
    return T;
  }
};

uint64_t evaluate(const OracleScenario& s, uint64_t idx) {
  int mode[kMaxTools];
  decode_mapping(idx, s.n, mode);
  Simulation sim(s, mode);
  return sim.run();
}

// Index of the b-th mapping of the binary decision space.
uint64_t binary_to_index(uint64_t b, int n) {
  uint64_t idx = 0, p = 1;
  for (int i = 0; i < n; ++i, p *= 3)
    if ((b >> i) & 1) idx += p;
  return idx;
}

uint64_t num_mappings(int n) {
  uint64_t p = 1;
  for (int i = 0; i < n; ++i) p *= 3;
  return p;
}

struct Best {
  uint64_t makespan = kInfinity;
  uint64_t index = kInfinity;
  bool found = false;
  void offer(uint64_t ms, uint64_t idx) {
    if (ms == kInfeasibleMakespan) return;
    if (!found || ms < makespan || (ms == makespan && idx < index)) {
      makespan = ms;
      index = idx;
      found = true;
    }
  }
};

int clamp_threads(int nthreads, uint64_t count) {
  if (nthreads < 1) nthreads = 1;
  if ((uint64_t)nthreads > count) nthreads = (int)(count ? count : 1);
  return nthreads;
}

}  // namespace

extern "C" {

int bf_oracle_flat_words(void) { return kFlatWords; }

// Makespan of mapping `idx`; 0xFFFFFFFF when infeasible.
uint64_t bf_oracle_evaluate(const uint32_t* flat, uint64_t idx) {
  return evaluate(unpack(flat), idx);
}

// Makespans and feasibility flags of mappings [first, first+count), split over
// `nthreads` host threads (contiguous ranges).
void bf_oracle_eval_range(const uint32_t* flat, uint64_t first, uint64_t count,
                          uint64_t* out_makespan, uint8_t* out_feasible, int nthreads) {
  const OracleScenario s = unpack(flat);
  nthreads = clamp_threads(nthreads, count);
  std::vector<std::thread> pool;
  for (int t = 0; t < nthreads; ++t) {
    uint64_t lo = count * t / nthreads, hi = count * (t + 1) / nthreads;
    pool.emplace_back([&, lo, hi]() {
      for (uint64_t j = lo; j < hi; ++j) {
        uint64_t ms = evaluate(s, first + j);
        out_makespan[j] = ms;
        out_feasible[j] = ms != kInfeasibleMakespan;
      }
    });
  }
  for (auto& th : pool) th.join();
}

// Best feasible mapping over [first, first+count): writes its index and
// makespan; returns 1 if one was found, 0 otherwise.
int bf_oracle_search_range(const uint32_t* flat, uint64_t first, uint64_t count,
                           uint64_t* out_index, uint64_t* out_makespan, int nthreads) {
  const OracleScenario s = unpack(flat);
  nthreads = clamp_threads(nthreads, count);
  std::vector<Best> best(nthreads);
  std::vector<std::thread> pool;
  for (int t = 0; t < nthreads; ++t) {
    uint64_t lo = count * t / nthreads, hi = count * (t + 1) / nthreads;
    pool.emplace_back([&, t, lo, hi]() {
      for (uint64_t j = lo; j < hi; ++j) best[t].offer(evaluate(s, first + j), first + j);
    });
  }
  for (auto& th : pool) th.join();
  Best all;
  for (auto& b : best)
    if (b.found) all.offer(b.makespan, b.index);
  if (!all.found) return 0;
  *out_index = all.index;
  *out_makespan = all.makespan;
  return 1;
}

// Summary of mappings [first, first+count) for comparing whole makespan
// streams without storing them: out[0] = number of feasible mappings,
// out[1] = sum of their makespans, out[2] = sum over every mapping of
// makespan(idx) * (idx * 2654435761 + 1) modulo 2^64 (infeasible counted as
// 0xFFFFFFFF), out[3] = best index, out[4] = best makespan (0xFFFFFFFF and
// index 2^64-1 when nothing is feasible).
void bf_oracle_summary_range(const uint32_t* flat, uint64_t first, uint64_t count,
                             uint64_t* out, int nthreads) {
  const OracleScenario s = unpack(flat);
  nthreads = clamp_threads(nthreads, count);
  std::vector<uint64_t> feasible(nthreads, 0), total(nthreads, 0), hash(nthreads, 0);
  std::vector<Best> best(nthreads);
  std::vector<std::thread> pool;
  for (int t = 0; t < nthreads; ++t) {
    uint64_t lo = count * t / nthreads, hi = count * (t + 1) / nthreads;
    pool.emplace_back([&, t, lo, hi]() {
      for (uint64_t j = lo; j < hi; ++j) {
        const uint64_t idx = first + j;
        const uint64_t ms = evaluate(s, idx);
        if (ms != kInfeasibleMakespan) {
          feasible[t] += 1;
          total[t] += ms;
        }
        hash[t] += ms * (idx * 2654435761ull + 1);
        best[t].offer(ms, idx);
      }
    });
  }
  for (auto& th : pool) th.join();
  Best all;
  out[0] = out[1] = out[2] = 0;
  for (int t = 0; t < nthreads; ++t) {
    out[0] += feasible[t];
    out[1] += total[t];
    out[2] += hash[t];
    if (best[t].found) all.offer(best[t].makespan, best[t].index);
  }
  out[3] = all.found ? all.index : kInfinity;
  out[4] = all.found ? all.makespan : kInfeasibleMakespan;
}

// Best feasible mapping of the binary decision space among its members
// b in [first, first+count) (b as above, 0 <= b < 2^n): writes its
// (ternary) index and makespan; returns 1 if one was found, 0 otherwise.
int bf_oracle_search_binary_range(const uint32_t* flat, uint64_t first, uint64_t count,
                                  uint64_t* out_index, uint64_t* out_makespan, int nthreads) {
  const OracleScenario s = unpack(flat);
  nthreads = clamp_threads(nthreads, count);
  std::vector<Best> best(nthreads);
  std::vector<std::thread> pool;
  for (int t = 0; t < nthreads; ++t) {
    uint64_t lo = count * t / nthreads, hi = count * (t + 1) / nthreads;
    pool.emplace_back([&, t, lo, hi]() {
      for (uint64_t j = lo; j < hi; ++j) {
        const uint64_t idx = binary_to_index(first + j, s.n);
        best[t].offer(evaluate(s, idx), idx);
      }
    });
  }
  for (auto& th : pool) th.join();
  Best all;
  for (auto& b : best)
    if (b.found) all.offer(b.makespan, b.index);
  if (!all.found) return 0;
  *out_index = all.index;
  *out_makespan = all.makespan;
  return 1;
}

// Full search of each of `count` scenarios (flat records back to back).
void bf_oracle_search_batch(const uint32_t* flats, uint64_t count, uint64_t* out_index,
                            uint64_t* out_makespan, int nthreads) {
  nthreads = clamp_threads(nthreads, count);
  std::vector<std::thread> pool;
  for (int t = 0; t < nthreads; ++t) {
    uint64_t lo = count * t / nthreads, hi = count * (t + 1) / nthreads;
    pool.emplace_back([&, lo, hi]() {
      for (uint64_t j = lo; j < hi; ++j) {
        const OracleScenario s = unpack(flats + j * kFlatWords);
        Best b;
        const uint64_t total = num_mappings(s.n);
        for (uint64_t idx = 0; idx < total; ++idx) b.offer(evaluate(s, idx), idx);
        out_index[j] = b.found ? b.index : kInfinity;
        out_makespan[j] = b.found ? b.makespan : kInfeasibleMakespan;
      }
    });
  }
  for (auto& th : pool) th.join();
}

}  // extern "C"
