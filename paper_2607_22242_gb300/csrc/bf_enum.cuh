// bf_enum.cuh -- how a warp enumerates its share of the mapping space (see
// bfk::Plan): the shared prefix simulation and each lane's mid/inner walk.
// Used by the kernels in bf_kernels.cu; sinks receive (index, makespan).
#pragma once

#include "bf_sim.cuh"

namespace bfk {

// Simulate prefix p once per warp and save its window state in `snap`.
// Returns false (warp-uniformly) when every mapping with this prefix is
// infeasible.
// NP >= n is the slot count of the prefix simulation.
template <int NP, typename TB>
__device__ __forceinline__ bool prefix_phase(const TB& tb, const SmemTables& sd, const Plan& plan,
                                             uint32_t p, Digits& dgp, Snapshot& snap) {
  dgp = decode(p, plan.P);
  bool ok = (dgp.que & tb.big_mask) == 0u;
  if (ok) {
    State<NP> s;
    init_state(s, tb.all_mask);
    const uint32_t later = tb.all_mask & ~((1u << plan.P) - 1u);
    ok = run<NP>(s, tb, sd, dgp, later) == kRunStopped;
    if (ok && (threadIdx.x & 31) == 0) save_window(s, plan.W0, tb.n - plan.W0, snap);
  }
  __syncwarp();
  return ok;
}

// Every mapping (p, m, i) of this lane, in window form, handed to
// sink(idx, makespan).  `ok` is the prefix verdict; the prefix digits dgp and
// the warp's snapshot come from prefix_phase.  `slot`/`stride` is this lane's
// shared-memory area of LaneWords<NW>::value words for the inner-level state.
template <int NW, typename TB, typename Sink>
__device__ __forceinline__ void lane_mappings(const TB& tw, const SmemTables& sdw, const Plan& plan,
                                              uint32_t p, bool ok, Digits dgp, const Snapshot& snap,
                                              uint32_t* slot, uint32_t stride, Sink& sink) {
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t shm = plan.P - plan.W0;          // first mid tool, window numbering
  const uint32_t shi = shm + plan.M;              // first inner tool, window numbering
  const uint32_t inner_mask = tw.all_mask & ~((1u << shi) - 1u);
  const uint64_t stride_i = (uint64_t)plan.pow3P * plan.pow3M;
  for (uint32_t m = lane; m < plan.pow3M; m += 32) {
    // Inner combinations of (p, m) inside [first, last].
    const uint64_t base = (uint64_t)p + (uint64_t)plan.pow3P * m;
    uint32_t i_lo = plan.i_lo, i_hi = plan.i_hi;
    while (i_lo <= i_hi && base + stride_i * i_lo < plan.first) ++i_lo;
    while (i_hi >= i_lo && base + stride_i * i_hi > plan.last) {
      if (i_hi == 0) { i_lo = 1; break; }
      --i_hi;
    }
    if (i_lo > i_hi) continue;
    if (!ok) {
      for (uint32_t i = i_lo; i <= i_hi; ++i) sink((uint32_t)(base + stride_i * i), kInfeasible);
      continue;
    }
    const Digits dm = decode(m, plan.M);
    const Digits dmid{(dgp.now >> plan.W0) | (dm.now << shm), (dgp.que >> plan.W0) | (dm.que << shm)};
    State<NW> w;
    load_window(snap, w);
    uint32_t r = kRunInfeasible;
    if ((dmid.que & tw.big_mask) == 0u) r = run<NW>(w, tw, sdw, dmid, inner_mask);
    if (plan.I == 0u) {  // no inner level: the run went to the end
      sink((uint32_t)base, r == kRunFinished ? w.T : kInfeasible);
      continue;
    }
    if (r != kRunStopped) {  // infeasible before any inner tool started
      for (uint32_t i = i_lo; i <= i_hi; ++i) sink((uint32_t)(base + stride_i * i), kInfeasible);
      continue;
    }
    save_lane(w, slot, stride);
    for (uint32_t i = i_lo; i <= i_hi; ++i) {
      const Digits di = decode(i, plan.I);
      const Digits dg{dmid.now | (di.now << shi), dmid.que | (di.que << shi)};
      uint32_t ms = kInfeasible;
      if ((dg.que & tw.big_mask) == 0u) {
        if (i != i_lo) load_lane(slot, stride, w);
        ms = run<NW>(w, tw, sdw, dg, 0u) == kRunFinished ? w.T : kInfeasible;
      }
      sink((uint32_t)(base + stride_i * i), ms);
    }
  }
}

struct MinKeySink {
  unsigned long long best = ~0ull;
  __device__ __forceinline__ void operator()(uint32_t idx, uint32_t ms) {
    best = min(best, ((unsigned long long)ms << 32) | idx);
  }
};

struct StoreSink {
  uint32_t first;
  uint32_t* ms_out;
  uint8_t* fe_out;
  __device__ __forceinline__ void operator()(uint32_t idx, uint32_t ms) {
    ms_out[idx - first] = ms;
    fe_out[idx - first] = ms != kInfeasible;
  }
};

}  // namespace bfk
