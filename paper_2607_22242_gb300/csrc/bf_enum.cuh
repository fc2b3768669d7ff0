// bf_enum.cuh -- one warp task of the enumeration (see bfk::Plan): 32
// consecutive prefixes, one per lane, times a chunk of mid combinations, each
// with its inner combinations.  Used by the kernels in bf_kernels.cu; the
// sink receives (canonical index, makespan) for every mapping of the task
// that lies inside [plan.first, plan.last].
#pragma once

#include "bf_sim.cuh"

namespace bfk {

// Inner combinations [*lo, *hi] of (p, m) that fall inside [first, last];
// returns false when there is none.  base = p + 3^P * m.
__device__ __forceinline__ bool inner_range(const Plan& plan, uint64_t base, uint64_t stride_i, uint32_t* lo,
                                            uint32_t* hi) {
  uint32_t a = plan.i_lo, b = plan.i_hi;
  while (a <= b && base + stride_i * a < plan.first) ++a;
  while (a <= b && base + stride_i * b > plan.last) {
    if (b == 0u) return false;
    --b;
  }
  *lo = a;
  *hi = b;
  return a <= b;
}

// Simulate prefix p up to the first instant a tool >= P would become ready.
// Returns false if every mapping with this prefix is infeasible; otherwise
// *T_check is that instant and, when slotA is not null, the window state is
// saved there.
template <int NP, int NW, typename TBF>
__device__ __forceinline__ bool prefix_checkpoint(const TBF& tb, const SmemTables& sd, const uint32_t* rt,
                                                  const Plan& plan, uint32_t p, Digits* dgp, uint32_t* T_check,
                                                  uint32_t* slotA, uint32_t stride) {
  *dgp = decode(p, plan.P);
  if (dgp->que & tb.big_mask) return false;
  State<NP> s;
  init_state(s, tb.all_mask);
  const uint32_t later = tb.all_mask & ~((1u << plan.P) - 1u);
  if (run<NP>(s, tb, sd, rt, *dgp, later) != kRunStopped) return false;
  *T_check = s.T;
  if (slotA) save_prefix_window<NP, NW>(s, plan.W0, tb.n - plan.W0 - plan.last_apart, slotA, stride);
  return true;
}

// A warp task whose lanes hold prefixes p (valid when p_valid).  Mappings that
// the plan's bound proves worse than a known feasible mapping (pruned
// searches only) are skipped without reaching the sink.
template <int NP, int NW, typename TBF, typename TBW, typename Sink>
__device__ __forceinline__ void prefix_task(const TBF& tb, const SmemTables& sd, const uint32_t* rt, const TBW& tw,
                                            const SmemTables& sdw, const uint32_t* rtw, const Plan& plan,
                                            uint32_t p, bool p_valid, uint32_t part, uint32_t* slotA,
                                            uint32_t* slotB, uint32_t stride, Sink& sink) {
  // ---- this lane's prefix, up to the first instant a tool >= P is ready ----
  Digits dgp{0u, 0u};
  bool ok = false;
  if (p_valid) {
    uint32_t T_check = 0u;
    ok = prefix_checkpoint<NP, NW>(tb, sd, rt, plan, p, &dgp, &T_check, slotA, stride);
    if (ok && (uint64_t)T_check + plan.tail_p > plan.bound) p_valid = false;  // pruned
  }

  // ---- the task's mid combinations, in lockstep across the warp -----------
  const uint32_t shm = plan.P - plan.W0;  // first mid tool, window numbering
  const uint32_t shi = shm + plan.M;      // first inner tool, window numbering
  const uint32_t inner_mask = tw.all_mask & ~((1u << shi) - 1u);
  const uint64_t stride_i = (uint64_t)plan.pow3P * plan.pow3M;
  const Digits dgw{dgp.now >> plan.W0, dgp.que >> plan.W0};
  const uint32_t m0 = plan.m_lo + part * plan.m_chunk;
  const uint32_t m1 = min(m0 + plan.m_chunk - 1u, plan.m_hi);
  Digits dm = decode(m0, plan.M);
  for (uint32_t m = m0; m <= m1; ++m, increment(dm)) {
    const uint64_t base = (uint64_t)p + (uint64_t)plan.pow3P * m;
    uint32_t i_lo = 0u, i_hi = plan.pow3I - 1u;
    if (!p_valid) continue;
    if (!plan.full && !inner_range(plan, base, stride_i, &i_lo, &i_hi)) continue;
    if (!ok) {  // every mapping with this prefix is infeasible
      for (uint32_t i = i_lo; i <= i_hi; ++i) sink((uint32_t)(base + stride_i * i), kInfeasible);
      continue;
    }
    const Digits dmid{dgw.now | (dm.now << shm), dgw.que | (dm.que << shm)};
    State<NW> w;
    uint32_t r = kRunInfeasible;
    if ((dmid.que & tw.big_mask) == 0u) {
      load_lane(slotA, stride, w);
      r = run<NW>(w, tw, sdw, rtw, dmid, inner_mask);
    }
    if (plan.I == 0u) {  // no inner level: the run went to the end
      sink((uint32_t)base, r == kRunFinished ? w.T : kInfeasible);
      continue;
    }
    // The run stops when an inner tool would become ready; with the last tool
    // apart (the window lacks it) it ends when every other tool has ended.
    if (r != (plan.last_apart ? kRunFinished : kRunStopped)) {  // infeasible before that
      for (uint32_t i = i_lo; i <= i_hi; ++i) sink((uint32_t)(base + stride_i * i), kInfeasible);
      continue;
    }
    if ((uint64_t)w.T + plan.tail_q > plan.bound) continue;  // pruned at the inner checkpoint
    if (plan.last_apart || (plan.I == 1u && (w.done | inner_mask) == 0xFFFFFFFFu)) {
      // Everything but the last tool has ended: it runs alone from w.T.
      for (uint32_t i = i_lo; i <= i_hi; ++i) {
        const uint32_t d = plan.alone[i];
        sink((uint32_t)(base + stride_i * i), d == kInfeasible ? kInfeasible : w.T + d);
      }
      continue;
    }
    save_lane(w, slotB, stride);
    for (uint32_t i = i_lo; i <= i_hi; ++i) {
      const Digits di = decode(i, plan.I);
      const Digits dg{dmid.now | (di.now << shi), dmid.que | (di.que << shi)};
      uint32_t ms = kInfeasible;
      if ((dg.que & tw.big_mask) == 0u) {
        if (i != i_lo) load_lane(slotB, stride, w);
        ms = run<NW>(w, tw, sdw, rtw, dg, 0u) == kRunFinished ? w.T : kInfeasible;
      }
      sink((uint32_t)(base + stride_i * i), ms);
    }
  }
}

// Run one warp task of a plan: prefix group `g` (prefix p_lo + 32 g + lane)
// and mid chunk `part`.  NP >= n is the prefix simulation's slot count, NW >=
// the window's.  slotA / slotB are this lane's shared-memory areas of
// LaneWords<NW> words (stride `stride`) for the state at the prefix checkpoint
// and at the inner checkpoint; rt / rtw are the readiness tables of the full
// and window tables.
template <int NP, int NW, typename TBF, typename TBW, typename Sink>
__device__ __forceinline__ void warp_task(const TBF& tb, const SmemTables& sd, const uint32_t* rt, const TBW& tw,
                                          const SmemTables& sdw, const uint32_t* rtw, const Plan& plan, uint32_t g,
                                          uint32_t part, uint32_t* slotA, uint32_t* slotB, uint32_t stride,
                                          Sink& sink) {
  const uint64_t p64 = (uint64_t)plan.p_lo + 32ull * g + (threadIdx.x & 31u);
  prefix_task<NP, NW>(tb, sd, rt, tw, sdw, rtw, plan, (uint32_t)p64, p64 <= plan.p_hi, part, slotA, slotB, stride,
                      sink);
}

// The other assignment of lanes, for DAGs where the prefix settles nothing
// (the window is the whole DAG: most tools start at once, so lanes holding
// different early modes diverge from the first event): the warp shares
// prefix p (each lane simulates it, identically) and lane l takes mid
// combinations l, l + 32, ...; the lanes then differ only in later tools.
// Measured on 4096 random layered 10-tool DAGs: 8 % faster than lanes owning
// prefixes.
template <int NP, int NW, typename TBF, typename TBW, typename Sink>
__device__ __forceinline__ void mid_lane_task(const TBF& tb, const SmemTables& sd, const uint32_t* rt, const TBW& tw,
                                              const SmemTables& sdw, const uint32_t* rtw, const Plan& plan,
                                              uint32_t p, uint32_t* slotA, uint32_t* slotB, uint32_t stride,
                                              Sink& sink) {
  Digits dgp{0u, 0u};
  uint32_t T_check = 0u;
  const bool ok = prefix_checkpoint<NP, NW>(tb, sd, rt, plan, p, &dgp, &T_check, slotA, stride);
  const uint32_t shm = plan.P - plan.W0;
  const uint32_t shi = shm + plan.M;
  const uint32_t inner_mask = tw.all_mask & ~((1u << shi) - 1u);
  const uint64_t stride_i = (uint64_t)plan.pow3P * plan.pow3M;
  const Digits dgw{dgp.now >> plan.W0, dgp.que >> plan.W0};
  const uint32_t lane = threadIdx.x & 31u;
  for (uint32_t m0 = 0; m0 < plan.pow3M; m0 += 32u) {
    const uint32_t m = m0 + lane;
    if (m >= plan.pow3M) continue;
    const uint64_t base = (uint64_t)p + (uint64_t)plan.pow3P * m;
    if (!ok) {
      for (uint32_t i = 0; i < plan.pow3I; ++i) sink((uint32_t)(base + stride_i * i), kInfeasible);
      continue;
    }
    const Digits dm = decode(m, plan.M);
    const Digits dmid{dgw.now | (dm.now << shm), dgw.que | (dm.que << shm)};
    State<NW> w;
    uint32_t r = kRunInfeasible;
    if ((dmid.que & tw.big_mask) == 0u) {
      load_lane(slotA, stride, w);
      r = run<NW>(w, tw, sdw, rtw, dmid, inner_mask);
    }
    if (plan.I == 0u) {
      sink((uint32_t)base, r == kRunFinished ? w.T : kInfeasible);
      continue;
    }
    if (r != (plan.last_apart ? kRunFinished : kRunStopped)) {
      for (uint32_t i = 0; i < plan.pow3I; ++i) sink((uint32_t)(base + stride_i * i), kInfeasible);
      continue;
    }
    if (plan.last_apart || (plan.I == 1u && (w.done | inner_mask) == 0xFFFFFFFFu)) {  // the last tool runs alone
      for (uint32_t i = 0; i < plan.pow3I; ++i) {
        const uint32_t d = plan.alone[i];
        sink((uint32_t)(base + stride_i * i), d == kInfeasible ? kInfeasible : w.T + d);
      }
      continue;
    }
    save_lane(w, slotB, stride);
    for (uint32_t i = 0; i < plan.pow3I; ++i) {
      const Digits di = decode(i, plan.I);
      const Digits dg{dmid.now | (di.now << shi), dmid.que | (di.que << shi)};
      uint32_t ms = kInfeasible;
      if ((dg.que & tw.big_mask) == 0u) {
        if (i != 0u) load_lane(slotB, stride, w);
        ms = run<NW>(w, tw, sdw, rtw, dg, 0u) == kRunFinished ? w.T : kInfeasible;
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
