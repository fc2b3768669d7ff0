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

// Canonical index part of `count` tools from `first_tool` on, whose modes are
// bits 0.. of d: the sum of mode x 3^orig (plan.pv; 3^v for tables in the
// scenario's own numbering).
__device__ __forceinline__ uint32_t index_part(const Plan& plan, Digits d, uint32_t first_tool, uint32_t count) {
  uint32_t x = 0u;
#pragma unroll
  for (uint32_t k = 0; k < (uint32_t)kMaxTools; ++k) {
    if (k >= count) break;
    const uint32_t pv = plan.pv[first_tool + k];
    x += (((d.now >> k) & 1u) + 2u * ((d.que >> k) & 1u)) * pv;
  }
  return x;
}

// Offset of inner combination i (at most two inner tools, i < 9) in the
// canonical index.
__device__ __forceinline__ uint32_t inner_offset(const Plan& plan, uint32_t i) {
  const uint32_t d1 = (i * 11u) >> 5;  // i / 3 for i < 9
  return (i - 3u * d1) * plan.pvA + d1 * plan.pvB;
}

// Words of the mid-part table (3^M <= 729 entries), rounded up to 16 bytes.
__host__ __device__ inline uint32_t mid_part_words(uint32_t pow3M) { return (pow3M + 3u) & ~3u; }
constexpr uint32_t kMaxMidPartWords = 732;

// The canonical index part of every mid combination (block-cooperative).
__device__ __forceinline__ void fill_mid_parts(const Plan& plan, uint32_t* mpart) {
  for (uint32_t m = threadIdx.x; m < plan.pow3M; m += blockDim.x)
    mpart[m] = index_part(plan, decode(m, plan.M), plan.P, plan.M);
}

// The canonical index of mapping (p, m, i) of a warp task.  In the scenario's
// own numbering (RL = false) it is p + 3^P m + 3^(P+M) i; with renumbered
// tables (RL = true, whole-space searches) the prefix part of p's modes,
// mpart[m] and the inner part of i (Plan::pv, pvA, pvB).
template <bool RL>
struct TaskIndex {
  uint32_t cp;             // prefix part
  const uint32_t* mpart;   // RL only
  uint64_t stride_i;       // 3^(P+M) (RL: unused)
  __device__ __forceinline__ uint64_t base(const Plan& plan, uint32_t m) const {
    if constexpr (RL) return cp + mpart[m];
    else return (uint64_t)cp + (uint64_t)plan.pow3P * m;
  }
  __device__ __forceinline__ uint64_t inner(const Plan& plan, uint32_t i) const {
    if constexpr (RL) return inner_offset(plan, i);
    else return stride_i * i;
  }
  // The last tool's mode a when it is the only inner tool.
  __device__ __forceinline__ uint64_t last(const Plan& plan, uint32_t a) const {
    if constexpr (RL) return a * plan.pvA;
    else return stride_i * a;
  }
};

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
template <int NP, int NW, bool RL, typename TBF, typename TBW, typename Sink>
__device__ __forceinline__ void prefix_task(const TBF& tb, const SmemTables& sd, const uint32_t* rt, const TBW& tw,
                                            const SmemTables& sdw, const uint32_t* rtw, const Plan& plan,
                                            const uint32_t* mpart, uint32_t p, bool p_valid, uint32_t part,
                                            uint32_t* slotA, uint32_t* slotB, uint32_t stride, Sink& sink) {
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
  const TaskIndex<RL> ix{RL ? index_part(plan, dgp, 0u, plan.P) : p, mpart, (uint64_t)plan.pow3P * plan.pow3M};
  const Digits dgw{dgp.now >> plan.W0, dgp.que >> plan.W0};
  const uint32_t m0 = plan.m_lo + part * plan.m_chunk;
  const uint32_t m1 = min(m0 + plan.m_chunk - 1u, plan.m_hi);
  Digits dm = decode(m0, plan.M);
  for (uint32_t m = m0; m <= m1; ++m, increment(dm)) {
    const uint64_t base = ix.base(plan, m);
    uint32_t i_lo = 0u, i_hi = plan.pow3I - 1u;
    if (!p_valid) continue;
    // (a part of the space is always in the scenario's numbering)
    if (!plan.full && !inner_range(plan, base, ix.stride_i, &i_lo, &i_hi)) continue;
    if (!ok) {  // every mapping with this prefix is infeasible
      for (uint32_t i = i_lo; i <= i_hi; ++i) sink((uint32_t)(base + ix.inner(plan, i)), kInfeasible);
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
      for (uint32_t i = i_lo; i <= i_hi; ++i) sink((uint32_t)(base + ix.inner(plan, i)), kInfeasible);
      continue;
    }
    if ((uint64_t)w.T + plan.tail_q > plan.bound) continue;  // pruned at the inner checkpoint
    if (plan.last_apart || (plan.I == 1u && (w.done | inner_mask) == 0xFFFFFFFFu)) {
      // Everything but the last tool has ended: it runs alone from w.T.
      for (uint32_t i = i_lo; i <= i_hi; ++i) {
        const uint32_t d = plan.alone[i];
        sink((uint32_t)(base + ix.last(plan, i)), d == kInfeasible ? kInfeasible : w.T + d);
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
      sink((uint32_t)(base + ix.inner(plan, i)), ms);
    }
  }
}

// Run one warp task of a plan: prefix group `g` (prefix p_lo + 32 g + lane)
// and mid chunk `part`.  NP >= n is the prefix simulation's slot count, NW >=
// the window's.  slotA / slotB are this lane's shared-memory areas of
// LaneWords<NW> words (stride `stride`) for the state at the prefix checkpoint
// and at the inner checkpoint; rt / rtw are the readiness tables of the full
// and window tables.
template <int NP, int NW, bool RL, typename TBF, typename TBW, typename Sink>
__device__ __forceinline__ void warp_task(const TBF& tb, const SmemTables& sd, const uint32_t* rt, const TBW& tw,
                                          const SmemTables& sdw, const uint32_t* rtw, const Plan& plan,
                                          const uint32_t* mpart, uint32_t g, uint32_t part, uint32_t* slotA,
                                          uint32_t* slotB, uint32_t stride, Sink& sink) {
  const uint64_t p64 = (uint64_t)plan.p_lo + 32ull * g + (threadIdx.x & 31u);
  prefix_task<NP, NW, RL>(tb, sd, rt, tw, sdw, rtw, plan, mpart, (uint32_t)p64, p64 <= plan.p_hi, part, slotA, slotB,
                      stride, sink);
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
