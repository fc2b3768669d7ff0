// bf_tree.cuh -- the tree search: exact branch and bound over mode prefixes,
// for scenarios of up to 32 tools, over the full decision space (3 modes per
// tool) or the binary cpu/gpu_now space (§4.1: S1-S10 choose between CPU and
// GPU only).
//
// Tools are numbered as in the tables the search runs on (the scenario's
// tools with the sources first, host::relabel_sources_first); results carry
// canonical indices (TreeConsts::pow3).
//
// A node at level d assigns modes to tools [0, d) and holds the simulation
// state at its checkpoint: the first instant at which a tool >= d would
// become ready (bf_sim.cuh, resumable runs).  Until then no tool >= d has
// started, so that state is shared by every mapping extending the node.  A
// child assigns tool d and resumes the parent's state up to its own
// checkpoint.  Nodes at the leaf level L = n - D are not expanded further:
// the leaf kernel resumes each one for all radix^D modes of the last D tools
// and simulates them to the end.
//
// Pruning (Plan::bound's rule, with a per-node bound): the makespan of every
// mapping extending a node is at least the node's lower bound (below); a node
// whose bound exceeds the best makespan found so far (strictly) is dropped.
// The optimum and all its ties have every prefix within the bound, so the
// search returns the same (makespan, lowest index) as full enumeration.
#pragma once

#include "bf_plan.h"
#include "bf_sim.cuh"

namespace bfk {

constexpr int kTreeSlots = 32;
using TablesW = TablesT<kTreeSlots>;
using SmemTablesW = SmemTablesT<kTreeSlots>;

// Leaf window widths compiled for the leaf kernel: a window of nw tools runs
// in the narrowest that holds it.
#define BF_TREE_BUCKETS(X) X(8) X(12) X(16) X(20) X(24) X(32)

// Per-scenario constants of a tree search.
struct TreeConsts {
  uint32_t n;
  uint32_t radix;        // 2: {cpu, gpu_now}; 3: {cpu, gpu_now, gpu_queue}
  uint32_t leaf_level;   // L: nodes at this level go to the leaf kernel
  uint32_t D;            // n - L tools enumerated per leaf node
  uint32_t combos;       // radix^D
  uint32_t prune;        // 0: keep every node (full enumeration)
  uint32_t W0;           // leaf window start: tools below it have ended at every leaf checkpoint
  // 1 when every other tool precedes the last one: when it becomes ready it
  // runs alone, and ends alone[a] after that instant in mode a (0xFFFFFFFF: a
  // GPU mode over budget) -- the model's one remaining event at k = 1.
  uint32_t alone_last;
  uint32_t alone[3];
  uint32_t dmin[kTreeSlots];   // min(c, g + x): no mode runs tool v faster
  uint32_t sdown[kTreeSlots];  // longest path in dmin through v's successors (0 for a sink)
  // 1 when the tools are renumbered (sources first): tree slot v holds tool
  // orig[v] of the scenario, and ties compare canonical indices.
  uint32_t relabeled;
  uint64_t pow3[kTreeSlots];   // 3^(scenario position) of each slot's tool
  // pow3 when ties need it (renumbered tools), else nullptr.
  __device__ __forceinline__ const uint64_t* tie_pow3() const { return relabeled ? pow3 : nullptr; }
};

// A saved node: the state's words, then the digit masks; [word][node] layout
// with stride `cap` (nodes of one level sit side by side, so a warp's accesses
// to one word coalesce).
template <int NT>
struct NodeWords {
  static constexpr int value = 2 * NT + 11;
};

template <int NT>
__device__ __forceinline__ void store_node(const State<NT>& s, Digits dg, uint32_t* buf, uint32_t cap, uint32_t j) {
  uint32_t* p = buf + j;
#pragma unroll
  for (int i = 0; i < NT; ++i) {
    p[(size_t)(2 * i) * cap] = s.ec[i];
    p[(size_t)(2 * i + 1) * cap] = s.eg[i];
  }
  p += (size_t)(2 * NT) * cap;
  p[0 * (size_t)cap] = s.done;
  p[1 * (size_t)cap] = s.pend;
  p[2 * (size_t)cap] = s.run_g;
  p[3 * (size_t)cap] = s.qwait;
  p[4 * (size_t)cap] = s.T;
  p[5 * (size_t)cap] = s.V;
  p[6 * (size_t)cap] = s.L;
  p[7 * (size_t)cap] = s.tc;
  p[8 * (size_t)cap] = s.gmin;
  p[9 * (size_t)cap] = dg.now;
  p[10 * (size_t)cap] = dg.que;
}

template <int NT>
__device__ __forceinline__ void load_node(const uint32_t* buf, uint32_t cap, uint32_t j, State<NT>& s, Digits& dg) {
  const uint32_t* p = buf + j;
#pragma unroll
  for (int i = 0; i < NT; ++i) {
    s.ec[i] = p[(size_t)(2 * i) * cap];
    s.eg[i] = p[(size_t)(2 * i + 1) * cap];
  }
  p += (size_t)(2 * NT) * cap;
  s.done = p[0 * (size_t)cap];
  s.pend = p[1 * (size_t)cap];
  s.run_g = p[2 * (size_t)cap];
  s.qwait = p[3 * (size_t)cap];
  s.T = p[4 * (size_t)cap];
  s.V = p[5 * (size_t)cap];
  s.L = p[6 * (size_t)cap];
  s.tc = p[7 * (size_t)cap];
  s.gmin = p[8 * (size_t)cap];
  dg.now = p[9 * (size_t)cap];
  dg.que = p[10 * (size_t)cap];
}

// Lower bound on the makespan of every mapping that extends a node whose
// state `s` is at a checkpoint (before the admission at s.T), with the modes
// of the tools in `known` given by `dg`:
//   * a running CPU tool ends at ec (exact);
//   * a running GPU tool with r work units left ends no earlier than
//     T + ceil(r / 1024): f[k] >= f[1] = 1024, and the model rounds GPU
//     progress down and completion times up;
//   * a tool not started by T ends no earlier than T + its duration in its
//     mode (c, g + x or l + g + x), or T + min(c, g + x) if its mode is open;
//   * after a tool ends, its successors still need the longest path through
//     them in minimum durations (sdown);
//   * queued tools run one at a time, so all unfinished tools known to be
//     queued end no earlier than T + the sum of their remaining durations.
template <int NT, typename TB, typename Slots>
__device__ __forceinline__ uint64_t lower_bound_of(uint32_t done, uint32_t run_g, uint32_t T32, uint32_t V,
                                                   const Slots& slot, const TB& tb, const TreeConsts& tc, Digits dg,
                                                   uint32_t known) {
  const uint64_t T = T32;
  uint64_t lb = T, qsum = 0u;
#pragma unroll
  for (int v = 0; v < NT; ++v) {
    const uint32_t bit = 1u << v;
    if (done & bit) continue;
    const uint32_t ec = slot.ec(v);
    uint64_t fin;
    if (ec != 0xFFFFFFFFu) {
      fin = ec;
    } else if (run_g & bit) {
      const uint32_t r = slot.eg(v) - V;
      const uint32_t left = (r >> 10) + ((r & 1023u) != 0u);
      fin = T + left;
      if (dg.que & bit) qsum += left;
    } else {
      uint32_t d = tc.dmin[v];
      if (known & bit) {
        d = (dg.now & bit) ? (tb.wnow[v] >> 10) : (dg.que & bit) ? (tb.wq[v] >> 10) : tb.cpu[v];
        if (dg.que & bit) qsum += d;
      }
      fin = T + d;
    }
    lb = max(lb, fin + tc.sdown[v]);
  }
  return max(lb, T + qsum);
}

// Per-slot end times of a state held in registers, or of a node saved in HBM.
template <int NT>
struct StateSlots {
  const State<NT>& s;
  __device__ __forceinline__ uint32_t ec(int v) const { return s.ec[v]; }
  __device__ __forceinline__ uint32_t eg(int v) const { return s.eg[v]; }
};

struct NodeSlots {
  const uint32_t* p;  // word 0 of the node
  uint32_t cap;
  __device__ __forceinline__ uint32_t ec(int v) const { return p[(size_t)(2 * v) * cap]; }
  __device__ __forceinline__ uint32_t eg(int v) const { return p[(size_t)(2 * v + 1) * cap]; }
};

template <int NT, typename TB>
__device__ __forceinline__ uint64_t lower_bound(const State<NT>& s, const TB& tb, const TreeConsts& tc, Digits dg,
                                                uint32_t known) {
  return lower_bound_of<NT>(s.done, s.run_g, s.T, s.V, StateSlots<NT>{s}, tb, tc, dg, known);
}

// The bound of node j of a level buffer, read word by word from HBM.
template <typename TB>
__device__ __forceinline__ uint64_t node_lower_bound(const uint32_t* buf, uint32_t cap, uint32_t j, const TB& tb,
                                                     const TreeConsts& tc, Digits dg, uint32_t known) {
  const uint32_t* p = buf + j;
  const uint32_t* t = p + (size_t)(2 * kTreeSlots) * cap;
  return lower_bound_of<kTreeSlots>(t[0], t[2 * (size_t)cap], t[4 * (size_t)cap], t[5 * (size_t)cap],
                                    NodeSlots{p, cap}, tb, tc, dg, known);
}

// Copy node j of a level buffer into a lane's shared-memory state over the
// window [W0, W0 + NW) (slots past the last tool: no CPU end, stamp 0), with
// masks shifted to window numbering.  Every tool below W0 has ended at every
// leaf node's checkpoint, and no running tool lies outside the window.
template <int NW>
__device__ __forceinline__ void node_to_window(const uint32_t* buf, uint32_t cap, uint32_t j, uint32_t W0,
                                               uint32_t nw, uint32_t* slot, uint32_t stride) {
  const uint32_t* p = buf + j;
#pragma unroll
  for (int i = 0; i < NW; ++i) {
    const uint32_t v = W0 + (uint32_t)i;
    const bool in = v < (uint32_t)kTreeSlots;
    slot[(2 * i) * stride] = in ? p[(size_t)(2 * v) * cap] : 0xFFFFFFFFu;
    slot[(2 * i + 1) * stride] = in ? p[(size_t)(2 * v + 1) * cap] : 0u;
  }
  const uint32_t* t = p + (size_t)(2 * kTreeSlots) * cap;
  const uint32_t wmask = nw >= 32u ? 0xFFFFFFFFu : ((1u << nw) - 1u);
  uint32_t* q = slot + (2 * NW) * stride;
  q[0 * stride] = (t[0 * (size_t)cap] >> W0) | ~wmask;  // done
  q[1 * stride] = (t[1 * (size_t)cap] >> W0) & wmask;   // pend
  q[2 * stride] = t[2 * (size_t)cap] >> W0;             // run_g
  q[3 * stride] = t[3 * (size_t)cap] >> W0;             // qwait
  q[4 * stride] = t[4 * (size_t)cap];                   // T
  q[5 * stride] = t[5 * (size_t)cap];                   // V
  q[6 * stride] = t[6 * (size_t)cap];                   // L
  q[7 * stride] = t[7 * (size_t)cap];                   // tc
  q[8 * stride] = t[8 * (size_t)cap];                   // gmin
}

// The stronger bound of the expansions: the earliest finish EF of every
// unfinished tool, in index (topological) order -- a running CPU tool its end
// time, a running GPU tool T + ceil(r / 1024), any other tool the latest of T
// and its unfinished predecessors' EF, plus its duration in its mode (the
// least over the modes if open) -- and the makespan is at least the largest
// EF and the serial-queue sum of lower_bound().  Every start is no earlier
// than T and than the ends of its predecessors, and no tool runs faster than
// its isolated duration, so EF never exceeds the true end.  `ef` is a
// per-thread column of NT words in shared memory (stride `stride`).  Times fit
// in 32 bits: T plus the durations of a chain of remaining tools stays below
// the validated makespan bound.
template <int NT, typename TB>
__device__ __forceinline__ uint32_t forward_bound(const State<NT>& s, const TB& tb, const TreeConsts& tc, Digits dg,
                                                  uint32_t known, uint32_t* ef, uint32_t stride) {
  const uint32_t T = s.T;
  uint32_t lb = T, qsum = 0u;
#pragma unroll
  for (int v = 0; v < NT; ++v) {
    const uint32_t bit = 1u << v;
    if (s.done & bit) continue;
    uint32_t fin;
    if (s.ec[v] != 0xFFFFFFFFu) {
      fin = s.ec[v];
    } else if (s.run_g & bit) {
      const uint32_t r = s.eg[v] - s.V;
      const uint32_t left = (r >> 10) + ((r & 1023u) != 0u);
      fin = T + left;
      if (dg.que & bit) qsum += left;
    } else {
      uint32_t d = tc.dmin[v];
      if (known & bit) {
        d = (dg.now & bit) ? (tb.wnow[v] >> 10) : (dg.que & bit) ? (tb.wq[v] >> 10) : tb.cpu[v];
        if (dg.que & bit) qsum += d;
      }
      uint32_t start = T;
      for (uint32_t m = tb.pred[v] & ~s.done; m; m &= m - 1u) start = max(start, ef[(__ffs(m) - 1) * stride]);
      fin = start + d;
    }
    ef[v * stride] = fin;
    lb = max(lb, fin);
  }
  return max(lb, T + qsum);
}

// Child (tool d in mode a) of the node whose state and digits are in s / dg,
// advanced in place to the child's checkpoint.  Returns false when every
// mapping below the child is infeasible or, with pruning, provably worse
// than `bound` (forward_bound, scratch column `ef`).  Requires d + 1 < n.
template <int NT, typename TB, typename SD>
__device__ __forceinline__ bool expand_child(const TB& tb, const SD& sd, const uint32_t* rt, const TreeConsts& tc,
                                             State<NT>& s, Digits& dg, uint32_t d, uint32_t a, uint32_t bound,
                                             uint32_t* ef, uint32_t stride) {
  const uint32_t bit = 1u << d;
  if (a == 1u) dg.now |= bit;
  if (a == 2u) {
    if (tb.big_mask & bit) return false;  // a queued tool with m > M never starts
    dg.que |= bit;
  }
  const uint32_t assigned = (bit << 1) - 1u;  // tools [0, d]; all ones for d = 31
  if (run<NT>(s, tb, sd, rt, dg, tb.all_mask & ~assigned) != kRunStopped) return false;
  return !tc.prune || forward_bound<NT>(s, tb, tc, dg, assigned, ef, stride) <= bound;
}

// Digits of leaf combination c (tools [L, n)), as masks shifted to tool L.
__device__ __forceinline__ Digits leaf_digits(uint32_t c, uint32_t radix, uint32_t D, uint32_t L) {
  if (radix == 2u) return Digits{c << L, 0u};
  const Digits d = decode(c, D);
  return Digits{d.now << L, d.que << L};
}

// Canonical index of a mapping given as digit masks.
__device__ __forceinline__ uint64_t index_of(Digits dg, const uint64_t* pow3) {
  uint64_t idx = 0;
  for (uint32_t m = dg.now; m; m &= m - 1u) idx += pow3[__ffs(m) - 1];
  for (uint32_t m = dg.que; m; m &= m - 1u) idx += 2u * pow3[__ffs(m) - 1];
  return idx;
}

// a < b in slot order: the highest slot whose digits differ decides (the
// canonical order when the slots are not renumbered).
__device__ __forceinline__ bool index_less(Digits a, Digits b) {
  const uint32_t diff = (a.now ^ b.now) | (a.que ^ b.que);
  if (diff == 0u) return false;
  const uint32_t top = 1u << (31 - __clz(diff));
  const uint32_t da = ((a.now & top) ? 1u : 0u) + ((a.que & top) ? 2u : 0u);
  const uint32_t db = ((b.now & top) ? 1u : 0u) + ((b.que & top) ? 2u : 0u);
  return da < db;
}

// Best mapping seen: lowest makespan, ties to the lowest canonical index.
// pow3 (TreeConsts::tie_pow3) is nullptr when slot order is the scenario's
// order; otherwise ties compare the canonical indices it gives.
struct LaneBest {
  uint32_t ms = kInfeasible;
  Digits dg{0u, 0u};
  __device__ __forceinline__ void offer(uint32_t m, Digits d, const uint64_t* pow3) {
    if (m < ms ||
        (m == ms && m != kInfeasible && (pow3 ? index_of(d, pow3) < index_of(dg, pow3) : index_less(d, dg)))) {
      ms = m;
      dg = d;
    }
  }
};

// Simulate combinations [c0, c1) of the leaf node saved in `slot` (a lane's
// shared-memory window state, stride `stride`) whose digits are `dg` (all
// tools); tw/sdw/rtw are the window's tables.  `valid` false runs the loop
// without work (lanes of a warp stay in lockstep).
// With tc.alone_last, [c0, c1) are combinations of the leaf tools but the
// last one: each is simulated until the last tool becomes ready (everything
// else has ended then) and yields one makespan per mode of the last tool.
template <int NW, typename TBW, typename SD>
__device__ __forceinline__ void leaf_combos(const TBW& tw, const SD& sdw, const uint32_t* rtw, const TreeConsts& tc,
                                            const uint32_t* slot, uint32_t stride, Digits dg, bool valid,
                                            uint32_t c0, uint32_t c1, LaneBest& best) {
  const uint32_t L = tc.leaf_level, W0 = tc.W0;
  const Digits dgw{dg.now >> W0, dg.que >> W0};
  if (tc.alone_last) {
    const uint32_t last = tc.n - 1u, lastw = last - W0;
    for (uint32_t c = c0; c < c1; ++c) {
      if (!valid) continue;
      const Digits dc = leaf_digits(c, tc.radix, tc.D - 1u, L - W0);
      const Digits sim{dgw.now | dc.now, dgw.que | dc.que};
      if (sim.que & tw.big_mask) continue;
      State<NW> w;
      load_lane(slot, stride, w);
      if (run<NW>(w, tw, sdw, rtw, sim, 1u << lastw) != kRunStopped) continue;  // infeasible before it
      const Digits full{dg.now | (dc.now << W0), dg.que | (dc.que << W0)};
      for (uint32_t a = 0; a < tc.radix; ++a) {
        if (tc.alone[a] == kInfeasible) continue;
        best.offer(w.T + tc.alone[a],
                   Digits{full.now | (a == 1u ? 1u << last : 0u), full.que | (a == 2u ? 1u << last : 0u)},
                   tc.tie_pow3());
      }
    }
    return;
  }
  for (uint32_t c = c0; c < c1; ++c) {
    if (!valid) continue;
    const Digits dc = leaf_digits(c, tc.radix, tc.D, L - W0);
    const Digits sim{dgw.now | dc.now, dgw.que | dc.que};
    if (sim.que & tw.big_mask) continue;
    State<NW> w;
    load_lane(slot, stride, w);
    if (run<NW>(w, tw, sdw, rtw, sim, 0u) != kRunFinished) continue;
    best.offer(w.T, Digits{dg.now | (dc.now << W0), dg.que | (dc.que << W0)}, tc.tie_pow3());
  }
}

namespace host {

// Constants of a search over tables tb (the scenario's tools, renumbered or
// not) in the space of radix R (2: binary, 3: full): the leaf depth D (5 tools
// in the full space, 8 in the binary one, all of them for smaller scenarios),
// the leaf window, the lone last tool's durations, the per-tool minimum
// durations and downstream paths of the bounds, and each slot's place value
// in the canonical index.
inline void tree_consts(const TablesW& tb, uint32_t R, bool prune, TreeConsts* out) {
  TreeConsts& tc = *out;
  std::memset(&tc, 0, sizeof tc);
  const uint32_t n = tb.n;
  tc.n = n;
  tc.radix = R;
  tc.D = n < (R == 3 ? 5u : 8u) ? n : (R == 3 ? 5u : 8u);
  tc.leaf_level = n - tc.D;
  tc.combos = 1;
  for (uint32_t i = 0; i < tc.D; ++i) tc.combos *= R;
  tc.prune = prune ? 1u : 0u;
  tc.W0 = window_start(tb, tc.leaf_level);
  {
    uint32_t anc[kTreeSlots];
    ancestors(tb, anc);
    const uint32_t last = n - 1, others = (last >= 32u) ? ~0u : ((1u << last) - 1u);
    tc.alone_last = (tc.D >= 1u && (anc[last] & others) == others) ? 1u : 0u;
    const bool fits = tb.vram[last] <= tb.budget;
    tc.alone[0] = tb.cpu[last];
    tc.alone[1] = fits ? tb.wnow[last] >> 10 : 0xFFFFFFFFu;
    tc.alone[2] = fits ? tb.wq[last] >> 10 : 0xFFFFFFFFu;
  }
  uint64_t down[kTreeSlots] = {0};
  for (int v = (int)n - 1; v >= 0; --v) {
    const uint32_t gpu = tb.wnow[v] >> 10;
    tc.dmin[v] = tb.cpu[v] < gpu ? tb.cpu[v] : gpu;
    uint64_t longest = 0;
    for (uint32_t w = (uint32_t)v + 1; w < n; ++w)
      if ((tb.succ[v] >> w) & 1u) longest = down[w] > longest ? down[w] : longest;
    tc.sdown[v] = (uint32_t)(longest < 0xFFFFFFFFull ? longest : 0xFFFFFFFFull);
    down[v] = tc.dmin[v] + longest;
  }
  for (uint32_t i = 0; i < (uint32_t)kTreeSlots; ++i) tc.pow3[i] = pow3(i < n ? tb.orig[i] : i);
  tc.relabeled = tb.relabeled ? 1u : 0u;
}

}  // namespace host
}  // namespace bfk
