// Host build of the tree search's node logic (bf_tree.cuh, with bf_plan.h and
// bf_sim.cuh), for tests that run without a GPU: the same constants
// (host::tree_consts), the same sources-first renumbering, node expansion with
// its bound (expand_child), the leaf re-test (node_lower_bound), the leaf
// window (node_to_window) and the leaf enumeration with its tie rule
// (leaf_combos, LaneBest), walked depth first on one CPU thread.  Pruning is
// strict, so any order of the nodes gives the same optimum as the kernels'
// breadth-first levels.  Test infrastructure only; the library never runs this.
#include <algorithm>
#include <cstdint>
#include <cstring>
#include <vector>

#define __device__
#define __host__
#define __forceinline__ inline
using std::max;
using std::min;
static inline int __popc(unsigned x) { return __builtin_popcount(x); }
static inline int __ffs(unsigned x) { return __builtin_ffs((int)x); }
static inline int __clz(unsigned x) { return x ? __builtin_clz(x) : 32; }
static inline unsigned long long __umul64hi(unsigned long long a, unsigned long long b) {
  return (unsigned long long)(((unsigned __int128)a * b) >> 64);
}
struct HostDim {
  unsigned x;
};
static HostDim threadIdx{0}, blockDim{1};

#include "../paper_2607_22242_gb300/csrc/bf_tree.cuh"

using namespace bfk;

namespace {

template <int NW>
struct Search {
  const TablesW& tb;
  const TreeConsts& tc;
  SmemTablesW sd;
  std::vector<uint32_t> rt;
  TablesT<NW> tw;
  SmemTablesT<NW> sdw;
  std::vector<uint32_t> rtw, ef, node, slot;
  uint32_t bound;
  unsigned long long best_ms = ~0ull, best_idx = ~0ull, nodes = 0, leaves = 0;
  // Leaf nodes are reduced as the leaf kernel reduces its lanes: 32
  // consecutive ones through LaneBest::offer (the warp's shuffle tree and
  // the block's loop), then into the record by canonical index.
  LaneBest group;
  uint32_t in_group = 0;

  Search(const TablesW& t, const TreeConsts& c, uint32_t b)
      : tb(t), tc(c), rt(ReadyTable<kTreeSlots>::size), rtw(ReadyTable<NW>::size), ef(kTreeSlots),
        node(NodeWords<kTreeSlots>::value), slot(LaneWords<NW>::value), bound(b) {
    threadIdx.x = 0;
    load_smem_tables(tb, sd);
    fill_ready_table<kTreeSlots>(tb, rt.data());
    host::build_window(tb, tc.W0, &tw);
    load_smem_tables(tw, sdw);
    fill_ready_table<NW>(tw, rtw.data());
  }

  // A leaf-level node: the leaf kernel's re-test against the current bound,
  // then every combination of the last D tools (one node per "lane").
  void leaf(const State<kTreeSlots>& s, Digits dg) {
    store_node(s, dg, node.data(), 1u, 0u);
    if (tc.prune && node_lower_bound(node.data(), 1u, 0u, tb, tc, dg, tb.all_mask >> tc.D) > (uint64_t)bound) return;
    node_to_window<NW>(node.data(), 1u, 0u, tc.W0, tw.n, slot.data(), 1u);
    const uint32_t ncomb = tc.alone_last ? tc.combos / tc.radix : tc.combos;
    LaneBest lb;
    leaf_combos<NW>(tw, sdw, rtw.data(), tc, slot.data(), 1u, dg, true, 0u, ncomb, lb);
    leaves += ncomb * (tc.alone_last ? tc.radix : 1u);
    group.offer(lb.ms, lb.dg, tc.tie_pow3());
    if (++in_group == 32u) flush();
  }

  void flush() {
    const LaneBest b = group;
    group = LaneBest{};
    in_group = 0;
    if (b.ms == kInfeasible) return;
    bound = min(bound, b.ms);
    const unsigned long long idx = index_of(b.dg, tc.pow3);
    if (b.ms < best_ms || (b.ms == best_ms && idx < best_idx)) {
      best_ms = b.ms;
      best_idx = idx;
    }
  }

  void visit(const State<kTreeSlots>& s, Digits dg, uint32_t d) {
    ++nodes;
    if (d == tc.leaf_level) {
      leaf(s, dg);
      return;
    }
    for (uint32_t a = 0; a < tc.radix; ++a) {
      State<kTreeSlots> c = s;
      Digits cd = dg;
      if (expand_child<kTreeSlots>(tb, sd, rt.data(), tc, c, cd, d, a, bound, ef.data(), 1u)) visit(c, cd, d + 1);
    }
  }
};

template <int NW>
void run_search(const TablesW& tb, const TreeConsts& tc, uint32_t bound, unsigned long long* out) {
  Search<NW> sr(tb, tc, bound);
  State<kTreeSlots> s;
  init_state(s, tb.all_mask);
  sr.visit(s, Digits{0u, 0u}, 0u);
  sr.flush();
  out[0] = sr.best_ms;
  out[1] = sr.best_idx;
  out[2] = sr.nodes;
  out[3] = sr.leaves;
}

}  // namespace

// bf_search_tree's search over the space of radix `space` (2 or 3), starting
// from the incumbent makespan `bound` (0xFFFFFFFF: none), pruned or not.
// out[0..5] = best makespan (~0: none), its canonical index, nodes visited,
// leaf mappings simulated, renumbered (0/1), the leaf window width.
extern "C" int host_tree(const bf_scenario_desc* d, uint32_t space, uint32_t prune, uint32_t bound,
                         unsigned long long* out) {
  if (d->n < 1 || d->n > 32 || (space != 2 && space != 3)) return -1;
  TablesW t0, rt;
  host::build_tables(d, &t0);
  const bool relabeled = host::relabel_sources_first(t0, &rt);
  const TablesW& tb = relabeled ? rt : t0;
  TreeConsts tc;
  host::tree_consts(tb, space, prune != 0u, &tc);
  const uint32_t nw = tb.n - tc.W0;
  out[4] = relabeled ? 1u : 0u;
#define BF_TRY(NW)                            \
  if (nw <= (uint32_t)NW) {                   \
    out[5] = NW;                              \
    run_search<NW>(tb, tc, bound, out);       \
    return 0;                                 \
  }
  BF_TREE_BUCKETS(BF_TRY)
#undef BF_TRY
  return -1;
}
