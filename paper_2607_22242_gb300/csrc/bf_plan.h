// bf_plan.h -- host-side preparation of a scenario for the kernels: the
// device-format tables (per-tool work in 1/1024 units, successor masks, the
// per-k reciprocals of the slowdown table), the prefix/suffix split of the
// mapping index and the suffix window (see bfk::Plan in bf_sim.cuh).
// Host code only; no CUDA calls.
#pragma once

#include <stdint.h>

#include <algorithm>
#include <cstring>

#include "../../include/bf.h"
#include "bf_lanetree.cuh"
#include "bf_sim.cuh"

namespace bfk {
namespace host {

inline uint64_t pow3(uint32_t n) {
  uint64_t p = 1;
  for (uint32_t i = 0; i < n; ++i) p *= 3;
  return p;
}

// Tables of capacity CAP >= n (kMaxTools for the enumerating searches, 32 for
// the tree search and wide index lists).
template <int CAP>
inline void build_tables(const bf_scenario_desc* d, bfk::TablesT<CAP>* t) {
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
    t->orig[v] = v;
    if (d->vram_mib[v] > d->vram_budget_mib) t->big_mask |= 1u << v;
  }
  for (uint32_t k = 1; k <= (uint32_t)CAP; ++k) {
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

// Number of mid tools M of the pruned search's split (bf_search_pruned):
// more mid tools than the search's 4 leave fewer, shorter prefixes to filter.
inline uint32_t mid_tools(uint32_t n) {
  if (n >= 13) return 6;   // 729 combinations: 23 rounds of 32 lanes, 1% idle
  if (n >= 9) return 5;    // 243 combinations
  if (n >= 4) return 4;    // 81 combinations
  return n;
}

// Tools that are certainly done when the first tool of [from, n) becomes
// ready: the common ancestors of the "sources" of that range (tools >= from
// whose predecessors are all < from); the first tool of the range to become
// ready is one of them.
template <typename TB>
inline uint32_t done_when_first_ready(const uint32_t* anc, const TB& t, uint32_t from) {
  const uint32_t below = (from >= 32) ? ~0u : ((1u << from) - 1u);
  uint32_t done = below;
  for (uint32_t v = from; v < t.n; ++v)
    if ((t.pred[v] & ~below) == 0u) done &= anc[v];
  return done;
}

// Lowest tool not certainly done when the first tool of [P, n) becomes ready:
// the window start for a prefix of P tools.
template <typename TB>
inline uint32_t window_of(const uint32_t* anc, const TB& t, uint32_t P) {
  const uint32_t d = done_when_first_ready(anc, t, P);
  uint32_t w0 = 0;
  while (w0 < P && (d & (1u << w0))) ++w0;
  return w0;
}

// Forward pass on the mapping that runs every tool on its isolated-faster
// device (min(c, g + x)) with no contention and no VRAM limit: a tool becomes
// ready when its last predecessor ends.  Durations are >= 1 us, so every edge
// goes from an earlier to a strictly later ready time.
template <typename TB>
inline void ready_estimate(const TB& t, uint64_t* ready, uint64_t* fin) {
  for (uint32_t v = 0; v < t.n; ++v) {
    uint64_t r = 0;
    for (uint32_t u = 0; u < v; ++u)
      if ((t.pred[v] >> u) & 1u) r = fin[u] > r ? fin[u] : r;
    const uint64_t gpu = t.wnow[v] / 1024u;
    ready[v] = r;
    fin[v] = r + (t.cpu[v] < gpu ? t.cpu[v] : gpu);
  }
}

// R[from] (from in [0, n]): an estimate of how many tools have retired at the
// first instant a tool of [from, n) becomes ready, on the ready_estimate
// mapping; a tool ending at that instant counts as retired (retirement comes
// before admission).  Used only to choose the split: every plan enumerates the
// same mappings with the same results.
template <typename TB>
inline void retired_estimate(const TB& t, uint32_t* R) {
  const uint32_t n = t.n;
  uint64_t ready[BF_MAX_TOOLS], fin[BF_MAX_TOOLS];
  ready_estimate(t, ready, fin);
  for (uint32_t from = 0; from < n; ++from) {
    uint64_t first = ~0ull;
    for (uint32_t v = from; v < n; ++v) first = ready[v] < first ? ready[v] : first;
    uint32_t retired = 0;
    for (uint32_t u = 0; u < from; ++u) retired += fin[u] <= first ? 1u : 0u;
    R[from] = retired;
  }
  R[n] = n;
}

// Tables of the scenario's tools renumbered with the sources (tools without
// predecessors) first, each group in the scenario's order.  A topological
// order, and one that changes no result of the model: its only dependence on
// numbering is the queue's tie between tools that became ready at the same
// instant, and a source (ready at time 0) never ties with a tool that has a
// predecessor (ready only after it has run for at least 1 us), while each
// group keeps its order.  A late source then settles in the prefix instead of leaving the
// window open from time 0 (layered DAGs with sources in later layers: 16
// tools 3.38 -> 2.66 ms, 20 tools 1234 -> 245 ms; 4096 layered 10-tool DAGs
// 11 % faster; tree search of a 28-tool layered DAG 217 -> 0.98 s).  For
// searches over the whole space only (the mapping index of
// a renumbered prefix is not a contiguous range).  Returns false, with *r a
// copy of t, when the order is the scenario's own.
template <int CAP>
inline bool relabel_sources_first(const bfk::TablesT<CAP>& t, bfk::TablesT<CAP>* r) {
  const uint32_t n = t.n;
  uint32_t order[CAP], pos[CAP], k = 0;
  for (uint32_t v = 0; v < n; ++v)
    if (t.pred[v] == 0u) order[k++] = v;
  for (uint32_t v = 0; v < n; ++v)
    if (t.pred[v] != 0u) order[k++] = v;
  *r = t;
  bool same = true;
  for (uint32_t j = 0; j < n; ++j) {
    pos[order[j]] = j;
    same = same && order[j] == j;
  }
  if (same) return false;
  auto remap = [&](uint32_t mask) {
    uint32_t out = 0;
    for (uint32_t u = 0; u < n; ++u)
      if ((mask >> u) & 1u) out |= 1u << pos[u];
    return out;
  };
  for (uint32_t j = 0; j < n; ++j) {
    const uint32_t v = order[j];
    r->pred[j] = remap(t.pred[v]);
    r->succ[j] = remap(t.succ[v]);
    r->cpu[j] = t.cpu[v];
    r->wnow[j] = t.wnow[v];
    r->wq[j] = t.wq[v];
    r->vram[j] = t.vram[v];
    r->orig[j] = t.orig[v];
  }
  r->big_mask = remap(t.big_mask);
  r->relabeled = 1;
  return true;
}

// Ancestor masks of every tool (anc[v] = all tools with a path to v).
template <typename TB>
inline void ancestors(const TB& t, uint32_t* anc) {
  for (uint32_t v = 0; v < t.n; ++v) {
    anc[v] = t.pred[v];
    for (uint32_t u = 0; u < v; ++u)
      if (t.pred[v] & (1u << u)) anc[v] |= anc[u];
  }
}

// The plan for M mid tools: the inner level I, P = n - M - I prefix tools,
// the window start W0, the pruning tails and the lone last tool's durations;
// the window tables (tools [W0, n) renumbered from 0) are filled too.  anc:
// ancestor masks; R: retired_estimate.
inline void plan_for(const bfk::Tables& t, const uint32_t* anc, const uint32_t* R, uint32_t M, bool allow_apart,
                     bfk::Plan* pl, bfk::Tables* w) {
  const uint32_t n = t.n;
  // The inner level: the last I tools, whose modes each lane runs from a
  // second snapshot taken when the first of them can become ready; it pays
  // when that snapshot comes after most of the events.  With R:
  //  - every other tool has ended when the last one can start (R[n-1] =
  //    n-1): I = 1, and the kernels end the last tool in closed form
  //    whenever it runs alone;
  //  - the snapshot would settle fewer than 2 tools: no inner level;
  //  - otherwise I = 1, or 2 when the earlier snapshot of two inner tools
  //    settles as many tools and keeps the same window, which shares the
  //    events before it among 9 mappings instead of 3.
  // Full search of the 16-tool layered workload: I = 2 3.4 ms, I = 1
  // 5.6 ms, I = 0 11.9 ms.
  uint32_t I = 0;
  if (n >= M + 1) {
    if (R[n - 1] + 1u == n) {
      I = 1;
    } else if (R[n - 1] >= 2u) {
      I = 1;
      if (n >= M + 2 && R[n - 2] >= R[n - 1] &&
          window_of(anc, t, n - M - 2) == window_of(anc, t, n - M - 1))
        I = 2;
    }
  }
  const uint32_t P = n - M - I;
  const uint32_t w0 = window_of(anc, t, P);
  std::memset(pl, 0, sizeof *pl);
  pl->P = P;
  pl->M = M;
  pl->I = I;
  pl->W0 = w0;
  // Lower-bound tails: no mode runs a tool faster than min(c, g + x) (GPU
  // contention and the queue only slow it), and a tool starts after all its
  // predecessors end, so a tool not started by time T finishes the whole
  // mapping no earlier than T + tail[tool].
  uint64_t tail[BF_MAX_TOOLS] = {0};
  for (int v = (int)n - 1; v >= 0; --v) {
    const uint64_t gpu = t.wnow[v] / 1024u;
    const uint64_t dmin = t.cpu[v] < gpu ? t.cpu[v] : gpu;
    uint64_t longest = 0;
    for (uint32_t s = (uint32_t)v + 1; s < n; ++s)
      if ((t.succ[v] >> s) & 1u) longest = tail[s] > longest ? tail[s] : longest;
    tail[v] = dmin + longest;
  }
  uint64_t tp = 0, tq = 0;
  for (uint32_t v = P; v < n; ++v) tp = tail[v] > tp ? tail[v] : tp;
  for (uint32_t v = n - I; v < n; ++v) tq = tail[v] > tq ? tail[v] : tq;
  pl->tail_p = (uint32_t)(tp < 0xFFFFFFFFull ? tp : 0xFFFFFFFFull);
  pl->tail_q = (uint32_t)(tq < 0xFFFFFFFFull ? tq : 0xFFFFFFFFull);
  pl->bound = 0xFFFFFFFFu;
  {
    const uint32_t last = n - 1;
    const bool fits = t.vram[last] <= t.budget;
    pl->alone[0] = t.cpu[last];
    pl->alone[1] = fits ? t.wnow[last] / 1024u : 0xFFFFFFFFu;
    pl->alone[2] = fits ? t.wq[last] / 1024u : 0xFFFFFFFFu;
  }
  pl->pow3P = (uint32_t)pow3(P);
  pl->pow3M = (uint32_t)pow3(M);
  pl->pow3I = (uint32_t)pow3(I);
  pl->relabeled = t.relabeled;
  for (uint32_t v = 0; v < n; ++v) pl->pv[v] = (uint32_t)pow3(t.orig[v]);
  pl->pvA = I >= 1 ? pl->pv[n - I] : 0u;
  pl->pvB = I >= 2 ? pl->pv[n - I + 1] : 0u;
  // The last tool leaves the window when it waits for all others and that
  // lowers the compiled width (19-tool fan-out DAG: 8 -> 7 slots, 17.0 ->
  // 15.8 ms; at an unchanged width it measured 1 % slower).
  const uint32_t others = n >= 2 ? (1u << (n - 1)) - 1u : 0u;
  pl->last_apart = (allow_apart && I == 1 && anc[n - 1] == others && n - w0 >= 2 &&
                    bucket_for(n - w0 - 1) < bucket_for(n - w0))
                       ? 1u
                       : 0u;
  std::memset(w, 0, sizeof *w);
  const uint32_t nw = n - w0 - pl->last_apart;
  w->n = nw;
  w->budget = t.budget;
  w->all_mask = (1u << nw) - 1u;
  w->big_mask = t.big_mask >> w0;
  for (uint32_t j = 0; j < nw; ++j) {
    w->pred[j] = t.pred[w0 + j] >> w0;
    w->succ[j] = t.succ[w0 + j] >> w0;
    w->cpu[j] = t.cpu[w0 + j];
    w->wnow[j] = t.wnow[w0 + j];
    w->wq[j] = t.wq[w0 + j];
    w->vram[j] = t.vram[w0 + j];
    w->orig[j] = t.orig[w0 + j];
  }
  w->relabeled = t.relabeled;
  for (uint32_t k = 0; k <= (uint32_t)bfk::kMaxTools; ++k) {
    w->f[k] = t.f[k];
    w->fshift[k] = t.fshift[k];
    w->fmagic[k] = t.fmagic[k];
  }
}

// Plan of a scenario for the kernels whose lanes own prefixes (searches,
// evaluation, branch and bound).  M = 4 mid tools: a longer prefix settles
// more of the DAG in each lane's own simulation and often starts the window
// later (fewer slots per event).  When the last tool waits for every other
// one (it then ends in closed form and a mapping costs little beyond its mid
// run), M = 5 if that keeps the window and still leaves P >= 12 prefix tools
// (3^12 prefixes, many warps per SM): the prefix simulation, which is as long
// as the prefix, is shared by 3x more mappings.  Full searches, ms
// (M = 6 / 5 / 4): 19-tool fan-out DAG 17.28 / 16.99 / 17.32; random
// 20-tool DAG 412 / 416 / 362; layered 17 and 18 tools 14.8 / 14.9 / 13.5
// and 49.3 / 49.9 / 42.0; segmented 17, 18 and 20 tools 3.66 / 3.78 / 2.98,
// 3.43 / 2.49 / 1.69 and 14.1 / 10.8 / 10.8; 16-tool layered 3.40 / 3.51 /
// 3.32.
inline void split_and_window(const bfk::Tables& t, bfk::Plan* pl, bfk::Tables* w) {
  const uint32_t n = t.n;
  uint32_t anc[BF_MAX_TOOLS] = {}, R[BF_MAX_TOOLS + 1] = {};
  ancestors(t, anc);
  retired_estimate(t, R);
  plan_for(t, anc, R, n < 4 ? n : 4, true, pl, w);
  const uint32_t others = n >= 2 ? (1u << (n - 1)) - 1u : 0u;
  if (n >= 18 && pl->I == 1 && anc[n - 1] == others) {
    bfk::Plan p5;
    bfk::Tables w5;
    plan_for(t, anc, R, 5, true, &p5, &w5);
    if (p5.W0 == pl->W0 && p5.I == 1) {
      *pl = p5;
      *w = w5;
    }
  }
}

// Whether a renumbered split (tables rt, plan rp, window rw) should replace
// the scenario-numbered one (t, p, w): its prefix snapshot settles more tools
// (estimated), its window is narrower, or it has a deeper inner level.  The
// renumbered kernels compute canonical indices from tables, which costs a few
// per cent when the split gains nothing (a 17-tool layered DAG whose sources
// moved without changing the split: +9 %).
inline bool renumbering_helps(const bfk::Tables& t, const bfk::Plan& p, const bfk::Tables& w, const bfk::Tables& rt,
                              const bfk::Plan& rp, const bfk::Tables& rw) {
  uint32_t R[BF_MAX_TOOLS + 1], RR[BF_MAX_TOOLS + 1];
  retired_estimate(t, R);
  retired_estimate(rt, RR);
  return RR[rp.P] > R[p.P] || bucket_for(rw.n) < bucket_for(w.n) || rp.I > p.I;
}

// Plan of bf_search_pruned: mid_tools(n) mid tools, so that fewer, shorter
// prefixes go through its prefix filter (19-tool fan-out DAG: 0.26 ms with
// 3^12 prefixes, 0.52 ms with 3^13).
inline void split_and_window_pruned(const bfk::Tables& t, bfk::Plan* pl, bfk::Tables* w) {
  uint32_t anc[BF_MAX_TOOLS] = {}, R[BF_MAX_TOOLS + 1] = {};
  ancestors(t, anc);
  retired_estimate(t, R);
  plan_for(t, anc, R, mid_tools(t.n), true, pl, w);
}

// Lowest tool not certainly done when the first tool of [from, n) becomes ready.
template <typename TB>
inline uint32_t window_start(const TB& t, uint32_t from) {
  uint32_t anc[32] = {};
  ancestors(t, anc);
  return window_of(anc, t, from);
}

// Tables of tools [w0, n) renumbered from 0, in a table of capacity NW >= n - w0.
template <int NW, int CAP>
inline void build_window(const bfk::TablesT<CAP>& t, uint32_t w0, bfk::TablesT<NW>* w) {
  std::memset(w, 0, sizeof *w);
  const uint32_t nw = t.n - w0;
  w->n = nw;
  w->budget = t.budget;
  w->all_mask = nw >= 32 ? ~0u : ((1u << nw) - 1u);
  w->big_mask = t.big_mask >> w0;
  for (uint32_t j = 0; j < nw; ++j) {
    w->pred[j] = t.pred[w0 + j] >> w0;
    w->succ[j] = t.succ[w0 + j] >> w0;
    w->cpu[j] = t.cpu[w0 + j];
    w->wnow[j] = t.wnow[w0 + j];
    w->wq[j] = t.wq[w0 + j];
    w->vram[j] = t.vram[w0 + j];
    w->orig[j] = t.orig[w0 + j];
  }
  w->relabeled = t.relabeled;
  for (uint32_t k = 0; k <= (uint32_t)NW; ++k) {
    w->f[k] = t.f[k];
    w->fshift[k] = t.fshift[k];
    w->fmagic[k] = t.fmagic[k];
  }
}

// Restrict a scenario's plan to canonical indices [first, first+count),
// count >= 1, and split its work into warp tasks: prefix groups of 32 times
// chunks of mid combinations, about `target_tasks` tasks in all.  Each task
// re-simulates its lanes' prefixes; the mid combinations are split only when
// there are fewer prefix groups than target tasks, i.e. when prefixes are
// few and short, so chunks go down to one combination (8- and 12-tool
// searches: 0.063 -> 0.034 ms and 0.158 -> 0.061 ms against chunks of at
// least 16; no change on larger workloads).
inline bfk::Plan make_plan(const bfk::Plan& base, uint64_t first, uint64_t count, uint64_t target_tasks) {
  bfk::Plan pl = base;
  const uint64_t last = first + count - 1;
  pl.first = (uint32_t)first;
  pl.last = (uint32_t)last;
  const uint64_t pm = (uint64_t)pl.pow3P * pl.pow3M;
  pl.i_lo = (uint32_t)(first / pm);
  pl.i_hi = (uint32_t)(last / pm);
  const uint64_t s_lo = first / pl.pow3P, s_hi = last / pl.pow3P;  // s = m + 3^M i
  if (s_lo == s_hi) {
    pl.p_lo = (uint32_t)(first % pl.pow3P);
    pl.p_hi = (uint32_t)(last % pl.pow3P);
  } else {
    pl.p_lo = 0;
    pl.p_hi = pl.pow3P - 1;
  }
  if (s_lo / pl.pow3M == s_hi / pl.pow3M) {
    pl.m_lo = (uint32_t)(s_lo % pl.pow3M);
    pl.m_hi = (uint32_t)(s_hi % pl.pow3M);
  } else {
    pl.m_lo = 0;
    pl.m_hi = pl.pow3M - 1;
  }
  pl.groups = (pl.p_hi - pl.p_lo) / 32 + 1;
  const uint64_t num_m = (uint64_t)pl.m_hi - pl.m_lo + 1;
  uint64_t parts = (target_tasks + pl.groups - 1) / pl.groups;
  if (parts > num_m) parts = num_m;
  if (parts < 1) parts = 1;
  pl.m_chunk = (uint32_t)((num_m + parts - 1) / parts);
  pl.m_parts = (uint32_t)((num_m + pl.m_chunk - 1) / pl.m_chunk);
  pl.full = (first == 0 && last + 1 == (uint64_t)pl.pow3P * pl.pow3M * pl.pow3I) ? 1u : 0u;
  return pl;
}

// Warp tasks a single-scenario search is cut into (make_plan): several waves
// of the GPU's resident warps, so that uneven tasks even out.
constexpr uint64_t kSearchTasks = 32768;

// Whole-space searches on the search kernel (bf_search_best and
// bf_search_range over the whole space, bf_search_pruned) run on the tables
// renumbered with the sources first when that gives a better split
// (renumbering_helps); otherwise on t0 with its own split p0 and window w0.
// split: split_and_window, or the pruned search's split.
template <typename Split>
inline void whole_space_tables(const bfk::Tables& t0, const bfk::Plan& p0, const bfk::Tables& w0, Split split,
                               bfk::Tables* tb, bfk::Plan* plan, bfk::Tables* tw) {
  bfk::Tables rt, rw;
  bfk::Plan rp;
  if (relabel_sources_first(t0, &rt)) {
    split(rt, &rp, &rw);
    if (renumbering_helps(t0, p0, w0, rt, rp, rw)) {
      *tb = rt;
      *plan = rp;
      *tw = rw;
      return;
    }
  }
  *tb = t0;
  *plan = p0;
  *tw = w0;
}

// Mappings a block of the lane-tree batch kernel aims to search (a 10-tool
// scenario gets ceil(3^10 / 7381) = 9 blocks), and the fewest roots a block
// hands out (two per lane of 256).  Many short blocks keep every SM busy to
// the end of the launch: 4096 x 3^10 batch call, an earlier form of the
// kernel, from 16.2 ms at one block per scenario (1024+ roots) to 14.8 ms at
// 9 and 18.0 ms at 32 (128+); the current kernel at 7, 9, 12 and 16 blocks
// per scenario 13.5, 13.4, 13.6 and 13.8 ms, at 9 blocks with 256+ roots
// 13.4 ms.
constexpr uint64_t kLtBlockMappings = 7381;
constexpr uint64_t kLtMinRootsPerBlock = 512;
// Blocks one scenario of a batch gets at most: with 512 roots per block this
// keeps the roots of a 16-tool scenario at 12 tools (as its full search over
// the whole GPU takes them) instead of 14, and a 20-tool one's at 12 instead
// of 18 (472,000 blocks).  Scenarios of up to 14 tools stay below it.
constexpr uint64_t kLtMaxBlocksPerScenario = 1024;

// The levels of the lane-tree search of one scenario (n <= kLtMaxTools):
// roots [0, x), then [x, y), then [y, n).  Each level below the root holds at
// most kLtPartTools tools (its combinations come from one table), and the
// root at most kLtRootParts * kLtPartTools, with 3^x >= min_roots.  Among
// those, the split with the fewest estimated events: with R[b] the tools
// retired when the first tool >= b can become ready (retired_estimate), a
// root simulates about R[x] events, a level-1 job R[y] - R[x] and a level-2
// job n - R[y]; each job also costs about half an event to set up.  4096
// layered 10-tool DAGs (48 checked by enumeration): 2.9 events per mapping
// against 2.8 for the best split and 4.1 for the prefix/mid/inner split of
// the other batch kernel.
template <typename TB>
inline double lanetree_levels(const TB& t, uint64_t min_roots, uint32_t* x_out, uint32_t* y_out) {
  const uint32_t n = t.n;
  uint32_t R[BF_MAX_TOOLS + 1] = {};
  retired_estimate(t, R);
  uint32_t xmin = 0;
  while (xmin < n && pow3(xmin) < min_roots) ++xmin;
  if (n > 2u * kLtPartTools && xmin < n - 2u * kLtPartTools) xmin = n - 2u * kLtPartTools;
  double best = -1.0;
  uint32_t bx = n, by = n;
  for (uint32_t x = xmin; x <= n && x <= kLtRootParts * kLtPartTools; ++x) {
    for (uint32_t y = (x == n ? n : x + 1u); y <= n; ++y) {
      if (y - x > kLtPartTools || n - y > kLtPartTools) continue;
      const double px = (double)pow3(x), py = (double)pow3(y), pn = (double)pow3(n);
      const double cost = px * R[x] + py * (R[y] - R[x]) + pn * (n - R[y]) + 0.5 * (px + (y < n ? py : 0.0));
      if (best < 0.0 || cost < best) {
        best = cost;
        bx = x;
        by = y;
      }
    }
  }
  *x_out = bx;
  *y_out = by;
  return best;
}

// The batch's levels (every block gets kLtMinRootsPerBlock roots or more)
// and the blocks its scenario's roots are split over.
template <typename TB>
inline void lanetree_split(const TB& t, uint32_t* x_out, uint32_t* y_out, uint32_t* nblocks) {
  uint64_t want_blocks = (pow3(t.n) + kLtBlockMappings - 1) / kLtBlockMappings;
  if (want_blocks > kLtMaxBlocksPerScenario) want_blocks = kLtMaxBlocksPerScenario;
  lanetree_levels(t, kLtMinRootsPerBlock * want_blocks, x_out, y_out);
  const uint64_t cap = pow3(*x_out) / kLtMinRootsPerBlock;
  uint64_t nb = want_blocks < cap ? want_blocks : cap;
  *nblocks = (uint32_t)(nb < 1 ? 1 : nb);
}

// Sampled work of a one-scenario lane-tree search, for choosing its levels.
// A whole-GPU search runs millions of jobs per level, so its levels are
// worth a closer estimate than the batch's: the closed-form estimate of
// lanetree_levels took one level of 4 tools below roots of 12 for the
// 16-tool layered workload (2.37 events and 0.60 jobs per mapping on the
// host emulator, 1.67 ms), where one tool and then 3 take 2.17 and 0.63
// (1.59 ms).
//
// lt_sample_events simulates one mapping (mode[t] per tool of the record's
// numbering) with the model's arithmetic in 64-bit integers and returns, for
// every b in [0, n], ev[b] = the events before the first tool >= b becomes
// ready (all its events if none does) and reached[b] = whether one does
// (the mapping has not been found infeasible before).  Estimates only: no
// result depends on them.
inline void lt_sample_events(const bfk::LaneTreeRecord& r, const uint8_t* mode, uint32_t* ev, bool* reached) {
  const uint32_t n = r.n;
  uint32_t first[bfk::kLtMaxTools];
  uint64_t end[bfk::kLtMaxTools];  // CPU: real end; GPU: end stamp on the virtual clock
  uint32_t fifo[bfk::kLtMaxTools], qhead = 0, qtail = 0;
  uint32_t cpu = 0u, now = 0u, que = 0u;  // the modes as tool sets
  for (uint32_t t = 0; t < n; ++t) {
    first[t] = 0xFFFFFFFFu;
    cpu |= mode[t] == 0 ? 1u << t : 0u;
    now |= mode[t] == 1 ? 1u << t : 0u;
    que |= mode[t] == 2 ? 1u << t : 0u;
  }
  uint32_t pend = r.all_mask, run = 0u, done = 0u;
  uint64_t T = 0, V = 0, vram = 0;
  uint32_t events = 0;
  bool dead = false;
  for (;;) {
    uint32_t ready = 0u;
    for (uint32_t m = pend; m; m &= m - 1u) {
      const uint32_t t = (uint32_t)__builtin_ctz(m);
      if ((r.pred[t] & ~done) == 0u) ready |= 1u << t;
    }
    pend &= ~ready;
    for (uint32_t m = ready; m; m &= m - 1u) {
      const uint32_t t = (uint32_t)__builtin_ctz(m);
      first[t] = events;
      if ((que >> t) & 1u) {
        fifo[qtail++] = t;
      } else {
        end[t] = (cpu >> t) & 1u ? T + r.dur[0][t] : V + r.dur[1][t];
        vram += (now >> t) & 1u ? r.vram[t] : 0u;
        run |= 1u << t;
      }
    }
    if ((ready & now) && vram > r.budget) {
      dead = true;
      break;
    }
    if (qhead < qtail && !(run & que)) {
      const uint32_t h = fifo[qhead];
      if ((r.big_mask >> h) & 1u) {
        dead = true;
        break;
      }
      if (vram + r.vram[h] <= r.budget) {
        end[h] = V + r.dur[2][h];
        vram += r.vram[h];
        run |= 1u << h;
        ++qhead;
      }
    }
    if (!run) break;  // every tool has ended
    uint32_t k = 0;
    uint64_t tc = ~0ull, gm = ~0ull;
    for (uint32_t m = run; m; m &= m - 1u) {
      const uint32_t t = (uint32_t)__builtin_ctz(m);
      if ((cpu >> t) & 1u) {
        tc = end[t] < tc ? end[t] : tc;
      } else {
        ++k;
        gm = end[t] < gm ? end[t] : gm;
      }
    }
    const uint64_t f = r.f[k ? k : 1];
    const uint64_t tg = k ? T + (((gm - V) * f + 0xFFFFFull) >> 20) : ~0ull;
    const bool gpu_event = k && tg <= tc;
    if (gpu_event) {
      T = tg;
      V = gm;
    } else {
      if (k) V += ((tc - T) << 20) / f;
      T = tc;
    }
    ++events;
    for (uint32_t m = run; m; m &= m - 1u) {
      const uint32_t t = (uint32_t)__builtin_ctz(m);
      const bool ends = (cpu >> t) & 1u ? end[t] == T : (gpu_event && end[t] == V);
      if (ends) {
        run &= ~(1u << t);
        done |= 1u << t;
        vram -= (cpu >> t) & 1u ? 0u : r.vram[t];
      }
    }
  }
  uint32_t earliest = 0xFFFFFFFFu;
  ev[n] = events;
  reached[n] = !dead;
  for (uint32_t b = n; b-- > 0;) {
    earliest = first[b] < earliest ? first[b] : earliest;
    reached[b] = earliest != 0xFFFFFFFFu;
    ev[b] = reached[b] ? earliest : events;
  }
}

// Levels of a one-scenario record from kLtLevelSamples mappings drawn
// uniformly (a fixed seed: the same choice on every machine), for records the
// search will run (about 0.1 ms of host time at 16 tools): among the
// splits lanetree_levels allows, the one of least sampled cost -- a root
// runs its mappings' events up to ev[x], a level-1 job up to ev[y] from
// there, a leaf to the end, and a job costs half an event more; jobs exist
// only below checkpoints that were reached.
constexpr uint32_t kLtLevelSamples = 128;
inline void lanetree_sampled_levels(const bfk::LaneTreeRecord& r, uint64_t min_roots, uint32_t* x_out,
                                    uint32_t* y_out) {
  const uint32_t n = r.n;
  uint64_t S[bfk::kLtMaxTools + 1] = {}, A[bfk::kLtMaxTools + 1] = {};
  uint64_t state = 0x9E3779B97F4A7C15ull;
  uint8_t mode[bfk::kLtMaxTools];
  uint32_t ev[bfk::kLtMaxTools + 1];
  bool reached[bfk::kLtMaxTools + 1];
  for (uint32_t k = 0; k < kLtLevelSamples; ++k) {
    for (uint32_t t = 0; t < n; ++t) {  // splitmix64 (Steele, Lea and Flood, OOPSLA 2014)
      uint64_t z = (state += 0x9E3779B97F4A7C15ull);
      z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
      z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
      mode[t] = (uint8_t)((z ^ (z >> 31)) % 3u);
    }
    lt_sample_events(r, mode, ev, reached);
    for (uint32_t b = 0; b <= n; ++b) {
      S[b] += ev[b];
      A[b] += reached[b] ? 1u : 0u;
    }
  }
  uint32_t xmin = 0;
  while (xmin < n && pow3(xmin) < min_roots) ++xmin;
  if (n > 2u * kLtPartTools && xmin < n - 2u * kLtPartTools) xmin = n - 2u * kLtPartTools;
  uint64_t best = ~0ull;
  for (uint32_t x = xmin; x <= n && x <= kLtRootParts * kLtPartTools; ++x) {
    for (uint32_t y = (x == n ? n : x + 1u); y <= n; ++y) {
      if (y - x > kLtPartTools || n - y > kLtPartTools) continue;
      const uint64_t px = pow3(x), py = pow3(y), pn = pow3(n);
      // Twice the cost, summed over the samples (half events are whole).
      const uint64_t cost = 2u * (px * S[x] + py * (S[y] - S[x]) + pn * (S[n] - S[y])) + px * kLtLevelSamples +
                            (x < n ? py * A[x] : 0u) + (y < n ? pn * A[y] : 0u);
      if (cost < best) {
        best = cost;
        *x_out = x;
        *y_out = y;
      }
    }
  }
}

// The tables a lane-tree record's split estimate reads (n, pred, cpu, wnow).
struct LtView {
  uint32_t n;
  uint32_t pred[BF_MAX_TOOLS], cpu[BF_MAX_TOOLS], wnow[BF_MAX_TOOLS];
};

// Record of one scenario of a lane-tree search: its tools renumbered with the
// sources first (each group in the scenario's order: the order of
// relabel_sources_first) and its levels -- the batch's (min_roots == 0), or
// those of a search whose lanes share 3^x >= min_roots roots (nblocks = 1).
// Built straight from the desc; the slowdown constants are those of
// build_tables, taken over from the previous record built on this thread
// when the slowdown table is the same (the scenarios of a batch usually
// share one).  *events (if given) receives the levels' estimated events
// per mapping (lanetree_levels' cost over 3^n).
inline void lanetree_record(const bf_scenario_desc* d, bfk::LaneTreeRecord* r, uint64_t min_roots = 0,
                            double* events = nullptr) {
  const uint32_t n = d->n;
  uint32_t order[BF_MAX_TOOLS], pos[BF_MAX_TOOLS], k = 0;
  for (uint32_t v = 0; v < n; ++v)
    if (d->pred_mask[v] == 0u) order[k++] = v;
  for (uint32_t v = 0; v < n; ++v)
    if (d->pred_mask[v] != 0u) order[k++] = v;
  for (uint32_t j = 0; j < n; ++j) pos[order[j]] = j;
  std::memset(r, 0, sizeof *r);
  r->n = n;
  r->budget = d->vram_budget_mib;
  r->all_mask = (1u << n) - 1u;
  LtView view;
  view.n = n;
  for (uint32_t j = 0; j < n; ++j) {
    const uint32_t v = order[j];
    uint32_t pm = 0u;
    for (uint32_t u = 0; u < v; ++u)
      if ((d->pred_mask[v] >> u) & 1u) pm |= 1u << pos[u];
    r->pred[j] = view.pred[j] = pm;
    r->dur[0][j] = view.cpu[j] = d->cpu_us[v];
    r->dur[1][j] = view.wnow[j] = (d->gpu_us[v] + d->xfer_us[v]) * 1024u;
    r->dur[2][j] = (d->load_us[v] + d->gpu_us[v] + d->xfer_us[v]) * 1024u;
    r->vram[j] = d->vram_mib[v];
    r->pv[j] = (uint32_t)pow3(v);
    if (d->vram_mib[v] > d->vram_budget_mib) r->big_mask |= 1u << j;
  }
  thread_local uint32_t last_f[BF_MAX_TOOLS + 1] = {0};
  thread_local uint32_t last_n = 0;
  thread_local bfk::Tables last;
  if (last_n != n || std::memcmp(last_f, d->slowdown_q10, sizeof last_f) != 0) {
    build_tables(d, &last);
    std::memcpy(last_f, d->slowdown_q10, sizeof last_f);
    last_n = n;
  }
  for (uint32_t j = 0; j <= bfk::kLtMaxTools; ++j) {
    r->f[j] = last.f[j];
    r->fshift[j] = last.fshift[j];
    r->fmagic[j] = last.fmagic[j];
  }
  if (min_roots == 0) {
    lanetree_split(view, &r->x, &r->y, &r->nblocks);
  } else {
    const double cost = lanetree_levels(view, min_roots, &r->x, &r->y);
    r->nblocks = 1;
    if (events) *events = cost / (double)pow3(n);
  }
}

// Whether a full search of a scenario goes to the one-scenario lane-tree
// kernel (record rec, estimated events per mapping lt_events) rather than
// the search kernel (whole-space tables rt, plan rp, window rw).  The search
// kernel's cost per mapping grows with its events per mapping -- R-estimate
// events after its prefix checkpoint shared by 3^(M+I) mappings, its mid
// checkpoint by 3^I -- times its window width (each event scans the window),
// at full warp efficiency when its lanes follow the same structure; the
// lane tree's with its own events per mapping, at the divergence of lanes
// on different mappings.  Measured (full searches, 152-SM GB300): the lane
// tree is faster on every layered and fan-out/fan-in DAG of 12 to 16 tools
// tried (16-tool layered workload 2.70 -> 1.70 ms; layered 14 tools 0.60 ->
// 0.21 ms) and on the chain and spine DAGs of 13 and 14 tools; slower when
// its roots are whole mappings (x = n: the 12-tool fan-out/fan-in 0.053 ->
// 0.081 ms) and on chain and spine DAGs of 15 and 16 tools, whose narrow
// windows (4 to 6 slots) make the search kernel's events cheap (16-tool
// chain 0.67 ms against 0.82): there the search kernel's events x window
// width is 4.4 to 6.8 times the lane tree's estimate, in the cases the lane
// tree wins 6.7 to 21 times.  On 40 further DAGs of 13 to 16 tools (layered,
// sparse, fan-out/fan-in, spines with branches) the rule chose the lane tree
// for all 40, and it was the faster on all 40.
constexpr double kLtPreferRatio = 8.0;
// Above 16 tools the lane tree runs its wide form (5-bit queue entries in two
// words, 55 registers, 4 blocks per SM), whose events cost more: on layered
// DAGs of 17 to 20 tools it won 2.05 to 2.3 times at ratios of 18.4 to 19.8
// (the 24-tool layered workload's first 20 tools 850 -> 363 ms), 1.4 times
// at 17.3, and lost 1.6 times at 12.8; the 19-tool workload's ratio is 6.6.
// On 12 further DAGs of 17 to 19 tools it chose the lane tree for all 12,
// the faster on all 12.
constexpr double kLtPreferRatioWide = 15.0;
inline bool lanetree_preferred(const bfk::Tables& rt, const bfk::Plan& rp, const bfk::Tables& rw,
                               const bfk::LaneTreeRecord& rec, double lt_events) {
  const uint32_t n = rt.n;
  if (rec.x >= n) return false;
  if (n <= 14u) return true;
  uint32_t R[BF_MAX_TOOLS + 1] = {};
  retired_estimate(rt, R);
  const uint32_t P = rp.P, I = rp.I;
  const double sk_events = R[P] / (double)pow3(rp.M + I) + (R[n - I] - R[P]) / (double)pow3(I) + (n - R[n - I]);
  return sk_events * rw.n >= (n > kLtNarrowTools ? kLtPreferRatioWide : kLtPreferRatio) * lt_events;
}

}  // namespace host
}  // namespace bfk
