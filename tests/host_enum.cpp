// Host build of the search kernels' enumeration logic (bf_plan.h, bf_enum.cuh,
// bf_sim.cuh), for tests that run without a GPU: the warp tasks of a plan are
// executed lane by lane on the CPU with the same code the kernels run, and
// every mapping's makespan is stored at its canonical index.  Test
// infrastructure only; the library never runs this.
#include <algorithm>
#include <cstdint>
#include <cstring>
#include <vector>

#define __device__
#define __host__
#define __forceinline__ inline
using std::min;
static inline int __popc(unsigned x) { return __builtin_popcount(x); }
static inline int __ffs(unsigned x) { return __builtin_ffs((int)x); }
static inline unsigned long long __umul64hi(unsigned long long a, unsigned long long b) {
  return (unsigned long long)(((unsigned __int128)a * b) >> 64);
}
struct HostDim {
  unsigned x;
};
static HostDim threadIdx{0}, blockDim{1};

#include "../paper_2607_22242_gb300/csrc/bf_enum.cuh"
#include "../paper_2607_22242_gb300/csrc/bf_plan.h"

using namespace bfk;

namespace {


struct StoreAll {
  uint32_t first;
  uint32_t* out;
  void operator()(uint32_t idx, uint32_t ms) { out[idx - first] = ms; }
};

// Lane states of one emulated warp: [word][lane] as in shared memory, filled
// with garbage first (shared memory holds stale data on the GPU).
struct Lanes {
  std::vector<uint32_t> words;
  explicit Lanes(int lane_words) : words(2u * (uint32_t)lane_words * 32u, 0xA5A5A5A5u) {}
};

template <int NP, int NW, bool RL>
void run_tasks(const Tables& tb, const Tables& tw, const Plan& plan, uint32_t* out) {
  threadIdx.x = 0;
  SmemTables sd, sdw;
  load_smem_tables(tb, sd);
  load_smem_tables(tw, sdw);
  std::vector<uint32_t> rt(ReadyTable<NP>::size), rtw(ReadyTable<NW>::size), mpart(kMaxMidPartWords);
  fill_ready_table<NP>(tb, rt.data());
  fill_ready_table<NW>(tw, rtw.data());
  fill_mid_parts(plan, mpart.data());
  const int lw = LaneWords<NW>::value;
  StoreAll sink{plan.first, out};
  for (uint32_t g = 0; g < plan.groups; ++g)
    for (uint32_t part = 0; part < plan.m_parts; ++part) {
      Lanes lanes(lw);
      for (unsigned lane = 0; lane < 32; ++lane) {
        threadIdx.x = lane;
        warp_task<NP, NW, RL>(tb, sd, rt.data(), tw, sdw, rtw.data(), plan, mpart.data(), g, part,
                              lanes.words.data() + lane, lanes.words.data() + lw * 32 + lane, 32, sink);
      }
    }
}

template <int NW>
void run_width(const Tables& tb, const Tables& tw, const Plan& plan, uint32_t* out) {
  const bool rl = plan.relabeled != 0u;
  if (tb.n <= (uint32_t)NW) {
    if (rl) run_tasks<NW, NW, true>(tb, tw, plan, out);
    else run_tasks<NW, NW, false>(tb, tw, plan, out);
  } else {
    if (rl) run_tasks<kMaxTools, NW, true>(tb, tw, plan, out);
    else run_tasks<kMaxTools, NW, false>(tb, tw, plan, out);
  }
}

}  // namespace

// mode 0: the searches' plan in the scenario's numbering, over [first, first+count).
// mode 1: the whole space, renumbered with the sources first (when that
//         changes the order), as the whole-space searches may run it.
// Slots beyond a window count as done, so a width of 4, 7, 10, 14 or 20 slots
// serves every window up to it (the library compiles every width).
// info[0..5] = P, M, I, W0, window tools, flags (1 renumbered, 2 last tool apart).
extern "C" int host_eval(const bf_scenario_desc* d, uint64_t first, uint64_t count, uint32_t mode, uint32_t* out,
                         uint32_t* info) {
  Tables t0, tb, tw;
  Plan base;
  host::build_tables(d, &t0);
  const uint64_t total = host::pow3(d->n);
  Plan plan;
  if (mode == 0) {
    tb = t0;
    host::split_and_window(tb, &base, &tw);
    plan = host::make_plan(base, first, count, host::kSearchTasks);
  } else {
    if (first != 0 || count != total) return -1;
    if (mode != 1) return -1;
    host::relabel_sources_first(t0, &tb);
    host::split_and_window(tb, &base, &tw);
    plan = host::make_plan(base, first, count, host::kSearchTasks);
  }
  info[0] = plan.P;
  info[1] = plan.M;
  info[2] = plan.I;
  info[3] = plan.W0;
  info[4] = tw.n;
  info[5] = (tb.relabeled ? 1u : 0u) | (plan.last_apart ? 2u : 0u);
  for (uint64_t j = 0; j < count; ++j) out[j] = 0xDEADBEEFu;
  if (tw.n <= 4) run_width<4>(tb, tw, plan, out);
  else if (tw.n <= 7) run_width<7>(tb, tw, plan, out);
  else if (tw.n <= 10) run_width<10>(tb, tw, plan, out);
  else if (tw.n <= 14) run_width<14>(tb, tw, plan, out);
  else run_width<20>(tb, tw, plan, out);
  return 0;
}

// The branch and bound of bf_search_pruned (its plan on the tables it runs
// on, renumbered when that improves the split) with incumbent makespan
// `bound`: pass 1 keeps the prefixes whose checkpoint bound does not exceed
// it, pass 2 enumerates their mappings with the bound at the inner
// checkpoint.  Returns the best key, (makespan << 32) | canonical index.
namespace {
struct MinKey {
  unsigned long long best = ~0ull;
  void operator()(uint32_t idx, uint32_t ms) {
    const unsigned long long k = ((unsigned long long)ms << 32) | idx;
    if (k < best) best = k;
  }
};

template <int NP, int NW>
unsigned long long pruned(const Tables& tb, const Tables& tw, Plan plan) {
  threadIdx.x = 0;
  SmemTables sd, sdw;
  load_smem_tables(tb, sd);
  load_smem_tables(tw, sdw);
  std::vector<uint32_t> rt(ReadyTable<NP>::size), rtw(ReadyTable<NW>::size), mpart(kMaxMidPartWords), surv;
  fill_ready_table<NP>(tb, rt.data());
  fill_ready_table<NW>(tw, rtw.data());
  fill_mid_parts(plan, mpart.data());
  for (uint32_t p = 0; p < plan.pow3P; ++p) {
    Digits dgp;
    uint32_t T = 0;
    if (prefix_checkpoint<NP, NW>(tb, sd, rt.data(), plan, p, &dgp, &T, nullptr, 0u) &&
        (uint64_t)T + plan.tail_p <= plan.bound)
      surv.push_back(p);
  }
  MinKey sink;
  const int lw = LaneWords<NW>::value;
  for (size_t g = 0; g < surv.size(); g += 32) {
    Lanes lanes(lw);
    for (unsigned lane = 0; lane < 32; ++lane) {
      threadIdx.x = lane;
      const bool valid = g + lane < surv.size();
      prefix_task<NP, NW, true>(tb, sd, rt.data(), tw, sdw, rtw.data(), plan, mpart.data(), valid ? surv[g + lane] : 0u,
                                valid, 0u, lanes.words.data() + lane, lanes.words.data() + lw * 32 + lane, 32, sink);
    }
  }
  return sink.best;
}

template <int NW>
unsigned long long pruned_width(const Tables& tb, const Tables& tw, const Plan& plan) {
  return tb.n <= (uint32_t)NW ? pruned<NW, NW>(tb, tw, plan) : pruned<kMaxTools, NW>(tb, tw, plan);
}
}  // namespace

extern "C" unsigned long long host_pruned(const bf_scenario_desc* d, uint32_t bound) {
  Tables t0, w0, tb, tw;
  Plan p0, base;
  host::build_tables(d, &t0);
  host::split_and_window(t0, &p0, &w0);
  host::whole_space_tables(t0, p0, w0, host::split_and_window, &tb, &base, &tw);
  host::split_and_window_pruned(tb, &base, &tw);
  Plan plan = host::make_plan(base, 0, host::pow3(d->n), host::kSearchTasks);
  plan.bound = bound;
  plan.m_lo = 0;
  plan.m_hi = plan.pow3M - 1u;
  plan.m_chunk = plan.pow3M;
  plan.m_parts = 1;
  if (tw.n <= 4) return pruned_width<4>(tb, tw, plan);
  if (tw.n <= 7) return pruned_width<7>(tb, tw, plan);
  if (tw.n <= 10) return pruned_width<10>(tb, tw, plan);
  if (tw.n <= 14) return pruned_width<14>(tb, tw, plan);
  return pruned_width<20>(tb, tw, plan);
}

// A lane-tree search (bf_lanetree.cuh) of one scenario: with min_roots == 0
// the batch kernel's (the record bf_search_batch builds, in its group's form:
// two 6-bit table chunks up to 12 tools, three up to 16, four and the wide
// queue above or when `wide` is set), otherwise the one-scenario kernel's (levels for at least
// min_roots roots -- the closed-form estimate's, or with `sampled` those of
// lanetree_sampled_levels, as bf_create_scenario takes them -- three chunks
// and the narrow queue up to 16 tools, four chunks and the wide queue up to
// 20, or the wide form at any size when `wide` is set).  The roots are split over the
// record's blocks, and every block's with `lanes` lanes, lane l taking the
// block's roots l, l + lanes, ... (the kernels hand roots out from counters;
// any order gives the same mappings).  Every mapping reported to the sink is
// stored at its canonical index; out[] starts at 0xFFFFFFFF (infeasible
// mappings are not reported) and a second report of one index stores
// 0xDEADBEEF.  info[0..2] = x, y, blocks.
template <uint32_t NC, bool W>
static int host_lanetree_nc(const bf_scenario_desc* d, uint32_t lanes, uint64_t min_roots, int sampled,
                            uint32_t* out, uint32_t* info) {
  LaneTreeRecord rec;
  host::lanetree_record(d, &rec, min_roots);
  if (sampled) host::lanetree_sampled_levels(rec, min_roots, &rec.x, &rec.y);
  info[0] = rec.x;
  info[1] = rec.y;
  info[2] = rec.nblocks;
  const uint64_t total = host::pow3(d->n), roots = host::pow3(rec.x);
  for (uint64_t j = 0; j < total; ++j) out[j] = 0xFFFFFFFFu;
  std::vector<LtSharedT<NC>> shared(1);
  LtSharedT<NC>& S = shared[0];
  S.rec = rec;
  threadIdx.x = 0;
  blockDim.x = 1;
  lt_fill_tables(S);
  struct Store {
    uint32_t* out;
    void operator()(uint32_t idx, uint32_t ms) { out[idx] = out[idx] == 0xFFFFFFFFu ? ms : 0xDEADBEEFu; }
  } sink{out};
  std::vector<uint32_t> rows((size_t)lt_rows<W>(d->n) * lanes, 0xA5A5A5A5u);  // stale shared memory
  for (uint32_t b = 0; b < rec.nblocks; ++b) {
    const uint32_t r0 = (uint32_t)(roots * b / rec.nblocks), r1 = (uint32_t)(roots * (b + 1) / rec.nblocks);
    for (uint32_t lane = 0; lane < lanes; ++lane) {
      uint32_t next = r0 + lane;
      lt_lane<NC, W>(S, rows.data() + lane, lanes,
              [&]() {
                const uint32_t r = next;
                next += lanes;
                return r < r1 ? r : 0xFFFFFFFFu;
              },
              sink);
    }
  }
  return 0;
}

extern "C" int host_lanetree(const bf_scenario_desc* d, uint32_t lanes, uint64_t min_roots, int sampled, int wide,
                             uint32_t* out, uint32_t* info) {
  if (lanes == 0 || d->n > kLtMaxTools) return -1;
  if (min_roots == 0) {  // the batch's records, in the form of the batch kernel's group
    if (wide) return host_lanetree_nc<4, true>(d, lanes, 0, 0, out, info);
    if (d->n <= kLtBatchTools) return host_lanetree_nc<2, false>(d, lanes, 0, 0, out, info);
    if (d->n <= kLtNarrowTools) return host_lanetree_nc<3, false>(d, lanes, 0, 0, out, info);
    return host_lanetree_nc<4, true>(d, lanes, 0, 0, out, info);
  }
  if (!wide && d->n <= kLtNarrowTools) return host_lanetree_nc<3, false>(d, lanes, min_roots, sampled, out, info);
  return host_lanetree_nc<4, true>(d, lanes, min_roots, sampled, out, info);
}
