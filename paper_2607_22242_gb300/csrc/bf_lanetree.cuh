// bf_lanetree.cuh -- the full search of a scenario of up to 20 tools as a
// tree of checkpoints walked by each lane: many small scenarios in one launch
// (the batch), or one scenario over the whole GPU.
//
// What it computes is the brute-force oracle of §2.3 / §4.1 under the integer
// latency model declared in include/bf.h: for one scenario, the feasible
// mapping of lowest makespan over all 3^n, ties to the lowest canonical
// index.  Every mapping is simulated event by event (Factor A's processor
// sharing, Factor B's VRAM budget, the single FIFO queue of §2.1); what is
// shared between mappings is only the part of a history that cannot depend
// on the modes of tools that have not yet become ready.
//
// The tools, renumbered with the sources first (a topological order that
// changes no result, see bf_plan.h relabel_sources_first), are cut into up to
// three levels [0, x), [x, y), [y, n).  A lane takes a root -- the modes of
// tools [0, x) -- simulates it from time 0 to the first instant a tool >= x
// would become ready, and saves that state (checkpoint 1).  For every
// combination of the modes of tools [x, y) it resumes checkpoint 1 up to the
// first instant a tool >= y would become ready (checkpoint 2), and for every
// combination of tools [y, n) it resumes checkpoint 2 to the end.  Until a
// tool of a level becomes ready nothing in the history depends on its mode,
// so every mapping's makespan is exactly that of a full simulation.
//
// GB300 form.  Divergence, not arithmetic, bounds the batch: random layered
// DAGs start most tools at once and lanes with different modes follow
// different event sequences.  So
//   * a lane's per-tool values live in shared memory (one word per tool,
//     written when the tool starts: the end time of a CPU tool, the end stamp
//     of a GPU tool on the virtual clock), and each
//     event touches only the tools it admits, retires or scans for the next
//     completion (bit loops over small sets) instead of every slot;
//   * the VRAM in use is a table lookup on the set of running GPU tools, the
//     ready set a lookup on the done set (one lookup per 6-bit chunk of the
//     tools: two up to 12 tools, three up to 16, four up to 20);
//   * the queue is a FIFO list of tool numbers -- 4-bit in one 64-bit word up
//     to 16 tools, 5-bit in two words above (the "wide" form):
//     tools join it in the order they become ready (in index order within
//     an instant), which is the model's (ready time, index) order, so its
//     head is the list's first entry;
//   * one pass over the running tools retires those that end and finds the
//     next CPU end and GPU end stamp;
//   * a lane moves to its next job (a level combination or a new root) the
//     moment its current one ends, instead of waiting for the warp's slowest
//     lane; roots come from a per-block counter in shared memory (in the
//     one-scenario search, once the block's share is gone, from a counter in
//     device memory);
//   * a checkpoint is nine state words (eleven in the wide form): the
//     per-tool words of the tools running at it are never written again
//     while it can still be resumed.
// Arithmetic is that of bf_sim.cuh: u32 real time, virtual clock modulo 2^32,
// GPU completion ceil(rem * f[k] / 2^20), the CPU-event advance
// floor(dt * 2^20 / f[k]) by the per-k reciprocal of Granlund and Montgomery
// (PLDI 1994, Thm 4.2).
#pragma once

#include <stdint.h>

#include "bf_sim.cuh"

namespace bfk {

constexpr uint32_t kLtBatchTools = 12;  // the batch sends scenarios of up to this many tools here
constexpr uint32_t kLtMaxTools = 20;    // record capacity
constexpr uint32_t kLtNarrowTools = 16; // up to this many tools the queue's numbers fit 4 bits
constexpr uint32_t kLtChunkBits = 6;    // readiness and VRAM tables: 6-bit chunks of the tools
constexpr uint32_t kLtChunk = 1u << kLtChunkBits;
constexpr uint32_t kLtPartTools = 4;    // tools per table-driven part of the mode combinations
constexpr uint32_t kLtPartCombos = 81;  // 3^kLtPartTools
constexpr uint32_t kLtRootParts = 4;    // root tools [0,4), [4,8), [8,12), [12,x)
constexpr uint32_t kLtParts = kLtRootParts + 2;  // the root's parts, level [x,y), level [y,n)
constexpr uint32_t kLtStateWords = 9;   // pend, run, qset, qlist (2 words), T, V, tc, gm
constexpr uint32_t kLtWideStateWords = 11;  // and the wide queue's second word (2 words)

// State words of a checkpoint in the narrow (W = false) or wide form.
template <bool W>
__host__ __device__ constexpr uint32_t lt_state_words() { return W ? kLtWideStateWords : kLtStateWords; }

// 6-bit chunks the tables of an n-tool scenario need.
__host__ __device__ constexpr uint32_t lt_chunks(uint32_t n) { return (n + kLtChunkBits - 1u) / kLtChunkBits; }

// One scenario of the batch, host-built (bf_plan.h lanetree_record); tools in
// the renumbered order.
struct LaneTreeRecord {
  uint32_t n, budget, all_mask, big_mask;  // big_mask: tools with m > M
  uint32_t x, y;                           // level boundaries, 1 <= x <= y <= n
  uint32_t nblocks;                        // batch: blocks the roots [0, 3^x) are split over
  uint32_t pad;
  uint32_t pred[kLtMaxTools];
  uint32_t dur[3][kLtMaxTools];  // per mode: c (us); (g + x) * 1024; (l + g + x) * 1024
  uint32_t vram[kLtMaxTools];
  uint32_t pv[kLtMaxTools];      // canonical place value 3^orig of each tool
  uint32_t f[kLtMaxTools + 1];
  uint32_t fshift[kLtMaxTools + 1];
  uint64_t fmagic[kLtMaxTools + 1];
};

// Per block: the record and the tables derived from it; NC 6-bit chunks
// cover the record's tools (NC = lt_chunks(n) or more).
template <uint32_t NC>
struct LtSharedT {
  LaneTreeRecord rec;
  uint32_t rt[NC][kLtChunk];  // rt[c][v]: tools whose predecessors in chunk c are all in v
  uint32_t lv[NC][kLtChunk];  // lv[c][v]: VRAM of the tools of chunk c in v
  // Mode combinations of the parts (see kLtParts): now / queue masks and the
  // canonical index part of combination j of each part.
  uint32_t cnow[kLtParts][kLtPartCombos];
  uint32_t cque[kLtParts][kLtPartCombos];
  uint32_t cidx[kLtParts][kLtPartCombos];
  uint32_t ck0[kLtWideStateWords];  // the state words at time 0 (a root's checkpoint)
  uint32_t root_next, root_end;  // this block's roots still to take: [root_next, root_end)
};
using LtShared = LtSharedT<2>;  // the batch: up to kLtBatchTools tools

// Lane state held in registers; the per-tool words are shared-memory rows.
// Every tool is pending, waiting in the queue (qset), running or done, so
// done = ~(pend | run | qset) (the slots beyond n count as done).
struct LtState {
  uint32_t pend, run, qset;
  uint64_t qlist;  // waiting queued tools by index, head in bits 0-3 (0-4 wide); qset says how many
  uint64_t qhi;    // wide form: entries 12 and up, 5 bits each
  uint32_t T, V;   // real time (us); virtual GPU clock (1/1024 us of isolated work, modulo 2^32)
  uint32_t tc;     // earliest end of a running CPU tool (0xFFFFFFFF if none)
  uint32_t gm;     // end stamp of the running GPU tool that ends first (when one runs)
};

// Rows of one lane ([row][thread], `stride` threads): the per-tool words
// [0, n), then the state words of checkpoint 1 [n, n + w) and of checkpoint
// 2 [n + w, n + 2w), w = lt_state_words<W>().  One set of per-tool words serves every level: a tool's
// word is written once per simulation, when it starts, and only read after
// that; a job resumed from a checkpoint starts only tools that were pending
// there, so it never overwrites the word of a tool running at any checkpoint
// it or a later job may resume from.  A checkpoint is its state words alone.
template <bool W = false>
__host__ __device__ inline uint32_t lt_rows(uint32_t n) { return n + 2u * lt_state_words<W>(); }

template <uint32_t NC>
__device__ __forceinline__ uint32_t lt_ready(const LtSharedT<NC>& S, uint32_t pend, uint32_t done) {
  uint32_t r = pend;
#pragma unroll
  for (uint32_t c = 0; c < NC; ++c) r &= S.rt[c][(done >> (kLtChunkBits * c)) & (kLtChunk - 1u)];
  return r;
}

template <uint32_t NC>
__device__ __forceinline__ uint32_t lt_vram(const LtSharedT<NC>& S, uint32_t gpu_running) {
  uint32_t m = 0u;
#pragma unroll
  for (uint32_t c = 0; c < NC; ++c) m += S.lv[c][(gpu_running >> (kLtChunkBits * c)) & (kLtChunk - 1u)];
  return m;
}

// Fill the block's tables from S.rec (block-cooperative; S.rec is in place).
template <uint32_t NC>
__device__ __forceinline__ void lt_fill_tables(LtSharedT<NC>& S) {
  const LaneTreeRecord& R = S.rec;
  for (uint32_t e = threadIdx.x; e < NC * kLtChunk; e += blockDim.x) {
    const uint32_t c = e / kLtChunk, v = e % kLtChunk, lo = kLtChunkBits * c;
    uint32_t ready = 0u, mem = 0u;
    for (uint32_t t = 0; t < R.n; ++t) {
      if ((((R.pred[t] >> lo) & (kLtChunk - 1u)) & ~v) == 0u) ready |= 1u << t;
      if (t >= lo && t < lo + kLtChunkBits && ((v >> (t - lo)) & 1u)) mem += R.vram[t];
    }
    S.rt[c][v] = ready;
    S.lv[c][v] = mem;
  }
  // Parts: root tools [0, min(x,4)), [4, min(x,8)), [8, min(x,12)), [12, x);
  // level tools [x, y), [y, n).
  for (uint32_t p = 0; p < kLtParts; ++p) {
    const uint32_t lo = p < kLtRootParts ? min(kLtPartTools * p, R.x) : (p == kLtRootParts ? R.x : R.y);
    const uint32_t hi = p < kLtRootParts ? min(kLtPartTools * p + kLtPartTools, R.x) : (p == kLtRootParts ? R.y : R.n);
    uint32_t combos = 1u;
    for (uint32_t t = lo; t < hi; ++t) combos *= 3u;
    for (uint32_t j = threadIdx.x; j < combos; j += blockDim.x) {
      uint32_t now = 0u, que = 0u, idx = 0u, v = j;
      for (uint32_t t = lo; t < hi; ++t) {
        const uint32_t a = v % 3u;
        v /= 3u;
        now |= (a == 1u) ? (1u << t) : 0u;
        que |= (a == 2u) ? (1u << t) : 0u;
        idx += a * R.pv[t];
      }
      S.cnow[p][j] = now;
      S.cque[p][j] = que;
      S.cidx[p][j] = idx;
    }
  }
  if (threadIdx.x == 0) {
    uint32_t* w = S.ck0;
    w[0] = R.all_mask;        // pend: every tool
    w[1] = w[2] = 0u;         // run, qset
    w[3] = w[4] = 0u;         // qlist
    w[5] = w[6] = 0u;         // T, V
    w[7] = 0xFFFFFFFFu;       // tc: no CPU tool runs
    w[8] = 0u;                // gm
    w[9] = w[10] = 0u;        // the wide queue's second word
  }
}

enum LtStep : uint32_t { kLtContinue = 0, kLtFinished = 1, kLtInfeasible = 2, kLtStopped = 3 };

// One step of a lane's simulation under modes (now, que; the other tools run
// on the CPU): the admission at T -- or kLtStopped, before it, when a tool of
// `stop` would become ready -- then the next event and the retirements at it.
// Returns kLtFinished once every tool has ended (the makespan is s.T).  The
// loops' bodies are written as selects: lanes of a warp are at different
// points of their simulations, and a branch in a body would run both sides.
template <uint32_t NC, bool W = false>
__device__ __forceinline__ uint32_t lt_step(const LtSharedT<NC>& S, LtState& s, uint32_t now, uint32_t que,
                                            uint32_t stop, uint32_t* e, uint32_t stride) {
  const LaneTreeRecord& R = S.rec;
  const uint32_t gpu = now | que;
  const uint32_t ready = lt_ready(S, s.pend, ~(s.pend | s.run | s.qset));
  if (ready & stop) return kLtStopped;
  // ---- admission at T: newly ready tools start in index order -------------
  if (ready) {
    s.pend &= ~ready;
    // cpu: real end T + c; gpu_now: end stamp V + (g + x) * 1024
    for (uint32_t m = ready & ~que; m; m &= m - 1u) {
      const uint32_t i = __ffs(m) - 1u;
      const bool isn = (now >> i) & 1u;
      const uint32_t w = R.dur[isn ? 1 : 0][i];
      const uint32_t val = (isn ? s.V : s.T) + w;
      e[i * stride] = val;
      const bool first = isn && (!(s.run & gpu) || w < s.gm - s.V);
      s.gm = first ? val : s.gm;
      s.tc = isn ? s.tc : min(s.tc, val);
      s.run |= 1u << i;
    }
    // queued: join the FIFO in index order (a row is written when the tool starts)
    for (uint32_t m = ready & que; m; m &= m - 1u) {
      const uint32_t i = __ffs(m) - 1u;
      const uint32_t pos = __popc(s.qset);
      if (W) {  // 12 entries of 5 bits in the first word, the rest in the second
        const uint32_t sh = 5u * pos;
        s.qlist |= pos < 12u ? (uint64_t)i << (sh & 63u) : 0ull;
        s.qhi |= pos >= 12u ? (uint64_t)i << ((sh - 60u) & 63u) : 0ull;
      } else {
        s.qlist |= (uint64_t)i << (4u * pos);
      }
      s.qset |= 1u << i;
    }
    if ((ready & now) && lt_vram(S, s.run & gpu) > R.budget) return kLtInfeasible;  // out of memory
  }
  // ---- queue head: the first tool of the FIFO --------------------------------
  if (s.qset && !(s.run & que)) {
    const uint32_t h = (uint32_t)(s.qlist & (W ? 31u : 15u)), hb = 1u << h;
    if (hb & R.big_mask) return kLtInfeasible;  // a head larger than M can never start
    const uint32_t rg = s.run & gpu;
    if (lt_vram(S, rg | hb) <= R.budget) {  // no bypass: otherwise the head waits
      const uint32_t w = R.dur[2][h], val = s.V + w;
      s.gm = (!rg || w < s.gm - s.V) ? val : s.gm;
      e[h * stride] = val;
      s.run |= hb;
      s.qset &= ~hb;
      if (W) {
        s.qlist = (s.qlist >> 5) | ((s.qhi & 31ull) << 55);
        s.qhi >>= 5;
      } else {
        s.qlist >>= 4;
      }
    }
  }
  // ---- next event -----------------------------------------------------------
  const uint32_t rg = s.run & gpu;
  const uint32_t k = __popc(rg), kk = k ? k : 1u;  // kk: a valid table index when no GPU tool runs
  const uint32_t rem = s.gm - s.V;
  const uint64_t tg = (uint64_t)s.T + (((uint64_t)rem * R.f[kk] + 0xFFFFFull) >> 20);
  const bool gpu_event = k != 0u && tg <= (uint64_t)s.tc;
  const uint32_t adv = (uint32_t)(__umul64hi(R.fmagic[kk], (uint64_t)(s.tc - s.T) << 20) >> R.fshift[kk]);
  s.V = gpu_event ? s.gm : (k ? s.V + adv : s.V);
  s.T = gpu_event ? (uint32_t)tg : s.tc;
  // ---- retire everything that ends at T; the next CPU end and GPU stamp -----
  // Only tools of the kinds that can end now are scanned: CPU tools when T
  // reached the earliest CPU end, GPU tools at a GPU event (at a CPU event V
  // stays below every running GPU tool's stamp); the other kind's earliest
  // end is unchanged.
  const bool cpu_event = s.tc == s.T;
  uint32_t ntc = cpu_event ? 0xFFFFFFFFu : s.tc, nrem = gpu_event ? 0xFFFFFFFFu : s.gm - s.V, ended = 0u;
  for (uint32_t m = (cpu_event ? s.run & ~gpu : 0u) | (gpu_event ? rg : 0u); m; m &= m - 1u) {
    const uint32_t i = __ffs(m) - 1u, b = 1u << i, end = e[i * stride];
    const bool isc = (gpu & b) == 0u;
    const bool hit = end == (isc ? s.T : s.V);
    ended |= hit ? b : 0u;
    ntc = (isc && !hit) ? min(ntc, end) : ntc;
    nrem = (!isc && !hit) ? min(nrem, end - s.V) : nrem;
  }
  s.run &= ~ended;
  s.tc = ntc;
  s.gm = s.V + nrem;
  return (s.pend | s.run | s.qset) == 0u ? kLtFinished : kLtContinue;
}

// One lane's share of the block's roots: every mapping below each root it
// takes reaches the sink as (canonical index, makespan); infeasible mappings
// are not reported (a search keeps the lowest feasible key).  `rows` is this
// lane's first row, `stride` the rows' stride.  take_root() returns the next
// root index or 0xFFFFFFFF when none is left.
//
// Every change of job goes through one code path (lanes of a warp change
// jobs at different steps): a finished or infeasible job moves to the next
// combination of the deepest level that has one left -- or to a new root,
// which loads the block's time-0 state like a checkpoint -- and a stopped
// job saves its state as the next level's checkpoint and continues with that
// level's first combination (every tool of it on the CPU).
template <uint32_t NC, bool W = false, typename TakeRoot, typename Sink>
__device__ __forceinline__ void lt_lane(const LtSharedT<NC>& S, uint32_t* rows, uint32_t stride, TakeRoot take_root,
                                        Sink& sink) {
  constexpr uint32_t SW = lt_state_words<W>();
  const LaneTreeRecord& R = S.rec;
  const uint32_t n = R.n;
  uint32_t* const cur = rows;
  const uint32_t stop0 = R.all_mask & ~((1u << R.x) - 1u);
  const uint32_t stop1 = R.all_mask & ~((1u << R.y) - 1u);
  const uint32_t lm1 = stop0 & ~stop1, lm2 = stop1;  // tools of levels 1 and 2
  uint32_t cnt1 = 1u, cnt2 = 1u;
  for (uint32_t t = R.x; t < R.y; ++t) cnt1 *= 3u;
  for (uint32_t t = R.y; t < n; ++t) cnt2 *= 3u;
  const uint32_t bound = n + 2u;  // steps of one job: each event retires a tool

  LtState s{};
  uint32_t now = 0u, que = 0u, stop = 0u, lvl = 0u, c1 = 0u, c2 = 0u;
  uint32_t idx0 = 0u, idx1 = 0u, idx2 = 0u, steps = 0u;
  uint32_t r = kLtInfeasible;  // "the current job is over": the first pass takes a root
  for (;;) {
    if (r != kLtContinue) {
      // ---- the next job --------------------------------------------------
      if (r == kLtFinished) sink(idx0 + idx1 + idx2, s.T);
      const bool descend = r == kLtStopped;
      const bool a2 = !descend && lvl == 2u && c2 + 1u < cnt2;
      const bool a1 = !descend && !a2 && lvl >= 1u && c1 + 1u < cnt1;
      const uint32_t L = descend ? lvl + 1u : (a2 ? 2u : (a1 ? 1u : 0u));
      c1 = (descend && L == 1u) ? 0u : (a1 ? c1 + 1u : c1);
      c2 = (descend && L == 2u) ? 0u : (a2 ? c2 + 1u : c2);
      uint32_t root = 0u;
      if (L == 0u) {
        root = take_root();
        if (root == 0xFFFFFFFFu) return;
      }
      uint32_t* const cw = rows + (L == 2u ? n + SW : n) * stride;  // checkpoint L's state words
      if (descend) {  // save the state words
        cw[0] = s.pend;
        cw[stride] = s.run;
        cw[2u * stride] = s.qset;
        cw[3u * stride] = (uint32_t)s.qlist;
        cw[4u * stride] = (uint32_t)(s.qlist >> 32);
        cw[5u * stride] = s.T;
        cw[6u * stride] = s.V;
        cw[7u * stride] = s.tc;
        cw[8u * stride] = s.gm;
        if (W) {
          cw[9u * stride] = (uint32_t)s.qhi;
          cw[10u * stride] = (uint32_t)(s.qhi >> 32);
        }
      } else {  // load a checkpoint's state words, or the time-0 state for a root
        const uint32_t* w = L == 0u ? S.ck0 : cw;
        const uint32_t ws = L == 0u ? 1u : stride;
        s.pend = w[0];
        s.run = w[ws];
        s.qset = w[2u * ws];
        s.qlist = (uint64_t)w[3u * ws] | ((uint64_t)w[4u * ws] << 32);
        s.T = w[5u * ws];
        s.V = w[6u * ws];
        s.tc = w[7u * ws];
        s.gm = w[8u * ws];
        if (W) s.qhi = (uint64_t)w[9u * ws] | ((uint64_t)w[10u * ws] << 32);
      }
      // Modes and index part of the new job's level: a root's four table
      // parts (base-81 digits of the root), or one level combination (the
      // first, all cpu, on a descent).
      uint32_t cn, cq, xi;
      if (L == 0u) {
        uint32_t q = root;
        cn = cq = xi = 0u;
#pragma unroll
        for (uint32_t p = 0; p < kLtRootParts; ++p) {
          const uint32_t d = p + 1u < kLtRootParts ? q % kLtPartCombos : q;
          q /= kLtPartCombos;
          cn |= S.cnow[p][d];
          cq |= S.cque[p][d];
          xi += S.cidx[p][d];
        }
      } else {
        const uint32_t pa = L == 1u ? kLtRootParts : kLtRootParts + 1u, ia = L == 1u ? c1 : c2;
        cn = S.cnow[pa][ia];
        cq = S.cque[pa][ia];
        xi = S.cidx[pa][ia];
      }
      const uint32_t clear = L == 0u ? 0xFFFFFFFFu : (L == 1u ? (lm1 | lm2) : lm2);
      now = (now & ~clear) | cn;
      que = (que & ~clear) | cq;
      idx0 = L == 0u ? xi : idx0;
      idx1 = L == 1u ? xi : (L == 0u ? 0u : idx1);
      idx2 = L == 2u ? xi : 0u;
      stop = L == 0u ? stop0 : (L == 1u ? stop1 : 0u);
      lvl = L;
      steps = 0u;
    }
    r = lt_step<NC, W>(S, s, now, que, stop, cur, stride);
    if (++steps > bound && r == kLtContinue) {  // never taken by a correct simulation
      s.T = kStalled;
      r = kLtFinished;
    }
  }
}

}  // namespace bfk
