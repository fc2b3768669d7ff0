// bf_sim.cuh -- device-side simulation of mappings under the integer latency
// model (version 1) declared in include/bf.h.
//
// The model (paper §2.1 problem statement; Factors A and B of §2.3; Table 1's
// gpu_queue = GPU + Load) is restated in bf.h.  This file is its GB300 form:
// every per-tool quantity of a simulated mapping lives in registers (fully
// unrolled loops over a compile-time slot count NT >= n), tool tables come
// from the kernel-parameter constant bank (or shared memory in the batched
// kernel), and all arithmetic is 32-bit integer except two 32x32->64
// products per event.
//
// Representation (all exact):
//   * Real time T and CPU end times: u32 microseconds (the scenario validator
//     guarantees every event time fits).
//   * Virtual GPU clock V and GPU end stamps eg[i]: kept modulo 2^32.  A
//     running GPU tool always has 0 <= vend - V < 2^32 (its whole work is
//     < 2^32 units), so the u32 difference eg[i] - V is its exact remaining
//     work and eg[i] == V exactly when it ends.  `gmin` is the stamp of the
//     running GPU tool that ends first; processor sharing runs every GPU tool
//     at the same rate, so it only changes when GPU tools start or end.
//   * The floor division of a CPU event, floor(dt * 2^20 / f[k]) with
//     dt * 2^20 < 2^52, uses a per-k reciprocal (Granlund & Montgomery,
//     "Division by invariant integers using multiplication", PLDI 1994,
//     Thm 4.2): m = ceil(2^(52+l) / f), l = max(12, ceil(log2 f));
//     q = umulhi(m, n) >> (l - 12).
//   * A queued tool with m > M can never start, so such a mapping is rejected
//     before simulating (the verdict the model reaches when that tool becomes
//     the queue head).
//
// Resumable runs.  run() can stop at the first admission at which a tool in
// `stop_mask` would become ready, leaving the state exactly as it was after
// that instant's retirements.  Until then no tool of stop_mask has started,
// so the history does not depend on their modes: the search kernels simulate
// a prefix once up to that instant and resume from the saved state for every
// combination of the remaining tools' modes.
#pragma once

#include <stdint.h>

namespace bfk {

constexpr int kMaxTools = 20;
constexpr uint32_t kInfeasible = 0xFFFFFFFFu;
// Returned if a run ever exceeded its event bound (each event retires at
// least one tool, so a correct simulation needs at most n events).  Scenario
// validation keeps real makespans <= 0xFFFFFFFD, so this value never collides.
constexpr uint32_t kStalled = 0xFFFFFFFEu;

enum RunResult : uint32_t { kRunFinished = 0, kRunInfeasible = 1, kRunStopped = 2 };

// Device-format scenario tables (per tool: index order), passed by value as a
// __grid_constant__ kernel parameter (constant bank) or staged in shared memory.
// CAP is the slot capacity: kMaxTools for the enumerating searches, 32 for the
// tree search and index lists beyond 20 tools.
template <int CAP>
struct TablesT {
  static constexpr int cap = CAP;
  uint32_t n;
  uint32_t budget;       // M
  uint32_t all_mask;     // (1 << n) - 1
  uint32_t big_mask;     // tools with m > M
  uint32_t pred[CAP];
  uint32_t succ[CAP];
  uint32_t cpu[CAP];   // c_i
  uint32_t wnow[CAP];  // (g_i + x_i) * 1024
  uint32_t wq[CAP];    // (l_i + g_i + x_i) * 1024
  uint32_t vram[CAP];  // m_i
  // Tool v of these tables is tool orig[v] of the scenario (host bookkeeping:
  // the searches over the whole space may number the tools differently, see
  // bf_plan.h relabel_sources_first; relabeled = 1 then).
  uint32_t orig[CAP];
  uint32_t relabeled;
  uint32_t f[CAP + 1];        // f[k]; f[0] unused
  uint32_t fshift[CAP + 1];   // l - 12
  uint64_t fmagic[CAP + 1];   // ceil(2^(52+l) / f[k])
};
using Tables = TablesT<kMaxTools>;

// How a search enumerates the mapping index idx = p + 3^P * (m + 3^M * i):
//   prefix p -> the modes of tools [0, P);
//   mid m    -> the modes of tools [P, P+M);
//   inner i  -> the modes of the last I tools [Q, n), Q = P+M.
// A warp task is 32 consecutive prefixes (one per lane) times a chunk of mid
// combinations.  Each lane simulates its own prefix once, up to the first
// instant a tool >= P would become ready, and saves that state.  Tools below
// W0 are done by then (they are ancestors of every tool >= P that can become
// ready first), so everything after it is simulated over the window [W0, n)
// only, renumbered from 0.  The warp then walks its mid combinations (and each
// one's inner combinations) in lockstep: the lanes differ only in the early
// tools of their prefixes, so their window simulations mostly follow the same
// control flow.  With I > 0 each lane saves its state again at the first
// instant an inner tool would become ready and resumes it for every inner
// combination.
struct Plan {
  uint32_t P, M, I, W0;
  uint32_t pow3P, pow3M, pow3I;
  uint32_t p_lo, p_hi;      // prefixes this launch covers (inclusive)
  uint32_t m_lo, m_hi;      // mid combinations this launch covers (inclusive)
  uint32_t i_lo, i_hi;      // inner combinations this launch covers (inclusive)
  uint32_t first, last;     // canonical index range (inclusive)
  uint32_t groups;          // ceil((p_hi - p_lo + 1) / 32) prefix groups
  uint32_t m_chunk;         // mid combinations per warp task
  uint32_t m_parts;         // warp tasks per prefix group
  uint32_t full;            // 1 if [first, last] is all of [0, 3^n)
  // Pruned searches only: a mapping whose state at the prefix (inner)
  // checkpoint has T + tail_p (T + tail_q) > bound cannot be optimal.
  // tail_p = the longest path, in minimum isolated durations min(c, g + x),
  // from any tool >= P to the end; tail_q likewise from tools >= Q.
  uint32_t tail_p, tail_q;
  uint32_t bound;           // 0xFFFFFFFF: no pruning
  // I = 1 only: the last tool's duration in each mode when it runs alone
  // (c; g + x; l + g + x), or 0xFFFFFFFF for a GPU mode whose footprint
  // exceeds M.  A lone tool runs at f[1] = 1024 and finds no VRAM in use, so
  // the model's one remaining event ends it exactly this long after it is
  // ready.
  uint32_t alone[3];
  // 1 when the last tool waits for every other tool (then I = 1) and leaving
  // it out narrows the window to a smaller compiled width: the window holds
  // tools [W0, n-1), its run ends when they have all ended -- the instant the
  // last tool becomes ready -- and the last tool then runs alone, ending
  // alone[a] later in mode a.
  uint32_t last_apart;
  // A mapping's canonical index is the sum over tools v of its mode of v times
  // pv[v] = 3^orig[v] (3^v unless the tables are relabeled, whole-space
  // searches only): the prefix part, a mid part per mid combination (a table
  // in shared memory) and the inner part d0 * pvA + d1 * pvB (pv of the first
  // and second inner tools, 0 when absent).
  uint32_t relabeled;
  uint32_t pvA, pvB;
  uint32_t pv[kMaxTools];
};

// Window widths: kernels are compiled for every NW in this list; a plan whose
// window has w tools runs the smallest NW >= w (slots w..NW-1 count as done).
// One unit per width: an exact width saves the empty slots' scans (17- and
// 18-tool layered DAGs 8 % faster than with the even widths alone).
#define BF_FOR_EACH_BUCKET(X) X(4) X(5) X(6) X(7) X(8) X(9) X(10) X(11) X(12) X(13) X(14) X(15) X(16) X(17) X(18) X(19) X(20)

inline int bucket_for(uint32_t w) {
  const int b[] = {4, 5, 6, 7, 8, 9, 10, 11, 12, 13, 14, 15, 16, 17, 18, 19, 20};
  for (int v : b)
    if ((int)w <= v) return v;
  return -1;
}

// Tables read with a per-thread (dynamic) index, staged in shared memory:
// the per-k slowdown constants and the predecessor masks.
template <int CAP>
struct SmemTablesT {
  uint64_t magic[CAP + 1];
  uint32_t f[CAP + 1];
  uint32_t shift[CAP + 1];
  uint32_t pred[CAP];
};
using SmemTables = SmemTablesT<kMaxTools>;

template <int CAP>
__device__ __forceinline__ void load_smem_tables(const TablesT<CAP>& tb, SmemTablesT<CAP>& s) {
  for (int k = threadIdx.x; k <= CAP; k += blockDim.x) {
    s.magic[k] = tb.fmagic[k];
    s.f[k] = tb.f[k];
    s.shift[k] = tb.fshift[k];
    if (k < CAP) s.pred[k] = tb.pred[k];
  }
}

// Base-3 digits of a mapping as two bitmasks: bit i of `now` <=> digit 1
// (gpu_now), bit i of `que` <=> digit 2 (gpu_queue).
struct Digits {
  uint32_t now, que;
};

// The low `digits` base-3 digits of v as masks (digits is a runtime count <= 20).
__device__ __forceinline__ Digits decode(uint32_t v, uint32_t digits) {
  Digits d{0u, 0u};
#pragma unroll
  for (uint32_t i = 0; i < (uint32_t)kMaxTools; ++i) {
    if (i >= digits) break;
    const uint32_t q = v / 3u;
    const uint32_t r = v - 3u * q;
    d.now |= (r == 1u) ? (1u << i) : 0u;
    d.que |= (r == 2u) ? (1u << i) : 0u;
    v = q;
  }
  return d;
}

// v -> v + 1 on the two digit masks: trailing 2-digits wrap to 0, the next
// digit steps 0 -> 1 or 1 -> 2.
__device__ __forceinline__ void increment(Digits& d) {
  const uint32_t low = ~d.que & (d.que + 1u);  // lowest digit that is not 2
  d.que &= ~(low - 1u);
  const uint32_t had = d.now & low;
  d.now ^= low;
  d.que |= had;
}

// Simulation state over NT slots.
template <int NT>
struct State {
  uint32_t ec[NT];   // running CPU tool: real end time; otherwise 0xFFFFFFFF
  uint32_t eg[NT];   // running GPU tool: virtual end stamp; waiting queued tool: ready time
  uint32_t done;     // retired tools (slots >= n count as done)
  uint32_t pend;     // not yet ready
  uint32_t run_g;    // running GPU tools
  uint32_t qwait;    // queued tools waiting
  uint32_t T, V, L;  // (k, the number of running GPU tools, is popc(run_g); the running
                     // queued tool, if any, is run_g & the gpu_queue digits)
  uint32_t tc;       // earliest CPU end (0xFFFFFFFF if none)
  uint32_t gmin;     // stamp of the first GPU tool to end (valid when k > 0)
};

template <int NT>
__device__ __forceinline__ void init_state(State<NT>& s, uint32_t all_mask) {
#pragma unroll
  for (int i = 0; i < NT; ++i) {
    s.ec[i] = 0xFFFFFFFFu;
    s.eg[i] = 0u;
  }
  s.done = ~all_mask;
  s.pend = all_mask;
  s.run_g = s.qwait = 0u;
  s.T = s.V = s.L = 0u;
  s.tc = 0xFFFFFFFFu;
  s.gmin = 0u;
}

// Advance `s` under modes `dg` until every tool is done (kRunFinished, the
// makespan is s.T), the mapping proves infeasible (kRunInfeasible), or a tool
// of `stop_mask` would become ready (kRunStopped, state left before that
// admission).  A stalled run reports kRunFinished with s.T = kStalled.
// Readiness tables.  A tool is ready when all its predecessors are done; the
// done-set is cut into chunks (the whole state when it has at most 10 slots,
// else 8 slots per chunk) and, for every value of a chunk, a table holds the
// tools whose predecessors inside that chunk are all done.  The ready set is
// the pending set ANDed with one table entry per chunk: one shared-memory load
// per chunk instead of a per-tool test.
template <int NT>
struct ReadyTable {
  static constexpr int chunk_bits = (NT <= 10) ? NT : 8;
  static constexpr int chunks = (NT + chunk_bits - 1) / chunk_bits;
  static constexpr int size = chunks << chunk_bits;
};

// Fill a readiness table for NT slots (block-cooperative).
template <int NT, typename TB>
__device__ __forceinline__ void fill_ready_table(const TB& tb, uint32_t* table) {
  constexpr int kBits = ReadyTable<NT>::chunk_bits;
  constexpr uint32_t kMask = (1u << kBits) - 1u;
  for (uint32_t e = threadIdx.x; e < (uint32_t)ReadyTable<NT>::size; e += blockDim.x) {
    const uint32_t c = e >> kBits, x = e & kMask;
    uint32_t r = 0u;
#pragma unroll
    for (int v = 0; v < NT; ++v)
      if ((((tb.pred[v] >> (c * kBits)) & kMask) & ~x) == 0u) r |= 1u << v;
    table[e] = r;
  }
}

template <int NT>
__device__ __forceinline__ uint32_t ready_of(const uint32_t* table, uint32_t pend, uint32_t done) {
  constexpr int kBits = ReadyTable<NT>::chunk_bits;
  constexpr uint32_t kMask = (1u << kBits) - 1u;
  uint32_t r = pend;
#pragma unroll
  for (int c = 0; c < ReadyTable<NT>::chunks; ++c) r &= table[(c << kBits) + ((done >> (c * kBits)) & kMask)];
  return r;
}

template <int NT, typename TB, typename SD>
__device__ __forceinline__ uint32_t run(State<NT>& s, const TB& tb, const SD& sd, const uint32_t* ready_table,
                                        Digits dg, uint32_t stop_mask) {
  static_assert(NT <= TB::cap, "state wider than its tables");
  const uint32_t cpu_mask = tb.all_mask & ~(dg.now | dg.que);
#pragma unroll 1
  for (uint32_t events = 0;; ++events) {
    if (events > (uint32_t)NT + 1u) {
      s.T = kStalled;
      return kRunFinished;
    }
    // ---- admission at T ---------------------------------------------------
    const uint32_t ready = ready_of<NT>(ready_table, s.pend, s.done);
    if (ready & stop_mask) return kRunStopped;
    if (ready) {
      s.pend &= ~ready;
      const uint32_t rc = ready & cpu_mask;
      const uint32_t rg = ready & dg.now;
      const uint32_t rq = ready & dg.que;
      if (rc) {
#pragma unroll
        for (int i = 0; i < NT; ++i) {
          if (rc & (1u << i)) {
            s.ec[i] = s.T + tb.cpu[i];
            s.tc = min(s.tc, s.ec[i]);
          }
        }
      }
      if (rg) {
        uint32_t wmin = 0xFFFFFFFFu;
#pragma unroll
        for (int i = 0; i < NT; ++i) {
          if (rg & (1u << i)) {
            s.eg[i] = s.V + tb.wnow[i];
            s.L += tb.vram[i];
            wmin = min(wmin, tb.wnow[i]);
          }
        }
        if (s.run_g == 0u || wmin < s.gmin - s.V) s.gmin = s.V + wmin;
        s.run_g |= rg;
        if (s.L > tb.budget) return kRunInfeasible;
      }
      if (rq) {
#pragma unroll
        for (int i = 0; i < NT; ++i)
          if (rq & (1u << i)) s.eg[i] = s.T;
        s.qwait |= rq;
      }
    }
    if (s.qwait && !(s.run_g & dg.que)) {
      // Queue head: earliest ready time, ties to the lower index.
      uint32_t best = 0xFFFFFFFFu, hm = 0u, hv = 0u, hw = 0u;
#pragma unroll
      for (int i = 0; i < NT; ++i) {
        if ((s.qwait & (1u << i)) && s.eg[i] < best) {
          best = s.eg[i];
          hm = 1u << i;
          hv = tb.vram[i];
          hw = tb.wq[i];
        }
      }
      if (s.L + hv <= tb.budget) {
#pragma unroll
        for (int i = 0; i < NT; ++i)
          if (hm & (1u << i)) s.eg[i] = s.V + hw;
        if (s.run_g == 0u || hw < s.gmin - s.V) s.gmin = s.V + hw;
        s.L += hv;
        s.run_g |= hm;
        s.qwait &= ~hm;
      }
    }
    if (s.done == 0xFFFFFFFFu) return kRunFinished;

    // ---- next event ---------------------------------------------------------
    const uint32_t k = __popc(s.run_g);
    const uint32_t kk = min(k, (uint32_t)NT);  // k <= NT always; keeps indexing in bounds
    bool gpu_event = false;
    if (k) {
      const uint32_t rem = s.gmin - s.V;
      const uint64_t tg = (uint64_t)s.T + (((uint64_t)rem * sd.f[kk] + 0xFFFFFull) >> 20);
      if (tg <= (uint64_t)s.tc) {
        s.T = (uint32_t)tg;
        s.V = s.gmin;
        gpu_event = true;
      } else {
        const uint64_t num = (uint64_t)(s.tc - s.T) << 20;
        s.V += (uint32_t)(__umul64hi(sd.magic[kk], num) >> sd.shift[kk]);
        s.T = s.tc;
      }
    } else {
      s.T = s.tc;
    }

    // ---- retire everything that ends at T ------------------------------------
    if (s.tc == s.T) {
      uint32_t ntc = 0xFFFFFFFFu;
#pragma unroll
      for (int i = 0; i < NT; ++i) {
        if (s.ec[i] == s.T) {
          s.ec[i] = 0xFFFFFFFFu;
          s.done |= 1u << i;
        }
        ntc = min(ntc, s.ec[i]);
      }
      s.tc = ntc;
    }
    if (gpu_event) {
      uint32_t rg = 0u, nrem = 0xFFFFFFFFu;
#pragma unroll
      for (int i = 0; i < NT; ++i) {
        if (s.run_g & (1u << i)) {
          if (s.eg[i] == s.V) {
            rg |= 1u << i;
            s.L -= tb.vram[i];
          } else {
            nrem = min(nrem, s.eg[i] - s.V);
          }
        }
      }
      s.run_g &= ~rg;
      s.done |= rg;
      s.gmin = s.V + nrem;
    }
  }
}

// Per-lane copy of a window state in shared memory, one word per row of a
// [word][thread] array (`stride` = threads per block), so that a warp's
// accesses to the same word hit 32 different banks.
template <int NW>
struct LaneWords {
  static constexpr int value = 2 * NW + 9;
};

template <int NW>
__device__ __forceinline__ void save_lane(const State<NW>& s, uint32_t* slot, uint32_t stride) {
#pragma unroll
  for (int i = 0; i < NW; ++i) {
    slot[(2 * i) * stride] = s.ec[i];
    slot[(2 * i + 1) * stride] = s.eg[i];
  }
  uint32_t* t = slot + (2 * NW) * stride;
  t[0 * stride] = s.done;
  t[1 * stride] = s.pend;
  t[2 * stride] = s.run_g;
  t[3 * stride] = s.qwait;
  t[4 * stride] = s.T;
  t[5 * stride] = s.V;
  t[6 * stride] = s.L;
  t[7 * stride] = s.tc;
  t[8 * stride] = s.gmin;
}

template <int NW>
__device__ __forceinline__ void load_lane(const uint32_t* slot, uint32_t stride, State<NW>& s) {
#pragma unroll
  for (int i = 0; i < NW; ++i) {
    s.ec[i] = slot[(2 * i) * stride];
    s.eg[i] = slot[(2 * i + 1) * stride];
  }
  const uint32_t* t = slot + (2 * NW) * stride;
  s.done = t[0 * stride];
  s.pend = t[1 * stride];
  s.run_g = t[2 * stride];
  s.qwait = t[3 * stride];
  s.T = t[4 * stride];
  s.V = t[5 * stride];
  s.L = t[6 * stride];
  s.tc = t[7 * stride];
  s.gmin = t[8 * stride];
}

// Save the window part [W0, n) of a prefix state (NP slots) as a window state
// of NW slots.  Window slots past the prefix state's last slot are written as
// unused (no CPU end, stamp 0), so every slot a window run reads is defined.
template <int NP, int NW>
__device__ __forceinline__ void save_prefix_window(const State<NP>& s, uint32_t W0, uint32_t nw, uint32_t* slot,
                                                   uint32_t stride) {
#pragma unroll
  for (int i = 0; i < NP; ++i) {
    const uint32_t j = (uint32_t)i - W0;
    if ((uint32_t)i >= W0 && j < (uint32_t)NW) {
      slot[(2 * j) * stride] = s.ec[i];
      slot[(2 * j + 1) * stride] = s.eg[i];
    }
  }
  for (uint32_t j = (uint32_t)NP - W0; j < (uint32_t)NW; ++j) {
    slot[(2 * j) * stride] = 0xFFFFFFFFu;
    slot[(2 * j + 1) * stride] = 0u;
  }
  const uint32_t wmask = (nw >= 32u) ? 0xFFFFFFFFu : ((1u << nw) - 1u);
  uint32_t* t = slot + (2 * NW) * stride;
  t[0 * stride] = (s.done >> W0) | ~wmask;
  t[1 * stride] = (s.pend >> W0) & wmask;
  t[2 * stride] = s.run_g >> W0;
  t[3 * stride] = s.qwait >> W0;
  t[4 * stride] = s.T;
  t[5 * stride] = s.V;
  t[6 * stride] = s.L;
  t[7 * stride] = s.tc;
  t[8 * stride] = s.gmin;
}

}  // namespace bfk
