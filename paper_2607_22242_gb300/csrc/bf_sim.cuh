// bf_sim.cuh -- device-side simulation of one mapping under the integer
// latency model (version 1) declared in include/bf.h.
//
// The model (paper §2.1 problem statement; Factor A/B of §2.3; Table 1's
// gpu_queue = GPU + Load) is restated in bf.h.  This file is the GB300 form of
// it: every per-tool quantity of one simulated mapping lives in registers
// (fully unrolled loops over a compile-time tool count NT >= n), the tool
// tables come from the kernel-parameter constant bank (or shared memory in
// the batched kernel), and everything is 32-bit integer arithmetic except
// two 32x32->64 products per event.
//
// Representation (all exact):
//   * Real time T and CPU end times: u32 microseconds (the scenario validator
//     guarantees every event time fits).
//   * Virtual GPU clock V and GPU end stamps `eg[i]`: kept modulo 2^32.  A
//     running GPU tool always has 0 <= vend - V < 2^32 (its whole work is
//     < 2^32 units), so the u32 difference eg[i] - V is its exact remaining
//     work and eg[i] == V exactly when it ends.
//   * The floor division of a CPU event, floor(dt * 2^20 / f[k]) with
//     dt * 2^20 < 2^52, uses a per-k reciprocal (Granlund & Montgomery, "Division
//     by invariant integers using multiplication", PLDI 1994, Thm 4.2):
//     m = ceil(2^(52+l) / f), l = max(12, ceil(log2 f)); q = umulhi(m, n) >> (l-12).
//   * A queued tool with m > M can never start, so such a mapping is rejected
//     before simulating (the same verdict the model reaches when that tool
//     becomes the queue head).
#pragma once

#include <stdint.h>

namespace bfk {

constexpr int kMaxTools = 20;
constexpr uint32_t kInfeasible = 0xFFFFFFFFu;
// Returned if the event loop ever exceeded its bound (each event retires at
// least one tool, so a correct simulation needs at most n events).  Scenario
// validation keeps real makespans <= 0xFFFFFFFD, so this value never collides.
constexpr uint32_t kStalled = 0xFFFFFFFEu;

// Device-format scenario tables, passed by value as a __grid_constant__
// kernel parameter (constant bank) or staged in shared memory.
struct Tables {
  uint32_t n;
  uint32_t budget;       // M
  uint32_t all_mask;     // (1 << n) - 1
  uint32_t big_mask;     // tools with m > M
  uint32_t pred[kMaxTools];
  uint32_t succ[kMaxTools];
  uint32_t cpu[kMaxTools];   // c_i
  uint32_t wnow[kMaxTools];  // (g_i + x_i) * 1024
  uint32_t wq[kMaxTools];    // (l_i + g_i + x_i) * 1024
  uint32_t vram[kMaxTools];  // m_i
  uint32_t f[kMaxTools + 1];        // f[k]; f[0] unused
  uint32_t fshift[kMaxTools + 1];   // l - 12
  uint64_t fmagic[kMaxTools + 1];   // ceil(2^(52+l) / f[k])
};

// Tables read with a per-thread (dynamic) index, staged in shared memory:
// the per-k slowdown constants and the predecessor masks.
struct SmemTables {
  uint64_t magic[kMaxTools + 1];
  uint32_t f[kMaxTools + 1];
  uint32_t shift[kMaxTools + 1];
  uint32_t pred[kMaxTools];
};

template <typename TB>
__device__ __forceinline__ void load_smem_tables(const TB& tb, SmemTables& s) {
  for (int k = threadIdx.x; k <= kMaxTools; k += blockDim.x) {
    s.magic[k] = tb.fmagic[k];
    s.f[k] = tb.f[k];
    s.shift[k] = tb.fshift[k];
    if (k < kMaxTools) s.pred[k] = tb.pred[k];
  }
}

// Base-3 digits of a mapping as two bitmasks: bit i of `now` <=> digit 1
// (gpu_now), bit i of `que` <=> digit 2 (gpu_queue).
struct Digits {
  uint32_t now, que;
};

template <int NT>
__device__ __forceinline__ Digits decode(uint32_t idx) {
  Digits d{0u, 0u};
#pragma unroll
  for (int i = 0; i < NT; ++i) {
    const uint32_t q = idx / 3u;
    const uint32_t r = idx - 3u * q;
    d.now |= (r == 1u) ? (1u << i) : 0u;
    d.que |= (r == 2u) ? (1u << i) : 0u;
    idx = q;
  }
  return d;
}

// idx -> idx + 1 on the two masks: trailing 2-digits wrap to 0, the next digit
// steps 0->1 or 1->2.
__device__ __forceinline__ void increment(Digits& d) {
  const uint32_t low = ~d.que & (d.que + 1u);  // lowest digit that is not 2
  d.que &= ~(low - 1u);
  const uint32_t had = d.now & low;
  d.now ^= low;
  d.que |= had;
}

// Makespan of one mapping (kInfeasible if infeasible).  `TB` is the tables'
// storage (constant-bank parameter or shared memory).
template <int NT, typename TB>
__device__ __forceinline__ uint32_t simulate(const TB& tb, const SmemTables& sd, Digits dg) {
  if (dg.que & tb.big_mask) return kInfeasible;
  const uint32_t cpu_mask = tb.all_mask & ~(dg.now | dg.que);

  uint32_t ec[NT];   // end time of a running CPU tool, else 0xFFFFFFFF
  uint32_t eg[NT];   // running GPU tool: virtual end stamp; waiting queued tool: ready time
#pragma unroll
  for (int i = 0; i < NT; ++i) {
    ec[i] = 0xFFFFFFFFu;
    eg[i] = 0u;
  }
  uint32_t done = ~tb.all_mask;  // tools >= n count as done
  uint32_t pend = tb.all_mask;   // not yet ready
  uint32_t run_g = 0u;           // running GPU tools
  uint32_t qwait = 0u;           // queued tools waiting
  uint32_t qrun = 0u;            // the running queued tool (0 or one bit)
  uint32_t T = 0u, V = 0u, L = 0u, k = 0u;
  uint32_t tc = 0xFFFFFFFFu;     // earliest CPU end

  // Candidate tools for readiness are the successors of retired tools; at
  // T = 0 every tool is a candidate.
  uint32_t cand = tb.all_mask;

#pragma unroll 1
  for (uint32_t events = 0;; ++events) {
    if (events > (uint32_t)NT) return kStalled;
    // ---- admission at T -------------------------------------------------
    uint32_t ready = 0u;
    {
      uint32_t c = cand & pend;
      const uint32_t notdone = ~done;
      while (c) {
        const int v = __ffs(c) - 1;
        c &= c - 1u;
        if ((sd.pred[v] & notdone) == 0u) ready |= 1u << v;
      }
    }
    if (ready) {
      pend &= ~ready;
      const uint32_t rc = ready & cpu_mask;
      const uint32_t rg = ready & dg.now;
      const uint32_t rq = ready & dg.que;
      if (rc) {
#pragma unroll
        for (int i = 0; i < NT; ++i) {
          if (rc & (1u << i)) {
            ec[i] = T + tb.cpu[i];
            tc = min(tc, ec[i]);
          }
        }
      }
      if (rg) {
#pragma unroll
        for (int i = 0; i < NT; ++i) {
          if (rg & (1u << i)) {
            eg[i] = V + tb.wnow[i];
            L += tb.vram[i];
          }
        }
        run_g |= rg;
        k += __popc(rg);
        if (L > tb.budget) return kInfeasible;
      }
      if (rq) {
#pragma unroll
        for (int i = 0; i < NT; ++i)
          if (rq & (1u << i)) eg[i] = T;
        qwait |= rq;
      }
    }
    if (qwait && !qrun) {
      // Queue head: earliest ready time, ties to the lower index.
      uint32_t best = 0xFFFFFFFFu, hm = 0u, hv = 0u, hw = 0u;
#pragma unroll
      for (int i = 0; i < NT; ++i) {
        if ((qwait & (1u << i)) && eg[i] < best) {
          best = eg[i];
          hm = 1u << i;
          hv = tb.vram[i];
          hw = tb.wq[i];
        }
      }
      if (L + hv <= tb.budget) {
#pragma unroll
        for (int i = 0; i < NT; ++i)
          if (hm & (1u << i)) eg[i] = V + hw;
        L += hv;
        k += 1u;
        run_g |= hm;
        qrun = hm;
        qwait &= ~hm;
      }
    }
    if (done == 0xFFFFFFFFu) break;

    // ---- next event -------------------------------------------------------
    uint32_t rem = 0xFFFFFFFFu;  // remaining work of the first GPU tool to end
#pragma unroll
    for (int i = 0; i < NT; ++i)
      if (run_g & (1u << i)) rem = min(rem, eg[i] - V);
    const uint32_t kk = min(k, (uint32_t)kMaxTools);  // k <= n always; the clamp keeps indexing in bounds
    uint64_t tg = 0xFFFFFFFFFFFFFFFFull;
    if (k) {
      const uint64_t prod = (uint64_t)rem * sd.f[kk];
      tg = (uint64_t)T + ((prod + 0xFFFFFull) >> 20);
    }
    bool gpu_event;
    if (tg <= (uint64_t)tc) {
      T = (uint32_t)tg;
      V += rem;
      gpu_event = true;
    } else {
      if (k) {
        const uint64_t num = (uint64_t)(tc - T) << 20;
        V += (uint32_t)(__umul64hi(sd.magic[kk], num) >> sd.shift[kk]);
      }
      T = tc;
      gpu_event = false;
    }

    // ---- retire everything that ends at T ----------------------------------
    cand = 0u;
    if (tc == T) {
      uint32_t ntc = 0xFFFFFFFFu;
#pragma unroll
      for (int i = 0; i < NT; ++i) {
        if (ec[i] == T) {
          ec[i] = 0xFFFFFFFFu;
          done |= 1u << i;
          cand |= tb.succ[i];
        }
        ntc = min(ntc, ec[i]);
      }
      tc = ntc;
    }
    if (gpu_event) {
      uint32_t rg = 0u;
#pragma unroll
      for (int i = 0; i < NT; ++i) {
        if ((run_g & (1u << i)) && eg[i] == V) {
          rg |= 1u << i;
          L -= tb.vram[i];
          cand |= tb.succ[i];
        }
      }
      run_g &= ~rg;
      done |= rg;
      k -= __popc(rg);
      if (rg & qrun) qrun = 0u;
    }
  }
  return T;
}

}  // namespace bfk
