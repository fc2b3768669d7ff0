// bf_plan.h -- host-side preparation of a scenario for the kernels: the
// device-format tables (per-tool work in 1/1024 units, successor masks, the
// per-k reciprocals of the slowdown table), the prefix/suffix split of the
// mapping index and the suffix window (see bfk::Plan in bf_sim.cuh).
// Host code only; no CUDA calls.
#pragma once

#include <stdint.h>

#include <cstring>

#include "../../include/bf.h"
#include "bf_sim.cuh"

namespace bfk {
namespace host {

inline uint64_t pow3(uint32_t n) {
  uint64_t p = 1;
  for (uint32_t i = 0; i < n; ++i) p *= 3;
  return p;
}

inline void build_tables(const bf_scenario_desc* d, bfk::Tables* t) {
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
    if (d->vram_mib[v] > d->vram_budget_mib) t->big_mask |= 1u << v;
  }
  for (uint32_t k = 1; k <= BF_MAX_TOOLS; ++k) {
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

// Number of suffix tools K (their modes vary across a warp's lanes): large
// enough to keep 32 lanes busy, small enough to leave many prefixes (warps).
inline uint32_t suffix_tools(uint32_t n) {
  if (n >= 13) return 6;   // 729 suffixes: 23 rounds of 32 lanes, 1% idle
  if (n >= 9) return 5;    // 243 suffixes
  if (n >= 4) return 4;    // 81 suffixes
  return n;
}

// Split the tools at P = n - K and find the window start W0: the tools that
// every "suffix source" (a tool >= P whose predecessors are all < P) depends
// on, transitively, are done by the time the first suffix tool becomes ready
// (that tool is a suffix source).  W0 is the lowest tool outside that set.
inline void split_and_window(const bfk::Tables& t, uint32_t* P, uint32_t* K, uint32_t* W0, bfk::Tables* w) {
  const uint32_t n = t.n;
  *K = suffix_tools(n);
  *P = n - *K;
  const uint32_t prefix_mask = (*P >= 32) ? ~0u : ((1u << *P) - 1u);
  uint32_t anc[BF_MAX_TOOLS];
  uint32_t done_at_split = prefix_mask;
  for (uint32_t v = 0; v < n; ++v) {
    anc[v] = t.pred[v];
    for (uint32_t u = 0; u < v; ++u)
      if (t.pred[v] & (1u << u)) anc[v] |= anc[u];
    if (v >= *P && (t.pred[v] & ~prefix_mask) == 0u) done_at_split &= anc[v];
  }
  uint32_t w0 = 0;
  while (w0 < *P && (done_at_split & (1u << w0))) ++w0;
  *W0 = w0;
  std::memset(w, 0, sizeof *w);
  const uint32_t nw = n - w0;
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
  }
  for (uint32_t k = 0; k <= BF_MAX_TOOLS; ++k) {
    w->f[k] = t.f[k];
    w->fshift[k] = t.fshift[k];
    w->fmagic[k] = t.fmagic[k];
  }
}

// Plan covering canonical indices [first, first+count), count >= 1.
inline bfk::Plan make_plan(uint32_t n, uint32_t P, uint32_t K, uint32_t W0, uint64_t first, uint64_t count) {
  bfk::Plan pl;
  std::memset(&pl, 0, sizeof pl);
  pl.P = P;
  pl.K = K;
  pl.W0 = W0;
  pl.pow3P = (uint32_t)pow3(P);
  pl.pow3K = (uint32_t)pow3(K);
  const uint64_t last = first + count - 1;
  pl.first = (uint32_t)first;
  pl.last = (uint32_t)last;
  pl.s_lo = (uint32_t)(first / pl.pow3P);
  pl.s_hi = (uint32_t)(last / pl.pow3P);
  if (pl.s_lo == pl.s_hi) {
    pl.p_lo = (uint32_t)(first % pl.pow3P);
    pl.p_hi = (uint32_t)(last % pl.pow3P);
  } else {
    pl.p_lo = 0;
    pl.p_hi = pl.pow3P - 1;
  }
  (void)n;
  return pl;
}

}  // namespace host
}  // namespace bfk
