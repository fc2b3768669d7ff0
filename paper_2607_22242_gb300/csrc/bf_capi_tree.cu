// bf_capi_tree.cu -- bf_search_tree (include/bf.h): the host side of the tree
// search, whose kernels are in bf_tree.cu.  The host keeps the level sizes and
// decides, step by step, which level to pop next; every step that expands
// nodes waits (bounded) for the count of their surviving children.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstddef>
#include <cstring>
#include <new>
#include <chrono>
#include <vector>

#include "bf_capi_internal.h"

using namespace bfcapi;
using bfk::host::pow3;

namespace {

int search_tree_impl(const bf_scenario* scn_const, uint32_t space, uint32_t flags, uint64_t hint_index,
                     bf_result* out, bf_tree_stats* stats, void* cuda_stream) {
  const char* who = "bf_search_tree";
  if (!scn_const || !out) return fail(BF_EINVAL, "%s: NULL argument", who);
  if (space != BF_SPACE_BINARY && space != BF_SPACE_FULL)
    return fail(BF_EINVAL, "%s: space %u is neither BF_SPACE_BINARY (2) nor BF_SPACE_FULL (3)", who, space);
  if (flags & ~(uint32_t)BF_TREE_NO_PRUNE) return fail(BF_EINVAL, "%s: unknown flags 0x%x", who, flags);
  if (const int rc = check_device(scn_const, who)) return rc;
  // The handle's lazily allocated level buffers are scratch, not state.
  bf_scenario* scn = const_cast<bf_scenario*>(scn_const);
  // The tree runs on the tools renumbered with the sources first
  // (relabel_sources_first): a source in a later layer is then decided near
  // the root instead of keeping every node's window open from time 0, and the
  // model's results do not change.  Indices stay canonical: slot v holds tool
  // tb.orig[v], whose digit weighs 3^orig[v].
  bfk::TablesW renumbered;
  const bool relabeled = bfk::host::relabel_sources_first(scn->wide, &renumbered);
  const bfk::TablesW& tb = relabeled ? renumbered : scn->wide;
  const uint32_t n = scn->desc.n, R = space;
  const bool prune = !(flags & BF_TREE_NO_PRUNE);
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);

  // Constants: the leaf depth, the bound's per-tool durations, digit powers.
  bfk::TreeConsts tc;
  bfk::host::tree_consts(tb, R, prune, &tc);

  // Level buffers: level d holds up to R * kPop nodes (one pop of its parent
  // level); nodes are popped from the deepest non-empty level, so no level
  // ever holds more.
  constexpr uint32_t kPop = 65536;
  const uint32_t cap = R * kPop;
  const uint32_t levels = tc.leaf_level + 1;
  const size_t level_words = bfk::tree_node_words() * cap;
  const size_t need = sizeof(uint32_t) * level_words * levels;
  cudaError_t e = cudaSuccess;
  if (scn->levels_bytes < need) {
    if (scn->d_levels) cudaFree(scn->d_levels);
    scn->d_levels = nullptr;
    scn->levels_bytes = 0;
    e = lib_malloc(reinterpret_cast<void**>(&scn->d_levels), need);
    if (e != cudaSuccess) return cuda_fail(e, who);
    scn->levels_bytes = need;
  }
  auto level = [&](uint32_t d) { return scn->d_levels + level_words * d; };

  bf_scratch* h = scn->h_scratch;
  bf_scratch* dv = scn->d_scratch;
  uint32_t launches = 0;

  // 1. Incumbent: the best feasible of a few mappings of the space (the hint
  //    if it lies in it, all-cpu, all-gpu_now, each tool on its isolated-faster
  //    device, and all-gpu_queue in the full space).
  uint32_t bound = 0xFFFFFFFFu;
  if (prune) {
    const uint64_t total = pow3(n);
    uint32_t nc = 0;
    bool hint_ok = hint_index < total;
    if (hint_ok && R == 2)
      for (uint64_t v = hint_index; v; v /= 3) hint_ok = hint_ok && (v % 3 != 2);
    if (hint_ok) h->idx[nc++] = hint_index;
    const bfk::TablesW& tsc = scn->wide;  // the scenario's numbering
    uint64_t now = 0, fast = 0, p = 1;
    for (uint32_t i = 0; i < n; ++i, p *= 3) {
      now += p;
      if ((tsc.wnow[i] >> 10) < tsc.cpu[i]) fast += p;
    }
    h->idx[nc++] = 0;
    h->idx[nc++] = now;
    h->idx[nc++] = fast;
    if (R == 3) h->idx[nc++] = 2 * now;
    e = cudaMemcpyAsync(dv->idx, h->idx, sizeof(uint64_t) * nc, cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess) e = launch_list(scn, dv->idx, nc, dv->ms, dv->fe, 1, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(h->ms, dv->ms, sizeof(uint32_t) * nc, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(h->fe, dv->fe, nc, cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return cuda_fail(e, who);
    const int rc = wait_stream(st, who);
    if (rc != BF_OK) return rc;
    ++launches;
    for (uint32_t j = 0; j < nc; ++j)
      if (h->fe[j] == 1 && h->ms[j] < bound) bound = h->ms[j];
  }

  // 2. Reset the record, bound and counters; write the root node.
  h->best.ms = ~0ull;
  h->best.idx = ~0ull;
  h->bound = bound;
  h->appended = 0;
  std::memset(&h->ctr, 0, sizeof h->ctr);
  e = cudaMemcpyAsync(&dv->best, &h->best,
                      offsetof(bf_scratch, idx) - offsetof(bf_scratch, best), cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = bfk::launch_tree_root(tb, level(0), cap, st);
  if (e != cudaSuccess) return cuda_fail(e, who);
  ++launches;

  // 3. Depth first over levels: pop up to kPop nodes (a whole leaf-level
  //    buffer) from the deepest non-empty level, and expand them into the
  //    next level or enumerate their leaves.  A large tree starts with a
  //    dive: pops of kDive nodes reach the leaves after one expansion per
  //    level, and the first leaves' makespans become the bound; the dive's
  //    other nodes are then dropped and the search restarts from the root
  //    (the root stays in the level-0 buffer), now pruning the wide levels
  //    with that bound.  (Measured: 8192 beat 64 and 1024, and beat diving
  //    without the restart.)
  constexpr uint32_t kDive = 8192;
  // The whole search, not only each wait, is held to the wait limit.
  const auto t_start = std::chrono::steady_clock::now();
  const uint32_t limit_ms = wait_limit_ms();
  std::vector<uint32_t> size(levels, 0);
  size[0] = 1;
  uint64_t nodes = 1;
  uint64_t leaf_level_nodes = 1;  // radix^L, saturating
  for (uint32_t i = 0; i < tc.leaf_level && leaf_level_nodes <= kPop; ++i) leaf_level_nodes *= R;
  bool diving = prune && leaf_level_nodes > kPop;
  for (;;) {
    int d = (int)levels - 1;
    while (d >= 0 && size[d] == 0) --d;
    if (d < 0) break;
    const uint32_t L = (uint32_t)d;
    const uint32_t pop = diving ? kDive : kPop;
    const uint32_t take = L == tc.leaf_level ? size[L] : (size[L] < pop ? size[L] : pop);
    if (diving && L == tc.leaf_level) {
      e = bfk::launch_tree_leaf(tb, tc, level(L), cap, size[L] - take, take, 16384, &dv->bound, &dv->best, &dv->ctr,
                                st);
      if (e != cudaSuccess) return cuda_fail(e, who);
      ++launches;
      std::fill(size.begin(), size.end(), 0u);
      size[0] = 1;
      diving = false;
      continue;
    }
    const uint32_t lo = size[L] - take;
    size[L] = lo;
    if (L == tc.leaf_level) {
      e = bfk::launch_tree_leaf(tb, tc, level(L), cap, lo, take, 16384, &dv->bound, &dv->best, &dv->ctr, st);
      if (e != cudaSuccess) return cuda_fail(e, who);
      ++launches;
      continue;
    }
    const unsigned long long before = h->appended;
    e = bfk::launch_tree_expand(tb, tc, level(L), cap, lo, take, L, level(L + 1), cap, &dv->appended, before,
                                &dv->bound, &dv->ctr, st);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(&h->appended, &dv->appended, sizeof(unsigned long long), cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return cuda_fail(e, who);
    const int rc = wait_stream(st, who);
    if (rc != BF_OK) return rc;
    if (limit_ms) {
      const auto ms = std::chrono::duration_cast<std::chrono::milliseconds>(std::chrono::steady_clock::now() - t_start);
      if (ms.count() > (long long)limit_ms)
        return fail(BF_ETIMEOUT, "%s: search not finished after %u ms", who, limit_ms);
    }
    ++launches;
    const uint32_t added = (uint32_t)(h->appended - before);
    size[L + 1] = added;
    nodes += added;
  }

  // 4. The record.
  e = cudaMemcpyAsync(&h->best, &dv->best,
                      offsetof(bf_scratch, idx) - offsetof(bf_scratch, best), cudaMemcpyDeviceToHost, st);
  if (e != cudaSuccess) return cuda_fail(e, who);
  const int rc = wait_stream(st, who);
  if (rc != BF_OK) return rc;
  if (h->ctr.error) return fail(BF_ECUDA, "%s: internal error 0x%x in the tree kernels", who, h->ctr.error);
  std::memset(out, 0, sizeof *out);
  if (h->best.ms >= 0xFFFFFFFFull) {
    out->makespan_us = 0xFFFFFFFFu;
  } else {
    out->index = h->best.idx;
    out->makespan_us = (uint32_t)h->best.ms;
    out->feasible = 1;
    uint64_t idx = out->index;
    for (uint32_t i = 0; i < n; ++i, idx /= 3) out->mode[i] = (uint8_t)(idx % 3);
  }
  if (stats) {
    stats->nodes = nodes;
    stats->leaf_nodes = h->ctr.leaf_nodes;
    stats->leaves = h->ctr.leaves;
    stats->launches = launches;
    stats->leaf_depth = tc.D;
    stats->incumbent_us = bound;
  }
  return BF_OK;
}

}  // namespace

extern "C" {

// Host allocation failures and other C++ exceptions stay inside the library.
int bf_search_tree(const bf_scenario* scn, uint32_t space, uint32_t flags, uint64_t hint_index, bf_result* out,
                   bf_tree_stats* stats, void* cuda_stream) {
  try {
    return search_tree_impl(scn, space, flags, hint_index, out, stats, cuda_stream);
  } catch (const std::bad_alloc&) {
    return fail(BF_ENOMEM, "bf_search_tree: host allocation failed");
  } catch (const std::exception& ex) {
    return fail(BF_EINVAL, "bf_search_tree: %s", ex.what());
  }
}

}  // extern "C"
