// bf_tree.h -- internal interface between the C ABI (bf_capi.cu) and the tree
// search kernels (bf_tree.cu): the best-so-far record, the counters and the
// launchers.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "bf_tree.cuh"

namespace bfk {

// Best mapping found so far: makespan, then canonical index (lexicographic
// minimum, updated by 16-byte compare-and-swap).  {~0, ~0} = none.
struct __align__(16) BestRecord {
  unsigned long long ms;
  unsigned long long idx;
};

// Device-side counters of one tree search.
struct TreeCounters {
  unsigned long long leaf_nodes;  // leaf-level nodes enumerated (counted by the warp task of their first chunk)
  unsigned long long leaves;      // mappings simulated to the end by the leaf kernel
  uint32_t error;                 // bit 0: a level buffer overflowed; bit 1: a best-record update gave up
  uint32_t pad;
};

size_t tree_node_words();
cudaError_t launch_tree_root(const TablesW& tb, uint32_t* buf, uint32_t cap, cudaStream_t st);
cudaError_t launch_tree_expand(const TablesW& tb, const TreeConsts& tc, const uint32_t* src, uint32_t src_cap,
                               uint32_t lo, uint32_t cnt, uint32_t d, uint32_t* dst, uint32_t dst_cap,
                               unsigned long long* appended, unsigned long long base_total, const uint32_t* bound,
                               TreeCounters* ctr, cudaStream_t st);
cudaError_t launch_tree_leaf(const TablesW& tb, const TreeConsts& tc, const uint32_t* src, uint32_t src_cap,
                             uint32_t lo, uint32_t cnt, uint32_t target_tasks, uint32_t* bound, BestRecord* best,
                             TreeCounters* ctr, cudaStream_t st);
cudaError_t launch_wide_list(const TablesW& tb, uint64_t total, const uint64_t* idx, uint64_t count, uint32_t* ms,
                             uint8_t* fe, int grid, cudaStream_t st);

}  // namespace bfk
