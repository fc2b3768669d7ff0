// bf_capi_internal.h -- what the C ABI's translation units share: the
// handle and its scratch, and the helpers for errors, allocation, bounded
// waits and index lists (defined in bf_capi.cu).  Not installed; not part of
// the ABI.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/bf.h"
#include "bf_lanetree_launch.h"
#include "bf_launch.h"
#include "bf_plan.h"
#include "bf_tree.h"

// Per-handle scratch, one block on the device and a pinned mirror on the host:
// the packed search key, the tree search's best record, bound and counters,
// the what-if probe list with its results, and the lane-tree record.
struct bf_scratch {
  bfk::SearchSync search;  // whole-space searches' launch state; search.key of the host mirror receives their result
  unsigned long long key;
  uint32_t survivors;   // pruned search: number of surviving prefixes
  uint32_t pruned_bound;  // pruned search: the incumbent's makespan (set with survivors)
  bfk::BestRecord best;      // tree search: best (makespan, index) so far
  uint32_t bound;            // tree search: makespan bound for pruning
  uint32_t pad2;
  unsigned long long appended;  // tree search: nodes appended by all expansions so far
  bfk::TreeCounters ctr;     // tree search: counters and error bits
  uint64_t idx[BF_MAX_PROBES];
  uint32_t ms[BF_MAX_PROBES];
  uint8_t fe[BF_MAX_PROBES];
  bfk::LaneTreeRecord lt;  // whole-space search by the lane-tree kernel (bf_scenario::lanetree)
};

struct bf_scenario {
  bf_scenario_desc desc;
  bfk::TablesW wide;    // all n tools, 32 slots (index lists and the tree search)
  bfk::Tables tables;   // all n tools (n <= BF_MAX_TOOLS_ENUM; zero otherwise)
  bfk::Tables window;   // tools [W0, n), renumbered from 0
  bfk::Plan plan;       // enumeration split and window (see bfk::Plan), full range
  // Searches of the whole space: the tools renumbered with the sources first
  // (bf_plan.h relabel_sources_first; equal to the above when that order is
  // the scenario's own), with their split and window.
  bfk::Tables rtables;
  bfk::Tables rwindow;
  bfk::Plan rplan;
  bfk::Tables pwindow;  // bf_search_pruned: its window (of pplan, on rtables)
  bfk::Plan pplan;      // bf_search_pruned: its split (shorter prefixes: fewer to filter)
  // Searches of the whole space by the lane-tree kernel (scenarios of
  // kLtSingleMinTools to kLtMaxTools tools): its record's level boundary x
  // and the blocks of a launch; lanetree false otherwise.
  bool lanetree;
  uint32_t lt_x, lt_blocks;
  int device;
  bf_scratch* d_scratch;      // device scratch
  bf_scratch* h_scratch;      // pinned host mirror
  unsigned long long* d_key;  // &d_scratch->key
  unsigned long long* h_key;  // &h_scratch->key
  unsigned long long* d_host_search_key;  // &h_scratch->search.key as the device addresses it
  uint32_t* d_survivors;      // pruned search: 3^pplan.P prefix slots, allocated on first use
  uint32_t* d_levels;         // tree search: node buffers of every level, allocated on first use
  size_t levels_bytes;
};

namespace bfcapi {

// Record `code` and a printf-style message as this thread's last error; returns code.
int fail(int code, const char* fmt, ...);
// A failed CUDA call: BF_ENOMEM for allocation failures, else BF_ECUDA.
int cuda_fail(cudaError_t e, const char* what);
// cudaMalloc / cudaMallocHost with the test-only failure injection.
cudaError_t lib_malloc(void** p, size_t bytes);
cudaError_t lib_malloc_host(void** p, size_t bytes);
// Wait for `st` with the process-wide time limit (BF_ETIMEOUT when it passes).
int wait_stream(cudaStream_t st, const char* who);
// That limit in milliseconds (0: none).
uint32_t wait_limit_ms();
// BF_EINVAL unless the handle's device is current.
int check_device(const bf_scenario* scn, const char* who);
// Makespans of a list of mappings on the index-list kernel for the scenario's width.
cudaError_t launch_list(const bf_scenario* scn, const uint64_t* idx, uint64_t count, uint32_t* ms, uint8_t* fe,
                        int grid, cudaStream_t st);

}  // namespace bfcapi
