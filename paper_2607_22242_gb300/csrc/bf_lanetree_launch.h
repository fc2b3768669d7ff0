// bf_lanetree_launch.h -- internal interface between the C ABI (bf_capi.cu)
// and the lane-tree kernels (bf_lanetree.cu).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "bf_lanetree.cuh"
#include "bf_launch.h"

namespace bfk {

// The lane-tree batch kernel: scenarios of up to kLtMaxTools tools, one launch
// per group of the same table form (up to kLtBatchTools tools, up to
// kLtNarrowTools, up to kLtMaxTools; nmax, the group's largest n, picks it);
// d_first_block[count + 1] holds each scenario's first block (prefix sums of
// LaneTreeRecord::nblocks), `blocks` = its last entry.
// keys[s] must hold ~0 before the launch; it receives the lowest key
// (makespan << 32 | canonical index) of scenario s.
cudaError_t launch_lanetree(const LaneTreeRecord* d_recs, const uint32_t* d_first_block, uint32_t count,
                            uint32_t blocks, uint32_t nmax, unsigned long long* keys, cudaStream_t st);

constexpr uint32_t kLtLaunchThreads = 256;  // threads per block of both kernels

// The one-scenario lane-tree search: every lane of the current device on one
// record of kLtSingleMinTools to kLtMaxTools tools (full searches of such
// scenarios take it when bf_plan.h lanetree_preferred says so).  The record's x gives 3^x >= lanes *
// kLtSingleRootsPerLane roots; the blocks are dealt kLtStaticShare of them
// in advance, the rest go to whichever lanes ask first.
constexpr uint32_t kLtSingleMinTools = 10;
constexpr uint64_t kLtSingleRootsPerLane = 2;
constexpr uint64_t kLtStaticShareNum = 1, kLtStaticShareDen = 2;

// Blocks of one launch for an n-tool record on the current device: every
// resident slot of every SM.
cudaError_t lanetree_single_blocks(uint32_t n, uint32_t* blocks);

// One launch over d_rec (n tools, roots [0, 3^x)); *sync must hold (~0, 0, 0)
// and is left so; the lowest key (makespan << 32 | canonical index, ~0 when
// no mapping is feasible) is written to *host_key by the last block.
cudaError_t launch_lanetree_single(const LaneTreeRecord* d_rec, uint32_t n, uint32_t x, uint32_t blocks,
                                   SearchSync* sync, unsigned long long* host_key, cudaStream_t st);

}  // namespace bfk
