// bf_lanetree_launch.h -- internal interface between the C ABI (bf_capi.cu)
// and the lane-tree batch kernel (bf_lanetree.cu).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "bf_lanetree.cuh"

namespace bfk {

// The lane-tree batch kernel: scenarios of up to kLtBatchTools tools;
// d_first_block[count + 1] holds each scenario's first block (prefix sums of
// LaneTreeRecord::nblocks), `blocks` = its last entry, nmax the largest n.
// keys[s] must hold ~0 before the launch; it receives the lowest key
// (makespan << 32 | canonical index) of scenario s.
cudaError_t launch_lanetree(const LaneTreeRecord* d_recs, const uint32_t* d_first_block, uint32_t count,
                            uint32_t blocks, uint32_t nmax, unsigned long long* keys, cudaStream_t st);

}  // namespace bfk
