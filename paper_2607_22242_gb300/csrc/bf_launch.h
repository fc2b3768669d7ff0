// bf_launch.h -- internal interface between the C ABI (bf_capi.cu) and the
// kernel translation units (bf_kernels.cu, compiled once per window width).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "bf_sim.cuh"

namespace bfk {

constexpr int kThreads = 256;  // threads per block of every kernel (8 warps, one prefix each)

// Raise a kernel's dynamic shared memory limit to `bytes` on the current
// device, once per device: the attribute belongs to the kernel's instance on
// each device.  `done` is that kernel's set of devices already prepared.
template <typename K>
inline cudaError_t allow_dyn_smem(K kernel, size_t bytes, std::atomic<uint64_t>* done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = (dev >= 0 && dev < 64) ? (1ull << dev) : 0ull;
  if (bit && (done->load(std::memory_order_acquire) & bit)) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e == cudaSuccess && bit) done->fetch_or(bit, std::memory_order_acq_rel);
  return e;
}

// State of one launch of a whole-space search (the search kernel or the
// lane-tree search of one scenario), in device memory: the best key found so
// far, the blocks that have finished and the next root of the lane tree's
// shared tail.  It holds (~0, 0, 0) between launches: the last block of a
// launch writes the result out and puts it back.
struct SearchSync {
  unsigned long long key;
  uint32_t blocks_done;
  uint32_t next_root;
};

#define BF_DECLARE_BUCKET(NW)                                                                       \
  cudaError_t launch_eval_nw##NW(const Tables& tb, const Tables& tw, const Plan& plan, uint32_t* ms, \
                                 uint8_t* fe, cudaStream_t st);                                     \
  cudaError_t launch_search_nw##NW(const Tables& tb, const Tables& tw, const Plan& plan,             \
                                   SearchSync* sync, unsigned long long* host_key, cudaStream_t st);  \
  cudaError_t launch_list_nw##NW(const Tables& tb, uint64_t total, const uint64_t* idx, uint64_t count, \
                                 uint32_t* ms, uint8_t* fe, int grid, cudaStream_t st);             \
  cudaError_t launch_prefix_filter_nw##NW(const Tables& tb, const Plan& plan, const uint32_t* cand_ms,   \
                                          const uint8_t* cand_fe, uint32_t ncand, uint32_t* survivors,   \
                                          uint32_t* count, uint32_t* bound_out, cudaStream_t st);        \
  cudaError_t launch_pruned_search_nw##NW(const Tables& tb, const Tables& tw, const Plan& plan,       \
                                          const uint32_t* survivors, uint32_t nsurv,                 \
                                          unsigned long long* key, cudaStream_t st);
BF_FOR_EACH_BUCKET(BF_DECLARE_BUCKET)
#undef BF_DECLARE_BUCKET

}  // namespace bfk
