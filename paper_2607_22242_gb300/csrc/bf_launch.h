// bf_launch.h -- internal interface between the C ABI (bf_capi.cu) and the
// kernel translation units (bf_kernels.cu, compiled once per tool-count bucket).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "bf_sim.cuh"

namespace bfk {

constexpr int kThreads = 256;  // threads per block of every kernel

// Tool-count buckets: kernels are compiled for NT in this list; a scenario
// with n tools runs the smallest NT >= n (tools n..NT-1 count as done).
#define BF_FOR_EACH_BUCKET(X) X(4) X(6) X(8) X(10) X(12) X(14) X(16) X(18) X(19) X(20)

inline int bucket_for(uint32_t n) {
  const int b[] = {4, 6, 8, 10, 12, 14, 16, 18, 19, 20};
  for (int v : b)
    if ((int)n <= v) return v;
  return -1;
}

#define BF_DECLARE_BUCKET(NT)                                                                   \
  cudaError_t launch_eval_nt##NT(const Tables& tb, uint32_t first, uint64_t count,               \
                                 uint32_t* ms, uint8_t* fe, int grid, cudaStream_t st);          \
  cudaError_t launch_search_nt##NT(const Tables& tb, uint32_t first, uint64_t count,             \
                                   uint32_t per_thread, unsigned long long* key, cudaStream_t st); \
  cudaError_t launch_batch_nt##NT(const Tables* d_tables, uint32_t count, uint32_t per_thread,   \
                                  uint32_t blocks_per_scenario, unsigned long long* keys,        \
                                  cudaStream_t st);
BF_FOR_EACH_BUCKET(BF_DECLARE_BUCKET)
#undef BF_DECLARE_BUCKET

}  // namespace bfk
