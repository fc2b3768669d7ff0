// bf_kernels.cu -- the three search kernels, compiled once per tool-count
// bucket (-DBF_NT=<NT>).  All integer ALU work; no tensor cores, no HBM
// streaming beyond the eval kernel's 5 bytes of output per mapping.
//
//   eval   : one mapping per thread (grid-stride), coalesced stores of the
//            makespan (u32) and feasibility flag (u8) -- §2.1's T_e2e per mapping.
//   search : each thread walks a chunk of consecutive indices (decode once,
//            then base-3 increment), keeps the smallest packed key
//            (makespan << 32 | index), then warp shuffle-min -> block min ->
//            one 64-bit atomicMin per block.  Ties go to the lowest index
//            because the index is the key's low word.  This is the brute-force
//            oracle of §2.3 / §4.1 under the integer model.
//   batch  : as search, for many independent scenarios in one launch; each
//            block stages its scenario's tables in shared memory.
#include "bf_launch.h"

#ifndef BF_NT
#error "compile with -DBF_NT=<tool-count bucket>"
#endif

namespace bfk {
namespace {

__device__ __forceinline__ unsigned long long warp_min(unsigned long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = min(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  return v;
}

// Block-wide min of `v`, then one atomicMin into *dst from thread 0 (skipped
// when the block saw no mapping).
__device__ __forceinline__ void block_min_to(unsigned long long v, unsigned long long* dst) {
  __shared__ unsigned long long warp_best[kThreads / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_min(v);
  if (lane == 0) warp_best[warp] = v;
  __syncthreads();
  if (warp == 0) {
    v = lane < (int)(blockDim.x >> 5) ? warp_best[lane] : ~0ull;
    v = warp_min(v);
    if (lane == 0 && v != ~0ull) atomicMin(dst, v);
  }
}

template <int NT, typename TB>
__device__ __forceinline__ unsigned long long search_chunk(const TB& tb, const SmemTables& sd,
                                                           uint32_t idx, uint32_t cnt) {
  unsigned long long best = ~0ull;
  Digits dg = decode<NT>(idx);
#pragma unroll 1
  for (uint32_t j = 0; j < cnt; ++j) {
    const uint32_t ms = simulate<NT>(tb, sd, dg);
    best = min(best, ((unsigned long long)ms << 32) | (idx + j));
    increment(dg);
  }
  return best;
}

template <int NT>
__global__ void __launch_bounds__(kThreads) eval_kernel(const __grid_constant__ Tables tb,
                                                        uint32_t first, uint64_t count,
                                                        uint32_t* __restrict__ ms_out,
                                                        uint8_t* __restrict__ fe_out) {
  __shared__ SmemTables sd;
  load_smem_tables(tb, sd);
  __syncthreads();
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t j = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; j < count; j += stride) {
    const uint32_t ms = simulate<NT>(tb, sd, decode<NT>(first + (uint32_t)j));
    ms_out[j] = ms;
    fe_out[j] = ms != kInfeasible;
  }
}

template <int NT>
__global__ void __launch_bounds__(kThreads) search_kernel(const __grid_constant__ Tables tb,
                                                          uint32_t first, uint64_t count,
                                                          uint32_t per_thread,
                                                          unsigned long long* key) {
  __shared__ SmemTables sd;
  load_smem_tables(tb, sd);
  __syncthreads();
  const uint64_t off = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) * per_thread;
  unsigned long long best = ~0ull;
  if (off < count) {
    const uint32_t cnt = (uint32_t)min((uint64_t)per_thread, count - off);
    best = search_chunk<NT>(tb, sd, first + (uint32_t)off, cnt);
  }
  block_min_to(best, key);
}

template <int NT>
__global__ void __launch_bounds__(kThreads) batch_kernel(const Tables* __restrict__ all,
                                                         uint32_t per_thread,
                                                         uint32_t blocks_per_scenario,
                                                         unsigned long long* keys) {
  __shared__ Tables tb;
  __shared__ SmemTables sd;
  const uint32_t s = blockIdx.x / blocks_per_scenario;
  const uint32_t b = blockIdx.x - s * blocks_per_scenario;
  {
    const uint32_t* src = reinterpret_cast<const uint32_t*>(all + s);
    uint32_t* dst = reinterpret_cast<uint32_t*>(&tb);
    for (uint32_t w = threadIdx.x; w < sizeof(Tables) / 4; w += blockDim.x) dst[w] = src[w];
  }
  __syncthreads();
  load_smem_tables(tb, sd);
  __syncthreads();
  uint32_t total = 1;
  for (uint32_t i = 0; i < tb.n; ++i) total *= 3u;
  const uint64_t off = ((uint64_t)b * blockDim.x + threadIdx.x) * per_thread;
  unsigned long long best = ~0ull;
  if (off < total) {
    const uint32_t cnt = (uint32_t)min((uint64_t)per_thread, (uint64_t)total - off);
    best = search_chunk<NT>(tb, sd, (uint32_t)off, cnt);
  }
  block_min_to(best, keys + s);
}

}  // namespace

#define BF_PASTE2(a, b) a##b
#define BF_PASTE(a, b) BF_PASTE2(a, b)

cudaError_t BF_PASTE(launch_eval_nt, BF_NT)(const Tables& tb, uint32_t first, uint64_t count,
                                            uint32_t* ms, uint8_t* fe, int grid, cudaStream_t st) {
  eval_kernel<BF_NT><<<grid, kThreads, 0, st>>>(tb, first, count, ms, fe);
  return cudaGetLastError();
}

cudaError_t BF_PASTE(launch_search_nt, BF_NT)(const Tables& tb, uint32_t first, uint64_t count,
                                              uint32_t per_thread, unsigned long long* key,
                                              cudaStream_t st) {
  const uint64_t threads = (count + per_thread - 1) / per_thread;
  const uint64_t blocks = (threads + kThreads - 1) / kThreads;
  search_kernel<BF_NT><<<(unsigned)blocks, kThreads, 0, st>>>(tb, first, count, per_thread, key);
  return cudaGetLastError();
}

cudaError_t BF_PASTE(launch_batch_nt, BF_NT)(const Tables* d_tables, uint32_t count,
                                             uint32_t per_thread, uint32_t blocks_per_scenario,
                                             unsigned long long* keys, cudaStream_t st) {
  const uint64_t blocks = (uint64_t)count * blocks_per_scenario;
  batch_kernel<BF_NT><<<(unsigned)blocks, kThreads, 0, st>>>(d_tables, per_thread,
                                                              blocks_per_scenario, keys);
  return cudaGetLastError();
}

}  // namespace bfk
