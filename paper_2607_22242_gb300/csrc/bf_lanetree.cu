// bf_lanetree.cu -- the lane-tree batch kernel (bf_lanetree.cuh): the full
// search of many small scenarios in one launch, one or more blocks per
// scenario, every lane walking its roots' trees of checkpoints.
#include "bf_enum.cuh"
#include "bf_lanetree_launch.h"
#include "bf_launch.h"

namespace bfk {
namespace {

constexpr int kLtThreads = 256;

__device__ __forceinline__ unsigned long long lt_warp_min(unsigned long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = min(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  return v;
}

// Block b searches roots [3^x * j / nblocks, 3^x * (j + 1) / nblocks) of
// scenario s, where first_block[s] <= b < first_block[s + 1] and j = b -
// first_block[s]; the lowest key (makespan << 32 | canonical index) it finds
// goes to keys[s] by one atomicMin per warp.
__global__ void __launch_bounds__(kLtThreads) lanetree_kernel(const LaneTreeRecord* __restrict__ recs,
                                                             const uint32_t* __restrict__ first_block,
                                                             uint32_t count, unsigned long long* keys) {
  extern __shared__ uint32_t lt_rows_smem[];
  __shared__ LtShared S;
  uint32_t lo = 0u, hi = count;  // first_block[lo] <= blockIdx.x < first_block[hi]
  while (hi - lo > 1u) {
    const uint32_t mid = (lo + hi) >> 1;
    if (first_block[mid] <= blockIdx.x) lo = mid;
    else hi = mid;
  }
  const uint32_t sc = lo;
  {
    const uint32_t* src = reinterpret_cast<const uint32_t*>(recs + sc);
    uint32_t* dst = reinterpret_cast<uint32_t*>(&S.rec);
    for (uint32_t w = threadIdx.x; w < sizeof(LaneTreeRecord) / 4; w += blockDim.x) dst[w] = src[w];
  }
  __syncthreads();
  lt_fill_tables(S);
  if (threadIdx.x == 0) {
    uint32_t roots = 1u;
    for (uint32_t t = 0; t < S.rec.x; ++t) roots *= 3u;
    const uint64_t j = blockIdx.x - first_block[sc], nb = S.rec.nblocks;
    S.root_next = (uint32_t)(roots * j / nb);
    S.root_end = (uint32_t)(roots * (j + 1u) / nb);
  }
  __syncthreads();
  MinKeySink sink;
  LtShared& Sref = S;
  lt_lane(S, lt_rows_smem + threadIdx.x, blockDim.x,
          [&Sref]() {
            const uint32_t r = atomicAdd(&Sref.root_next, 1u);
            return r < Sref.root_end ? r : 0xFFFFFFFFu;
          },
          sink);
  const unsigned long long best = lt_warp_min(sink.best);
  if ((threadIdx.x & 31u) == 0u && best != ~0ull) atomicMin(keys + sc, best);
}

}  // namespace

cudaError_t launch_lanetree(const LaneTreeRecord* d_recs, const uint32_t* d_first_block, uint32_t count,
                            uint32_t blocks, uint32_t nmax, unsigned long long* keys, cudaStream_t st) {
  static std::atomic<uint64_t> ready{0};
  const size_t smem = sizeof(uint32_t) * lt_rows(kLtBatchTools) * kLtThreads;
  cudaError_t e = allow_dyn_smem(lanetree_kernel, smem, &ready);
  if (e != cudaSuccess) return e;
  lanetree_kernel<<<blocks, kLtThreads, sizeof(uint32_t) * lt_rows(nmax) * kLtThreads, st>>>(d_recs, d_first_block,
                                                                                           count, keys);
  return cudaGetLastError();
}

}  // namespace bfk
