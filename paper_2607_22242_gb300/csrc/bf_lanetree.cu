// bf_lanetree.cu -- the lane-tree kernels (bf_lanetree.cuh): the full search
// of many small scenarios in one launch, one or more blocks per scenario, and
// the full search of one scenario by every lane of the GPU; every lane walks
// its roots' trees of checkpoints.
#include "bf_enum.cuh"
#include "bf_lanetree_launch.h"
#include "bf_launch.h"

namespace bfk {
namespace {

constexpr int kLtThreads = (int)kLtLaunchThreads;
// Resident blocks per SM both kernels are compiled for: the registers of 5
// blocks of 256 threads (up to 48 a thread) instead of the 44-47 the
// compiler picks unbounded, same occupancy: batch call 12.86 -> 12.70 ms,
// 16-tool full search 1.60 -> 1.58 ms.
constexpr int kLtBlocksPerSm = 5;
// The wide one-scenario kernel (17 to 20 tools) holds 11 state words per
// checkpoint and 20 per-tool words per lane: 4 blocks fit an SM.
constexpr int kLtWideBlocksPerSm = 4;

__device__ __forceinline__ unsigned long long lt_warp_min(unsigned long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = min(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  return v;
}

// The block's copy of a record and the tables derived from it.
template <uint32_t NC>
__device__ __forceinline__ void lt_load_record(LtSharedT<NC>& S, const LaneTreeRecord* rec) {
  const uint32_t* src = reinterpret_cast<const uint32_t*>(rec);
  uint32_t* dst = reinterpret_cast<uint32_t*>(&S.rec);
  for (uint32_t w = threadIdx.x; w < sizeof(LaneTreeRecord) / 4; w += blockDim.x) dst[w] = src[w];
  __syncthreads();
  lt_fill_tables(S);
}

// Block b searches roots [3^x * j / nblocks, 3^x * (j + 1) / nblocks) of
// scenario s, where first_block[s] <= b < first_block[s + 1] and j = b -
// first_block[s]; the lowest key (makespan << 32 | canonical index) it finds
// goes to keys[s] by one atomicMin per warp.  NC table chunks and the queue
// form W as for the one-scenario kernel: <2, false> up to 12 tools, <3,
// false> up to 16, <4, true> up to 20.
template <uint32_t NC, bool W>
__global__ void __launch_bounds__(kLtThreads, W ? kLtWideBlocksPerSm : kLtBlocksPerSm)
    lanetree_kernel(const LaneTreeRecord* __restrict__ recs, const uint32_t* __restrict__ first_block, uint32_t count,
                    unsigned long long* keys) {
  extern __shared__ uint32_t lt_rows_smem[];
  __shared__ LtSharedT<NC> S;
  uint32_t lo = 0u, hi = count;  // first_block[lo] <= blockIdx.x < first_block[hi]
  while (hi - lo > 1u) {
    const uint32_t mid = (lo + hi) >> 1;
    if (first_block[mid] <= blockIdx.x) lo = mid;
    else hi = mid;
  }
  const uint32_t sc = lo;
  lt_load_record(S, recs + sc);
  if (threadIdx.x == 0) {
    uint32_t roots = 1u;
    for (uint32_t t = 0; t < S.rec.x; ++t) roots *= 3u;
    const uint64_t j = blockIdx.x - first_block[sc], nb = S.rec.nblocks;
    S.root_next = (uint32_t)(roots * j / nb);
    S.root_end = (uint32_t)(roots * (j + 1u) / nb);
  }
  __syncthreads();
  MinKeySink sink;
  LtSharedT<NC>& Sref = S;
  lt_lane<NC, W>(S, lt_rows_smem + threadIdx.x, blockDim.x,
          [&Sref]() {
            const uint32_t r = atomicAdd(&Sref.root_next, 1u);
            return r < Sref.root_end ? r : 0xFFFFFFFFu;
          },
          sink);
  const unsigned long long best = lt_warp_min(sink.best);
  if ((threadIdx.x & 31u) == 0u && best != ~0ull) atomicMin(keys + sc, best);
}

// The whole search of one scenario, one block per resident slot of the GPU.
// Roots [0, static_roots) are split evenly over the blocks and handed out by
// a counter in each block's shared memory; a lane whose block has none left
// takes the next root of [static_roots, 3^x) from sync->next_root (one
// atomic per group of lanes of a warp asking at once), so lanes keep busy
// until the last roots.  The lowest key goes to sync->key; the last block to
// finish copies it to *host_key (pinned host memory the device addresses)
// and puts sync back to (~0, 0, 0).
// NC table chunks, W the wide queue form: <3, false> up to 16 tools, <4,
// true> up to 20.
template <uint32_t NC, bool W>
__global__ void __launch_bounds__(kLtThreads, W ? kLtWideBlocksPerSm : kLtBlocksPerSm)
    lanetree_single_kernel(const LaneTreeRecord* __restrict__ rec, uint32_t static_roots, SearchSync* sync,
                           unsigned long long* host_key) {
  extern __shared__ uint32_t lt_rows_smem[];
  __shared__ LtSharedT<NC> S;
  lt_load_record(S, rec);
  if (threadIdx.x == 0) {
    const uint64_t j = blockIdx.x, nb = gridDim.x;
    S.root_next = (uint32_t)(static_roots * j / nb);
    S.root_end = (uint32_t)(static_roots * (j + 1u) / nb);
  }
  __syncthreads();
  uint32_t roots = 1u;
  for (uint32_t t = 0; t < S.rec.x; ++t) roots *= 3u;
  MinKeySink sink;
  LtSharedT<NC>& Sref = S;
  lt_lane<NC, W>(S, lt_rows_smem + threadIdx.x, blockDim.x,
          [&Sref, sync, static_roots, roots]() {
            const uint32_t r = atomicAdd(&Sref.root_next, 1u);
            if (r < Sref.root_end) return r;
            const uint32_t group = __activemask(), lane = threadIdx.x & 31u;
            const uint32_t leader = __ffs(group) - 1u;
            uint32_t base = 0u;
            if (lane == leader) base = atomicAdd(&sync->next_root, (uint32_t)__popc(group));
            base = __shfl_sync(group, base, leader);
            const uint32_t t = static_roots + base + __popc(group & ((1u << lane) - 1u));
            return t < roots ? t : 0xFFFFFFFFu;
          },
          sink);
  const unsigned long long best = lt_warp_min(sink.best);
  if ((threadIdx.x & 31u) == 0u && best != ~0ull) atomicMin(&sync->key, best);
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    if (atomicAdd(&sync->blocks_done, 1u) == gridDim.x - 1u) {
      *host_key = atomicExch(&sync->key, ~0ull);
      sync->blocks_done = 0u;
      sync->next_root = 0u;
      __threadfence_system();
    }
  }
}

template <bool W = false>
size_t lt_smem_bytes(uint32_t n) { return sizeof(uint32_t) * lt_rows<W>(n) * kLtThreads; }

// The one-scenario kernel for n tools, with its dynamic shared memory allowed
// (once per device and form).
using SingleKernel = void (*)(const LaneTreeRecord*, uint32_t, SearchSync*, unsigned long long*);
cudaError_t single_kernel_for(uint32_t n, SingleKernel* k, size_t* smem) {
  static std::atomic<uint64_t> ready_narrow{0}, ready_wide{0};
  if (n <= kLtNarrowTools) {
    *k = lanetree_single_kernel<3, false>;
    *smem = lt_smem_bytes<false>(n);
    return allow_dyn_smem(lanetree_single_kernel<3, false>, lt_smem_bytes<false>(kLtNarrowTools), &ready_narrow);
  }
  *k = lanetree_single_kernel<4, true>;
  *smem = lt_smem_bytes<true>(n);
  return allow_dyn_smem(lanetree_single_kernel<4, true>, lt_smem_bytes<true>(kLtMaxTools), &ready_wide);
}

}  // namespace

cudaError_t launch_lanetree(const LaneTreeRecord* d_recs, const uint32_t* d_first_block, uint32_t count,
                            uint32_t blocks, uint32_t nmax, unsigned long long* keys, cudaStream_t st) {
  static std::atomic<uint64_t> ready2{0}, ready3{0}, ready4{0};
  cudaError_t e = cudaSuccess;
  if (nmax <= kLtBatchTools) {
    e = allow_dyn_smem(lanetree_kernel<2, false>, lt_smem_bytes<false>(kLtBatchTools), &ready2);
    if (e == cudaSuccess)
      lanetree_kernel<2, false><<<blocks, kLtThreads, lt_smem_bytes<false>(nmax), st>>>(d_recs, d_first_block, count,
                                                                                       keys);
  } else if (nmax <= kLtNarrowTools) {
    e = allow_dyn_smem(lanetree_kernel<3, false>, lt_smem_bytes<false>(kLtNarrowTools), &ready3);
    if (e == cudaSuccess)
      lanetree_kernel<3, false><<<blocks, kLtThreads, lt_smem_bytes<false>(nmax), st>>>(d_recs, d_first_block, count,
                                                                                       keys);
  } else {
    e = allow_dyn_smem(lanetree_kernel<4, true>, lt_smem_bytes<true>(kLtMaxTools), &ready4);
    if (e == cudaSuccess)
      lanetree_kernel<4, true><<<blocks, kLtThreads, lt_smem_bytes<true>(nmax), st>>>(d_recs, d_first_block, count,
                                                                                     keys);
  }
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t lanetree_single_blocks(uint32_t n, uint32_t* blocks) {
  SingleKernel k = nullptr;
  size_t smem = 0;
  cudaError_t e = single_kernel_for(n, &k, &smem);
  int dev = 0, sms = 0, per_sm = 0;
  if (e == cudaSuccess) e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, kLtThreads, smem);
  if (e != cudaSuccess) return e;
  *blocks = (uint32_t)(sms > 0 ? sms : 1) * (uint32_t)(per_sm > 0 ? per_sm : 1);
  return cudaSuccess;
}

cudaError_t launch_lanetree_single(const LaneTreeRecord* d_rec, uint32_t n, uint32_t x, uint32_t blocks,
                                   SearchSync* sync, unsigned long long* host_key, cudaStream_t st) {
  SingleKernel k = nullptr;
  size_t smem = 0;
  cudaError_t e = single_kernel_for(n, &k, &smem);
  if (e != cudaSuccess) return e;
  uint64_t roots = 1;
  for (uint32_t t = 0; t < x; ++t) roots *= 3u;
  const uint32_t static_roots = (uint32_t)(roots * kLtStaticShareNum / kLtStaticShareDen);
  k<<<blocks, kLtThreads, smem, st>>>(d_rec, static_roots, sync, host_key);
  return cudaGetLastError();
}

}  // namespace bfk
