// bf_kernels.cu -- the three search kernels, compiled once per window width
// (-DBF_NW=<slots>).  All integer ALU work: no tensor cores, and no HBM
// streaming beyond the eval kernel's 5 bytes of output per mapping.
//
// Work decomposition (the same in all three kernels; see bfk::Plan).  A
// mapping index is idx = p + 3^P * (m + 3^M * i).  Each warp owns one prefix
// p (the modes of tools [0, P)); its 32 lanes simulate that prefix together --
// identical control flow -- until the first instant a tool >= P would become
// ready, and lane 0 saves the state (restricted to the window [W0, n)) in
// shared memory.  Lane l then resumes it for mid combinations m = l, l+32, ...
// with a simulation only NW slots wide; with an inner level it saves its own
// state again when the first inner tool would become ready and resumes that
// for each inner combination i.  Every mapping's makespan is still simulated
// event by event; only the common part of the histories is shared.
//
//   eval   : writes the makespan (u32) and feasibility flag (u8) of every
//            mapping in [first, last] -- §2.1's T_e2e per mapping.
//   search : keeps the smallest packed key (makespan << 32 | index) per lane,
//            then warp shuffle-min -> block min -> one 64-bit atomicMin per
//            block.  Ties go to the lowest index (the key's low word).  This is
//            the brute-force oracle of §2.3 / §4.1 under the integer model.
//   batch  : as search, for many independent scenarios in one launch; each
//            block stages its scenario's tables and plan in shared memory.
#include "bf_enum.cuh"
#include "bf_launch.h"

#ifndef BF_NW
#error "compile with -DBF_NW=<window slot count>"
#endif

// Minimum resident blocks per SM requested from the compiler, which caps the
// registers per thread (measured on GB300: 4 blocks of 256 threads is fastest
// for windows of up to 8 slots, 3 up to 16, 2 above; 2 for the batch kernel,
// whose tables sit in shared memory).
#ifndef BF_MIN_BLOCKS
#if BF_NW <= 8
#define BF_MIN_BLOCKS 4
#elif BF_NW <= 16
#define BF_MIN_BLOCKS 3
#else
#define BF_MIN_BLOCKS 2
#endif
#endif
#ifndef BF_MIN_BLOCKS_BATCH
#define BF_MIN_BLOCKS_BATCH 2
#endif

namespace bfk {
namespace {

constexpr int kWarps = kThreads / 32;

__device__ __forceinline__ unsigned long long warp_min(unsigned long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = min(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  return v;
}

// Block-wide min of `v`, then one atomicMin into *dst from thread 0 (skipped
// when the block found nothing).
__device__ __forceinline__ void block_min_to(unsigned long long v, unsigned long long* dst) {
  __shared__ unsigned long long warp_best[kWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_min(v);
  if (lane == 0) warp_best[warp] = v;
  __syncthreads();
  if (warp == 0) {
    v = lane < kWarps ? warp_best[lane] : ~0ull;
    v = warp_min(v);
    if (lane == 0 && v != ~0ull) atomicMin(dst, v);
  }
}

template <int NP>
__global__ void __launch_bounds__(kThreads, BF_MIN_BLOCKS) eval_kernel(const __grid_constant__ Tables tb,
                                                        const __grid_constant__ Tables tw,
                                                        const __grid_constant__ Plan plan,
                                                        uint32_t* __restrict__ ms_out,
                                                        uint8_t* __restrict__ fe_out) {
  __shared__ SmemTables sd, sdw;
  __shared__ Snapshot snap[kWarps];
  __shared__ uint32_t lane_state[LaneWords<BF_NW>::value * kThreads];
  load_smem_tables(tb, sd);
  load_smem_tables(tw, sdw);
  __syncthreads();
  const int warp = threadIdx.x >> 5;
  const uint64_t p64 = (uint64_t)plan.p_lo + (uint64_t)blockIdx.x * kWarps + warp;
  if (p64 > plan.p_hi) return;  // no block-level synchronisation follows
  const uint32_t p = (uint32_t)p64;
  Digits dgp;
  const bool ok = prefix_phase<NP>(tb, sd, plan, p, dgp, snap[warp]);
  StoreSink sink{plan.first, ms_out, fe_out};
  lane_mappings<BF_NW>(tw, sdw, plan, p, ok, dgp, snap[warp], lane_state + threadIdx.x, kThreads, sink);
}

template <int NP>
__global__ void __launch_bounds__(kThreads, BF_MIN_BLOCKS) search_kernel(const __grid_constant__ Tables tb,
                                                          const __grid_constant__ Tables tw,
                                                          const __grid_constant__ Plan plan,
                                                          unsigned long long* key) {
  __shared__ SmemTables sd, sdw;
  __shared__ Snapshot snap[kWarps];
  __shared__ uint32_t lane_state[LaneWords<BF_NW>::value * kThreads];
  load_smem_tables(tb, sd);
  load_smem_tables(tw, sdw);
  __syncthreads();
  const int warp = threadIdx.x >> 5;
  const uint64_t p64 = (uint64_t)plan.p_lo + (uint64_t)blockIdx.x * kWarps + warp;
  MinKeySink sink;
  if (p64 <= plan.p_hi) {
    const uint32_t p = (uint32_t)p64;
    Digits dgp;
    if (prefix_phase<NP>(tb, sd, plan, p, dgp, snap[warp])) lane_mappings<BF_NW>(tw, sdw, plan, p, true, dgp, snap[warp], lane_state + threadIdx.x, kThreads, sink);
  }
  block_min_to(sink.best, key);
}

// One record per scenario of a batch: full tables, window tables and plan.
template <int NP>
__global__ void __launch_bounds__(kThreads, BF_MIN_BLOCKS_BATCH) batch_kernel(const BatchRecord* __restrict__ recs,
                                                         uint32_t blocks_per_scenario,
                                                         unsigned long long* keys) {
  __shared__ BatchRecord rec;
  __shared__ SmemTables sd, sdw;
  __shared__ Snapshot snap[kWarps];
  __shared__ uint32_t lane_state[LaneWords<BF_NW>::value * kThreads];
  const uint32_t sc = blockIdx.x / blocks_per_scenario;
  const uint32_t b = blockIdx.x - sc * blocks_per_scenario;
  {
    const uint32_t* src = reinterpret_cast<const uint32_t*>(recs + sc);
    uint32_t* dst = reinterpret_cast<uint32_t*>(&rec);
    for (uint32_t w = threadIdx.x; w < sizeof(BatchRecord) / 4; w += blockDim.x) dst[w] = src[w];
  }
  __syncthreads();
  load_smem_tables(rec.full, sd);
  load_smem_tables(rec.window, sdw);
  __syncthreads();
  const int warp = threadIdx.x >> 5;
  const uint64_t p64 = (uint64_t)rec.plan.p_lo + (uint64_t)b * kWarps + warp;
  MinKeySink sink;
  if (p64 <= rec.plan.p_hi) {
    const uint32_t p = (uint32_t)p64;
    Digits dgp;
    if (prefix_phase<NP>(rec.full, sd, rec.plan, p, dgp, snap[warp]))
      lane_mappings<BF_NW>(rec.window, sdw, rec.plan, p, true, dgp, snap[warp], lane_state + threadIdx.x,
                           kThreads, sink);
  }
  block_min_to(sink.best, keys + sc);
}

}  // namespace

#define BF_PASTE2(a, b) a##b
#define BF_PASTE(a, b) BF_PASTE2(a, b)

static unsigned blocks_for(const Plan& plan) {
  const uint64_t warps = (uint64_t)plan.p_hi - plan.p_lo + 1;
  return (unsigned)((warps + kWarps - 1) / kWarps);
}

// The prefix simulation runs BF_NW slots wide when the scenario fits (n <= BF_NW),
// else kMaxTools wide.
cudaError_t BF_PASTE(launch_eval_nw, BF_NW)(const Tables& tb, const Tables& tw, const Plan& plan,
                                            uint32_t* ms, uint8_t* fe, cudaStream_t st) {
  if (tb.n <= (uint32_t)BF_NW)
    eval_kernel<BF_NW><<<blocks_for(plan), kThreads, 0, st>>>(tb, tw, plan, ms, fe);
  else
    eval_kernel<kMaxTools><<<blocks_for(plan), kThreads, 0, st>>>(tb, tw, plan, ms, fe);
  return cudaGetLastError();
}

cudaError_t BF_PASTE(launch_search_nw, BF_NW)(const Tables& tb, const Tables& tw, const Plan& plan,
                                              unsigned long long* key, cudaStream_t st) {
  if (tb.n <= (uint32_t)BF_NW)
    search_kernel<BF_NW><<<blocks_for(plan), kThreads, 0, st>>>(tb, tw, plan, key);
  else
    search_kernel<kMaxTools><<<blocks_for(plan), kThreads, 0, st>>>(tb, tw, plan, key);
  return cudaGetLastError();
}

cudaError_t BF_PASTE(launch_batch_nw, BF_NW)(const BatchRecord* d_recs, uint32_t count, uint32_t nmax,
                                             uint32_t blocks_per_scenario, unsigned long long* keys,
                                             cudaStream_t st) {
  const uint64_t blocks = (uint64_t)count * blocks_per_scenario;
  if (nmax <= (uint32_t)BF_NW)
    batch_kernel<BF_NW><<<(unsigned)blocks, kThreads, 0, st>>>(d_recs, blocks_per_scenario, keys);
  else
    batch_kernel<kMaxTools><<<(unsigned)blocks, kThreads, 0, st>>>(d_recs, blocks_per_scenario, keys);
  return cudaGetLastError();
}

}  // namespace bfk
