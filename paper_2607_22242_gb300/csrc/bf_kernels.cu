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
// registers per thread.  Each thread keeps up to two saved window states of
// 2*NW+12 words in shared memory, so wider windows fit fewer blocks per SM.
#ifndef BF_MIN_BLOCKS
#if BF_NW <= 6
#define BF_MIN_BLOCKS 4
#elif BF_NW <= 12
#define BF_MIN_BLOCKS 3
#else
#define BF_MIN_BLOCKS 2
#endif
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
template <int WARPS = kWarps>
__device__ __forceinline__ void block_min_to(unsigned long long v, unsigned long long* dst) {
  __shared__ unsigned long long warp_best[WARPS];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_min(v);
  if (lane == 0) warp_best[warp] = v;
  __syncthreads();
  if (warp == 0) {
    v = lane < WARPS ? warp_best[lane] : ~0ull;
    v = warp_min(v);
    if (lane == 0 && v != ~0ull) atomicMin(dst, v);
  }
}

// Dynamic shared memory of every kernel: one saved window state per thread for
// the prefix checkpoint, and a second one for the inner checkpoint when the
// plan has an inner level; [word][thread] layout.
constexpr int kLaneWords = LaneWords<BF_NW>::value;
// Dynamic shared memory: the mid-part table (mid_part_words(3^M) words; the
// batch kernel reserves the largest) followed by the lane states.
constexpr size_t kDynSmemBytes = sizeof(uint32_t) * 2 * kLaneWords * kThreads;
constexpr size_t kDynSmemMaxBytes = sizeof(uint32_t) * kMaxMidPartWords + kDynSmemBytes;
inline size_t dyn_smem_bytes(uint32_t inner_levels, uint32_t mid_words) {
  return sizeof(uint32_t) * mid_words + (inner_levels ? kDynSmemBytes : kDynSmemBytes / 2);
}

template <int NP>
__global__ void __launch_bounds__(kThreads, BF_MIN_BLOCKS) eval_kernel(const __grid_constant__ Tables tb,
                                                                       const __grid_constant__ Tables tw,
                                                                       const __grid_constant__ Plan plan,
                                                                       uint32_t* __restrict__ ms_out,
                                                                       uint8_t* __restrict__ fe_out) {
  extern __shared__ uint32_t lane_state[];
  __shared__ SmemTables sd, sdw;
  __shared__ uint32_t rt[ReadyTable<NP>::size], rtw[ReadyTable<BF_NW>::size];
  load_smem_tables(tb, sd);
  load_smem_tables(tw, sdw);
  fill_ready_table<NP>(tb, rt);
  fill_ready_table<BF_NW>(tw, rtw);
  __syncthreads();
  const uint32_t task = blockIdx.x * kWarps + (threadIdx.x >> 5);
  if (task >= plan.groups * plan.m_parts) return;  // no block-level synchronisation follows
  StoreSink sink{plan.first, ms_out, fe_out};
  // Index ranges are always in the scenario's numbering.
  warp_task<NP, BF_NW, false>(tb, sd, rt, tw, sdw, rtw, plan, nullptr, task / plan.m_parts, task % plan.m_parts,
                       lane_state + threadIdx.x, lane_state + kLaneWords * kThreads + threadIdx.x, kThreads, sink);
}

// The search kernel's block shape: 128 threads, 7 per SM (72 registers, 28
// warps/SM instead of 24), for the 8-slot window, where that measured 3 %
// faster; the common shape elsewhere (wider windows spill at that register
// count).
constexpr int kSearchThreads = (BF_NW == 7 || BF_NW == 8) ? 128 : kThreads;
constexpr int kSearchWarps = kSearchThreads / 32;
constexpr int kSearchMinBlocks = (BF_NW == 7 || BF_NW == 8) ? 7 : BF_MIN_BLOCKS;
constexpr size_t kSearchSmemBytes = sizeof(uint32_t) * 2 * kLaneWords * kSearchThreads;
constexpr size_t kSearchSmemMaxBytes = sizeof(uint32_t) * kMaxMidPartWords + kSearchSmemBytes;

// RL: renumbered tables (whole-space searches, Plan::relabeled); the mid-part
// table then precedes the lane states in dynamic shared memory.
//
// Each block folds its minimum into sync->key; the last block to finish
// writes the result to *host_key (pinned host memory, mapped) and resets
// *sync for the next launch, so a search call is one launch with neither a
// key reset nor a result copy around it (8- and 12-tool searches 14 % and
// 5 % faster per call).  Persistent warps taking tasks from a counter and
// folding per warp measured slower: 16-tool layered search 2.70 -> 3.14 ms
// (issue 57 -> 48 % at the same occupancy), 19-tool search 0.5 %.
template <int NP, bool RL>
__global__ void __launch_bounds__(kSearchThreads, kSearchMinBlocks) search_kernel(const __grid_constant__ Tables tb,
                                                                                  const __grid_constant__ Tables tw,
                                                                                  const __grid_constant__ Plan plan,
                                                                                  SearchSync* sync,
                                                                                  unsigned long long* host_key) {
  extern __shared__ uint32_t dyn_smem[];
  uint32_t* const mpart = dyn_smem;
  uint32_t* const lane_state = dyn_smem + (RL ? mid_part_words(plan.pow3M) : 0u);
  __shared__ SmemTables sd, sdw;
  __shared__ uint32_t rt[ReadyTable<NP>::size], rtw[ReadyTable<BF_NW>::size];
  load_smem_tables(tb, sd);
  load_smem_tables(tw, sdw);
  fill_ready_table<NP>(tb, rt);
  fill_ready_table<BF_NW>(tw, rtw);
  if constexpr (RL) fill_mid_parts(plan, mpart);
  __syncthreads();
  const uint32_t task = blockIdx.x * kSearchWarps + (threadIdx.x >> 5), lane = threadIdx.x & 31u;
  MinKeySink sink;
  if (task < plan.groups * plan.m_parts)
    warp_task<NP, BF_NW, RL>(tb, sd, rt, tw, sdw, rtw, plan, mpart, task / plan.m_parts, task % plan.m_parts,
                         lane_state + threadIdx.x, lane_state + kLaneWords * kSearchThreads + threadIdx.x,
                         kSearchThreads, sink);
  (void)lane;
  block_min_to<kSearchWarps>(sink.best, &sync->key);
  if (threadIdx.x == 0) {
    __threadfence();
    if (atomicAdd(&sync->blocks_done, 1u) == gridDim.x - 1u) {
      // Every block has folded in its minimum: hand the result to the host
      // mirror and leave the launch state as the next launch expects it.
      *host_key = atomicExch(&sync->key, ~0ull);
      sync->blocks_done = 0u;
      __threadfence_system();
    }
  }
}

// Index-list evaluation: one mapping per thread (grid-stride), simulated from
// the start over NP >= n slots.  Indices >= total are flagged 0xFF.
template <int NP>
__global__ void __launch_bounds__(kThreads) list_kernel(const __grid_constant__ Tables tb, uint64_t total,
                                                        const uint64_t* __restrict__ idx, uint64_t count,
                                                        uint32_t* __restrict__ ms_out, uint8_t* __restrict__ fe_out) {
  __shared__ SmemTables sd;
  __shared__ uint32_t rt[ReadyTable<NP>::size];
  load_smem_tables(tb, sd);
  fill_ready_table<NP>(tb, rt);
  __syncthreads();
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t j = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; j < count; j += stride) {
    const uint64_t x = idx[j];
    uint32_t ms = kInfeasible;
    uint8_t fe = 0xFFu;
    if (x < total) {
      const Digits d = decode((uint32_t)x, tb.n);
      if ((d.que & tb.big_mask) == 0u) {
        State<NP> s;
        init_state(s, tb.all_mask);
        if (run<NP>(s, tb, sd, rt, d, 0u) == kRunFinished) ms = s.T;
      }
      fe = ms != kInfeasible;
    }
    ms_out[j] = ms;
    fe_out[j] = fe;
  }
}

// Pruned search, pass 1: one thread per prefix; keeps the prefixes whose
// checkpoint time plus the tail bound does not exceed the incumbent, the
// lowest feasible makespan among the ncand candidates the list kernel scored
// just before on the same stream (cand_ms / cand_fe).  Block 0's thread 0 also
// stores that bound for the host, which reads it with the survivor count.
template <int NP>
__global__ void __launch_bounds__(kThreads) prefix_filter_kernel(const __grid_constant__ Tables tb,
                                                                 const __grid_constant__ Plan plan,
                                                                 const uint32_t* __restrict__ cand_ms,
                                                                 const uint8_t* __restrict__ cand_fe, uint32_t ncand,
                                                                 uint32_t* __restrict__ survivors,
                                                                 uint32_t* __restrict__ count,
                                                                 uint32_t* __restrict__ bound_out) {
  __shared__ SmemTables sd;
  __shared__ uint32_t rt[ReadyTable<NP>::size];
  load_smem_tables(tb, sd);
  fill_ready_table<NP>(tb, rt);
  __syncthreads();
  uint32_t bound = kInfeasible;
  for (uint32_t j = 0; j < ncand; ++j)
    if (cand_fe[j] == 1u && cand_ms[j] < bound) bound = cand_ms[j];
  if (blockIdx.x == 0 && threadIdx.x == 0) *bound_out = bound;
  const uint64_t p = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (p >= plan.pow3P) return;
  Digits dgp;
  uint32_t T = 0u;
  if (prefix_checkpoint<NP, BF_NW>(tb, sd, rt, plan, (uint32_t)p, &dgp, &T, nullptr, 0u) &&
      (uint64_t)T + plan.tail_p <= bound)
    survivors[atomicAdd(count, 1u)] = (uint32_t)p;
}

// Pruned search, pass 2: warp tasks over the surviving prefixes (32 per group).
template <int NP>
__global__ void __launch_bounds__(kThreads, BF_MIN_BLOCKS) pruned_search_kernel(
    const __grid_constant__ Tables tb, const __grid_constant__ Tables tw, const __grid_constant__ Plan plan,
    const uint32_t* __restrict__ survivors, uint32_t nsurv, unsigned long long* key) {
  extern __shared__ uint32_t dyn_smem[];  // mid-part table, then the lane states
  uint32_t* const mpart = dyn_smem;
  uint32_t* const lane_state = dyn_smem + mid_part_words(plan.pow3M);
  __shared__ SmemTables sd, sdw;
  __shared__ uint32_t rt[ReadyTable<NP>::size], rtw[ReadyTable<BF_NW>::size];
  load_smem_tables(tb, sd);
  load_smem_tables(tw, sdw);
  fill_ready_table<NP>(tb, rt);
  fill_ready_table<BF_NW>(tw, rtw);
  fill_mid_parts(plan, mpart);
  __syncthreads();
  const uint32_t task = blockIdx.x * kWarps + (threadIdx.x >> 5);
  MinKeySink sink;
  if (task < plan.groups * plan.m_parts) {
    const uint32_t slot = (task / plan.m_parts) * 32u + (threadIdx.x & 31u);
    const bool valid = slot < nsurv;
    prefix_task<NP, BF_NW, true>(tb, sd, rt, tw, sdw, rtw, plan, mpart, valid ? survivors[slot] : 0u, valid,
                           task % plan.m_parts, lane_state + threadIdx.x,
                           lane_state + kLaneWords * kThreads + threadIdx.x, kThreads, sink);
  }
  block_min_to(sink.best, key);
}

}  // namespace

#define BF_PASTE2(a, b) a##b
#define BF_PASTE(a, b) BF_PASTE2(a, b)

static unsigned blocks_for(const Plan& plan) {
  const uint64_t tasks = (uint64_t)plan.groups * plan.m_parts;
  return (unsigned)((tasks + kWarps - 1) / kWarps);
}

// Each launcher picks the prefix width (BF_NW when the scenario fits, else 20).
#define BF_LAUNCH(KERNEL, FITS, INNER, MIDW, GRID, ...)                                         \
  do {                                                                                          \
    static std::atomic<uint64_t> ready_narrow{0}, ready_wide{0};                              \
    cudaError_t e_ = (FITS) ? allow_dyn_smem(KERNEL<BF_NW>, kDynSmemMaxBytes, &ready_narrow)   \
                            : allow_dyn_smem(KERNEL<kMaxTools>, kDynSmemMaxBytes, &ready_wide); \
    if (e_ != cudaSuccess) return e_;                                                           \
    const size_t smem_ = dyn_smem_bytes(INNER, MIDW);                                           \
    if (FITS)                                                                                \
      KERNEL<BF_NW><<<(GRID), kThreads, smem_, st>>>(__VA_ARGS__);                           \
    else                                                                                     \
      KERNEL<kMaxTools><<<(GRID), kThreads, smem_, st>>>(__VA_ARGS__);                       \
    return cudaGetLastError();                                                               \
  } while (0)

cudaError_t BF_PASTE(launch_eval_nw, BF_NW)(const Tables& tb, const Tables& tw, const Plan& plan,
                                            uint32_t* ms, uint8_t* fe, cudaStream_t st) {
  BF_LAUNCH(eval_kernel, tb.n <= (uint32_t)BF_NW, plan.I, 0u, blocks_for(plan), tb, tw, plan, ms, fe);
}

cudaError_t BF_PASTE(launch_search_nw, BF_NW)(const Tables& tb, const Tables& tw, const Plan& plan,
                                              SearchSync* sync, unsigned long long* host_key, cudaStream_t st) {
  static std::atomic<uint64_t> ready[4] = {};
  const bool fits = tb.n <= (uint32_t)BF_NW, rl = plan.relabeled != 0u;
  auto kernel = fits ? (rl ? search_kernel<BF_NW, true> : search_kernel<BF_NW, false>)
                     : (rl ? search_kernel<kMaxTools, true> : search_kernel<kMaxTools, false>);
  cudaError_t e = allow_dyn_smem(kernel, kSearchSmemMaxBytes, &ready[(fits ? 2 : 0) + (rl ? 1 : 0)]);
  if (e != cudaSuccess) return e;
  const size_t smem = sizeof(uint32_t) * (rl ? mid_part_words(plan.pow3M) : 0u) +
                      (plan.I ? kSearchSmemBytes : kSearchSmemBytes / 2);
  const uint64_t tasks = (uint64_t)plan.groups * plan.m_parts;
  const unsigned grid = (unsigned)((tasks + kSearchWarps - 1) / kSearchWarps);
  kernel<<<grid, kSearchThreads, smem, st>>>(tb, tw, plan, sync, host_key);
  return cudaGetLastError();
}

cudaError_t BF_PASTE(launch_prefix_filter_nw, BF_NW)(const Tables& tb, const Plan& plan, const uint32_t* cand_ms,
                                                     const uint8_t* cand_fe, uint32_t ncand, uint32_t* survivors,
                                                     uint32_t* count, uint32_t* bound_out, cudaStream_t st) {
  const unsigned grid = (unsigned)(((uint64_t)plan.pow3P + kThreads - 1) / kThreads);
  if (tb.n <= (uint32_t)BF_NW)
    prefix_filter_kernel<BF_NW><<<grid, kThreads, 0, st>>>(tb, plan, cand_ms, cand_fe, ncand, survivors, count,
                                                           bound_out);
  else
    prefix_filter_kernel<kMaxTools><<<grid, kThreads, 0, st>>>(tb, plan, cand_ms, cand_fe, ncand, survivors, count,
                                                               bound_out);
  return cudaGetLastError();
}

cudaError_t BF_PASTE(launch_pruned_search_nw, BF_NW)(const Tables& tb, const Tables& tw, const Plan& plan,
                                                     const uint32_t* survivors, uint32_t nsurv,
                                                     unsigned long long* key, cudaStream_t st) {
  BF_LAUNCH(pruned_search_kernel, tb.n <= (uint32_t)BF_NW, plan.I, mid_part_words(plan.pow3M), blocks_for(plan), tb,
            tw, plan, survivors, nsurv, key);
}

// Index lists run the whole scenario in one simulation: this unit handles n <= BF_NW.
cudaError_t BF_PASTE(launch_list_nw, BF_NW)(const Tables& tb, uint64_t total, const uint64_t* idx, uint64_t count,
                                            uint32_t* ms, uint8_t* fe, int grid, cudaStream_t st) {
  list_kernel<BF_NW><<<grid, kThreads, 0, st>>>(tb, total, idx, count, ms, fe);
  return cudaGetLastError();
}

}  // namespace bfk
