// bf_tree.cu -- kernels of the tree search (bf_tree.cuh) and the index-list
// evaluation for scenarios of up to 32 tools.  All state is 32 slots wide.
//
//   tree_root_kernel   : writes the root node (nothing assigned, T = 0).
//   tree_expand_kernel : one thread per (parent, mode of the next tool); the
//                        child is resumed to its checkpoint, bounded, and the
//                        survivors are appended to the next level's buffer
//                        (one atomicAdd per warp on a running total).
//   tree_leaf_kernel   : one warp per 32 leaf-level nodes (one per lane) and a
//                        chunk of the radix^D combinations of the last D tools,
//                        walked in lockstep over the leaf window (tools from the
//                        lowest one that can still be running at a leaf
//                        checkpoint; compiled for 8..32 slots); per-block best
//                        (makespan, index) merged into one 16-byte record by
//                        compare-and-swap.
//   wide_list_kernel   : makespan of each listed mapping, simulated whole.
#include <cuda_runtime.h>

#include "bf_launch.h"
#include "bf_plan.h"
#include "bf_tree.h"

namespace bfk {
namespace {

constexpr int kTreeThreads = 256;
constexpr int kTreeWarps = kTreeThreads / 32;
constexpr int kNW = NodeWords<kTreeSlots>::value;

__device__ __forceinline__ uint32_t read_bound(const uint32_t* bound) {
  return *reinterpret_cast<const volatile uint32_t*>(bound);
}

__global__ void tree_root_kernel(const __grid_constant__ TablesW tb, uint32_t* buf, uint32_t cap) {
  State<kTreeSlots> s;
  init_state(s, tb.all_mask);
  store_node(s, Digits{0u, 0u}, buf, cap, 0u);
}

__global__ void __launch_bounds__(kTreeThreads, 2) tree_expand_kernel(
    const __grid_constant__ TablesW tb, const __grid_constant__ TreeConsts tc, const uint32_t* __restrict__ src,
    uint32_t src_cap, uint32_t lo, uint32_t cnt, uint32_t d, uint32_t* __restrict__ dst, uint32_t dst_cap,
    unsigned long long* appended, unsigned long long base_total, const uint32_t* bound, TreeCounters* ctr) {
  __shared__ SmemTablesW sd;
  __shared__ uint32_t rt[ReadyTable<kTreeSlots>::size];
  __shared__ uint32_t ef[kTreeSlots * kTreeThreads];  // forward_bound scratch, [tool][thread]
  load_smem_tables(tb, sd);
  fill_ready_table<kTreeSlots>(tb, rt);
  __syncthreads();
  // Thread t: mode a = t / cnt of tool d for parent lo + t % cnt, so that a
  // warp's lanes hold neighbouring parents with the same new mode.
  const uint32_t t = blockIdx.x * kTreeThreads + threadIdx.x;
  const uint32_t a = t / max(cnt, 1u), j = t - a * cnt;
  bool keep = false;
  State<kTreeSlots> s;
  Digits dg{0u, 0u};
  if (a < tc.radix) {
    load_node(src, src_cap, lo + j, s, dg);
    keep = expand_child<kTreeSlots>(tb, sd, rt, tc, s, dg, d, a, read_bound(bound), ef + threadIdx.x, kTreeThreads);
  }
  const uint32_t ballot = __ballot_sync(0xFFFFFFFFu, keep);
  if (ballot == 0u) return;
  const uint32_t lane = threadIdx.x & 31u;
  const uint32_t leader = __ffs(ballot) - 1;
  // `appended` counts every node appended by every expansion of this search;
  // this launch's children get slots from base_total (its value at launch) on.
  unsigned long long base = 0ull;
  if (lane == leader) base = atomicAdd(appended, (unsigned long long)__popc(ballot));
  base = __shfl_sync(0xFFFFFFFFu, base, leader);
  if (!keep) return;
  const uint64_t slot = (base - base_total) + (uint64_t)__popc(ballot & ((1u << lane) - 1u));
  if (slot >= dst_cap) {  // cannot happen (cnt * radix <= dst_cap); recorded, never written
    atomicOr(&ctr->error, 1u);
    return;
  }
  store_node(s, dg, dst, dst_cap, (uint32_t)slot);
}

// Lexicographic (makespan, index) minimum of the 16-byte record at *p.  Every
// failed compare-and-swap means another block stored a smaller record, so the
// loop ends; it is bounded all the same and reports if it ever gave up.
__device__ void best_min(BestRecord* p, uint64_t ms, uint64_t idx, TreeCounters* ctr) {
  BestRecord cur = *p;
  for (int it = 0; it < 4096; ++it) {
    if (cur.ms < ms || (cur.ms == ms && cur.idx <= idx)) return;
    const BestRecord want{ms, idx};
    const BestRecord old = atomicCAS(p, cur, want);
    if (old.ms == cur.ms && old.idx == cur.idx) return;
    cur = old;
  }
  atomicOr(&ctr->error, 2u);
}

__device__ __forceinline__ LaneBest shfl_best(const LaneBest& b, int o) {
  LaneBest r;
  r.ms = __shfl_xor_sync(0xFFFFFFFFu, b.ms, o);
  r.dg.now = __shfl_xor_sync(0xFFFFFFFFu, b.dg.now, o);
  r.dg.que = __shfl_xor_sync(0xFFFFFFFFu, b.dg.que, o);
  return r;
}

// Leaf kernel over a window of NW slots (tools [W0, W0 + NW)).
// Block shape of the leaf kernel per window width: 256 threads for narrow
// windows, 128 for wide ones (their registers and per-lane shared state leave
// room for more small blocks than large ones: 20 warps/SM instead of 16 at
// 24 slots; measured 10-20 % faster there).
template <int NW>
struct LeafShape {
  static constexpr int threads = NW >= 16 ? 128 : 256;
  static constexpr int warps = threads / 32;
  static constexpr int min_blocks = NW <= 12 ? 4 : NW <= 16 ? 6 : NW <= 24 ? 5 : 4;
};

template <int NW>
__global__ void __launch_bounds__(LeafShape<NW>::threads, LeafShape<NW>::min_blocks) tree_leaf_kernel(
    const __grid_constant__ TablesW tb, const __grid_constant__ TablesT<NW> tw, const __grid_constant__ TreeConsts tc,
    const uint32_t* __restrict__ src, uint32_t src_cap, uint32_t lo, uint32_t cnt, uint32_t parts, uint32_t chunk,
    uint32_t* bound, BestRecord* best, TreeCounters* ctr) {
  extern __shared__ uint32_t lane_state[];
  __shared__ SmemTablesT<NW> sdw;
  __shared__ uint32_t rtw[ReadyTable<NW>::size];
  __shared__ uint32_t wb_ms[LeafShape<NW>::warps], wb_now[LeafShape<NW>::warps], wb_que[LeafShape<NW>::warps];
  load_smem_tables(tw, sdw);
  fill_ready_table<NW>(tw, rtw);
  __syncthreads();
  const uint32_t lane = threadIdx.x & 31u, warp = threadIdx.x >> 5;
  const uint32_t task = blockIdx.x * LeafShape<NW>::warps + warp;
  const uint32_t groups = (cnt + 31u) / 32u;
  LaneBest lb;
  if (task < groups * parts) {
    const uint32_t g = task / parts, part = task - g * parts;
    const uint32_t j = g * 32u + lane;
    bool valid = j < cnt;
    Digits dg{0u, 0u};
    uint32_t* slot = lane_state + threadIdx.x;
    if (valid) {
      const uint32_t* t = src + lo + j + (size_t)(2 * kTreeSlots) * src_cap;
      dg = Digits{t[9 * (size_t)src_cap], t[10 * (size_t)src_cap]};
      // the incumbent may have improved since this node was bounded
      if (tc.prune &&
          node_lower_bound(src, src_cap, lo + j, tb, tc, dg, tb.all_mask >> tc.D) > (uint64_t)read_bound(bound))
        valid = false;
      else
        node_to_window<NW>(src, src_cap, lo + j, tc.W0, tw.n, slot, LeafShape<NW>::threads);
    }
    const uint32_t ran = __ballot_sync(0xFFFFFFFFu, valid);
    // With a lone last tool, combinations cover the leaf tools but the last
    // one, each standing for radix mappings.
    const uint32_t ncomb = tc.alone_last ? tc.combos / tc.radix : tc.combos;
    const uint32_t c0 = part * chunk;
    const uint32_t c1 = min(c0 + chunk, ncomb);
    if (lane == 0 && ran) {
      if (part == 0) atomicAdd(&ctr->leaf_nodes, (unsigned long long)__popc(ran));
      atomicAdd(&ctr->leaves, (unsigned long long)__popc(ran) * (c1 - c0) * (tc.alone_last ? tc.radix : 1u));
    }
    if (ran) leaf_combos<NW>(tw, sdw, rtw, tc, slot, LeafShape<NW>::threads, dg, valid, c0, c1, lb);
  }
  // warp, then block minimum; one record update per block
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const LaneBest other = shfl_best(lb, o);
    lb.offer(other.ms, other.dg, tc.tie_pow3());
  }
  if (lane == 0) {
    wb_ms[warp] = lb.ms;
    wb_now[warp] = lb.dg.now;
    wb_que[warp] = lb.dg.que;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    LaneBest b;
    for (int w = 0; w < LeafShape<NW>::warps; ++w) b.offer(wb_ms[w], Digits{wb_now[w], wb_que[w]}, tc.tie_pow3());
    if (b.ms != kInfeasible) {
      atomicMin(bound, b.ms);
      best_min(best, b.ms, index_of(b.dg, tc.pow3), ctr);
    }
  }
}

// Digit masks of a canonical index of up to 32 digits.
__device__ __forceinline__ Digits decode64(uint64_t v, uint32_t n) {
  Digits d{0u, 0u};
  for (uint32_t i = 0; i < n; ++i) {
    const uint64_t q = v / 3u;
    const uint32_t r = (uint32_t)(v - 3u * q);
    d.now |= (r == 1u) ? (1u << i) : 0u;
    d.que |= (r == 2u) ? (1u << i) : 0u;
    v = q;
  }
  return d;
}

__global__ void __launch_bounds__(kTreeThreads) wide_list_kernel(const __grid_constant__ TablesW tb, uint64_t total,
                                                                  const uint64_t* __restrict__ idx, uint64_t count,
                                                                  uint32_t* __restrict__ ms_out,
                                                                  uint8_t* __restrict__ fe_out) {
  __shared__ SmemTablesW sd;
  __shared__ uint32_t rt[ReadyTable<kTreeSlots>::size];
  load_smem_tables(tb, sd);
  fill_ready_table<kTreeSlots>(tb, rt);
  __syncthreads();
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t j = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; j < count; j += stride) {
    const uint64_t x = idx[j];
    uint32_t ms = kInfeasible;
    uint8_t fe = 0xFFu;
    if (x < total) {
      const Digits d = decode64(x, tb.n);
      if ((d.que & tb.big_mask) == 0u) {
        State<kTreeSlots> s;
        init_state(s, tb.all_mask);
        if (run<kTreeSlots>(s, tb, sd, rt, d, 0u) == kRunFinished) ms = s.T;
      }
      fe = ms != kInfeasible;
    }
    ms_out[j] = ms;
    fe_out[j] = fe;
  }
}

}  // namespace

size_t tree_node_words() { return (size_t)kNW; }

cudaError_t launch_tree_root(const TablesW& tb, uint32_t* buf, uint32_t cap, cudaStream_t st) {
  tree_root_kernel<<<1, 1, 0, st>>>(tb, buf, cap);
  return cudaGetLastError();
}

cudaError_t launch_tree_expand(const TablesW& tb, const TreeConsts& tc, const uint32_t* src, uint32_t src_cap,
                               uint32_t lo, uint32_t cnt, uint32_t d, uint32_t* dst, uint32_t dst_cap,
                               unsigned long long* appended, unsigned long long base_total, const uint32_t* bound,
                               TreeCounters* ctr, cudaStream_t st) {
  const uint64_t threads = (uint64_t)cnt * tc.radix;
  const unsigned grid = (unsigned)((threads + kTreeThreads - 1) / kTreeThreads);
  tree_expand_kernel<<<grid, kTreeThreads, 0, st>>>(tb, tc, src, src_cap, lo, cnt, d, dst, dst_cap, appended, base_total, bound,
                                                    ctr);
  return cudaGetLastError();
}

template <int NW>
static cudaError_t leaf_launch(const TablesW& tb, const TreeConsts& tc, const uint32_t* src, uint32_t src_cap,
                               uint32_t lo, uint32_t cnt, uint32_t parts, uint32_t chunk, unsigned grid,
                               uint32_t* bound, BestRecord* best, TreeCounters* ctr, cudaStream_t st) {
  static std::atomic<uint64_t> ready{0};
  const size_t smem = sizeof(uint32_t) * LaneWords<NW>::value * LeafShape<NW>::threads;
  const cudaError_t e = allow_dyn_smem(tree_leaf_kernel<NW>, smem, &ready);
  if (e != cudaSuccess) return e;
  TablesT<NW> tw;
  host::build_window(tb, tc.W0, &tw);
  const unsigned blocks = (unsigned)(((uint64_t)grid * kTreeWarps + LeafShape<NW>::warps - 1) / LeafShape<NW>::warps);
  tree_leaf_kernel<NW><<<blocks, LeafShape<NW>::threads, smem, st>>>(tb, tw, tc, src, src_cap, lo, cnt, parts, chunk, bound, best,
                                                         ctr);
  return cudaGetLastError();
}

cudaError_t launch_tree_leaf(const TablesW& tb, const TreeConsts& tc, const uint32_t* src, uint32_t src_cap,
                             uint32_t lo, uint32_t cnt, uint32_t target_tasks, uint32_t* bound, BestRecord* best,
                             TreeCounters* ctr, cudaStream_t st) {
  // Split each group's combinations into parts so that about target_tasks
  // warp tasks exist, each covering at least 16 combinations.
  const uint32_t groups = (cnt + 31u) / 32u;
  const uint32_t ncomb = tc.alone_last ? tc.combos / tc.radix : tc.combos;
  uint32_t parts = (target_tasks + groups - 1u) / groups;
  const uint32_t max_parts = (ncomb + 15u) / 16u;
  if (parts > max_parts) parts = max_parts;
  if (parts < 1u) parts = 1u;
  const uint32_t chunk = (ncomb + parts - 1u) / parts;
  parts = (ncomb + chunk - 1u) / chunk;
  const uint64_t tasks = (uint64_t)groups * parts;
  const unsigned grid = (unsigned)((tasks + kTreeWarps - 1) / kTreeWarps);
  const uint32_t nw = tb.n - tc.W0;
#define BF_TRY(NW)                                                                                           \
  if (nw <= (uint32_t)NW)                                                                                    \
    return leaf_launch<NW>(tb, tc, src, src_cap, lo, cnt, parts, chunk, grid, bound, best, ctr, st);
  BF_TREE_BUCKETS(BF_TRY)
#undef BF_TRY
  return cudaErrorInvalidValue;
}

cudaError_t launch_wide_list(const TablesW& tb, uint64_t total, const uint64_t* idx, uint64_t count, uint32_t* ms,
                             uint8_t* fe, int grid, cudaStream_t st) {
  wide_list_kernel<<<grid, kTreeThreads, 0, st>>>(tb, total, idx, count, ms, fe);
  return cudaGetLastError();
}

}  // namespace bfk
