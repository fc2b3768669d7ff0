/*
 * bf.h -- C ABI of the brute-force optimal device-mapping search (libbf.so).
 *
 * The problem (§2.1 of "Agentic CPU-GPU Scheduling for Heterogeneous AI
 * Workloads"): a workflow is a DAG G=(V,E) of N tool invocations; each tool v
 * is mapped to a mode a_v in {cpu, gpu_now, gpu_queue}; a mapping is feasible
 * only if the VRAM of the GPU tools running at any instant stays within the
 * budget M; its end-to-end latency T_e2e is the largest completion time over
 * the sinks.  The brute-force oracle the paper grades its scheduler against
 * (§2.3, §4.1) is the feasible mapping of lowest T_e2e among all 3^N.
 *
 * The paper measures T_e2e on hardware.  This library evaluates it under a
 * fixed integer latency model (version 1), exact to the microsecond:
 *
 *   - Times are integer microseconds.  GPU progress is a virtual clock V in
 *     1/1024 isolated-microsecond units; a GPU tool of isolated time w that
 *     starts at V ends when V reaches V + 1024*w.
 *   - GPU contention (Factor A, §2.3): while k GPU tools run, each runs at
 *     1024/f[k] of its isolated speed (processor sharing).  CPU tools are
 *     unaffected; CPU cores are unlimited.
 *   - cpu: duration c.  gpu_now: isolated work g + x (Table 1's GPU time
 *     includes PCIe transfer), starts when its predecessors are done, holds
 *     its VRAM m while running; a start that brings live VRAM above M makes
 *     the mapping infeasible (out of memory, Factor B).  gpu_queue: waits in
 *     one serialised FIFO queue (ready time, then index) without holding VRAM;
 *     the head starts when no queued tool is running and live VRAM + m <= M;
 *     isolated work l + g + x (Table 1's gpu_queue column = GPU + Load).  A
 *     queued tool with m > M can never start: infeasible.  No bypass.
 *   - Event loop: next CPU completion vs next GPU completion
 *     T + ceil((Vmin - V) * f[k] / 2^20); if a CPU tool ends first, V advances
 *     by floor((t_cpu - T) * 2^20 / f[k]).  At each event every tool ending at
 *     that instant retires (freeing VRAM), then newly ready tools start in
 *     index order, then the queue head is tried.  Makespan = time of the last
 *     retirement; infeasible mappings have makespan 0xFFFFFFFF.
 *
 * Mapping index: idx = sum_i a_i * 3^i, a_i in {0=cpu, 1=gpu_now,
 * 2=gpu_queue}; tool 0 is the least-significant digit.  Searches return the
 * feasible mapping of lowest makespan, ties to the lowest index.  The all-cpu
 * mapping (index 0) is always feasible, so a full search always succeeds.
 *
 * Conventions for every entry point:
 *   - Return 0 (BF_OK) or a BF_E* status; bf_last_error() then describes the
 *     failure (thread-local string owned by the library, valid until the next
 *     call on that thread).  Outputs are written only on BF_OK.
 *   - Host pointers are caller-owned and only read during the call (inputs are
 *     copied).  Device pointers are caller-owned CUDA device memory on the
 *     current device.  `cuda_stream` is a cudaStream_t (NULL = legacy default
 *     stream); work is ordered on it.
 *   - A handle's scratch (search key, what-if list) is shared by the calls that
 *     use it: calls on one handle must not overlap in time.  A handle belongs
 *     to the device that was current when it was created; calls on it with
 *     another device current return BF_EINVAL.
 *   - Blocking calls wait with a time limit (bf_set_wait_timeout_ms) and
 *     return BF_ETIMEOUT if it passes; the GPU work is then still in flight,
 *     and the scenario must not be destroyed until the stream has finished.
 */
#ifndef BF_H_
#define BF_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Entry points are the library's only exported symbols (it is built with
 * hidden visibility). */
#if defined(__GNUC__)
#define BF_API __attribute__((visibility("default")))
#else
#define BF_API
#endif

#define BF_MAX_TOOLS 32       /* largest scenario (32-bit tool masks) */
#define BF_MAX_TOOLS_ENUM 20  /* largest scenario of the full-enumeration entry points
                                 (bf_eval_mappings, bf_search_best, bf_search_range,
                                 bf_search_pruned, bf_search_batch*): 3^20 < 2^32 */

enum bf_status {
  BF_OK = 0,
  BF_EINVAL = 1,    /* invalid argument or scenario */
  BF_ERANGE = 2,    /* index range outside [0, 3^n) */
  BF_ENOMEM = 3,    /* device or pinned-host allocation failed */
  BF_ECUDA = 4,     /* a CUDA runtime call failed (message names it) */
  BF_ETIMEOUT = 5   /* a blocking wait exceeded its time limit */
};

enum bf_mode { BF_MODE_CPU = 0, BF_MODE_GPU_NOW = 1, BF_MODE_GPU_QUEUE = 2 };

/*
 * One workflow (§2.1) with the per-tool profile of Table 1 / §3.1 plus a
 * transfer time.  Tools are numbered 0..n-1 in a topological order.
 * Validity (checked by every entry point that takes a desc):
 *   1 <= n <= 32 (the full-enumeration entry points take n <= 20 and return
 *   BF_EINVAL above); pred_mask[v] has bits only below v (u < v);
 *   cpu_us >= 1, gpu_us >= 1; load_us + gpu_us + xfer_us < 2^22;
 *   vram_mib <= 2^27, vram_budget_mib <= 2^31;
 *   slowdown_q10[1] == 1024, slowdown_q10[k] non-decreasing and <= 65536 for
 *   k = 1..n (entries 0 and > n are ignored);
 *   the makespan bound sum_i max(c_i, floor((l_i+g_i+x_i)*f[n]/1024) + n + 1)
 *   is <= 0xFFFFFFFD, so every makespan fits in 32 bits.
 * Entries at index >= n are ignored.
 */
typedef struct bf_scenario_desc {
  uint32_t n;                               /* number of tools, 1..32 */
  uint32_t pred_mask[BF_MAX_TOOLS];         /* bit u of pred_mask[v] <=> edge u->v */
  uint32_t cpu_us[BF_MAX_TOOLS];            /* c_i: CPU latency, us */
  uint32_t gpu_us[BF_MAX_TOOLS];            /* g_i: isolated GPU latency, us */
  uint32_t xfer_us[BF_MAX_TOOLS];           /* x_i: host<->device transfer, us (GPU modes only) */
  uint32_t load_us[BF_MAX_TOOLS];           /* l_i: gpu_queue load-in, us */
  uint32_t vram_mib[BF_MAX_TOOLS];          /* m_i: VRAM footprint, MiB */
  uint32_t vram_budget_mib;                 /* M */
  uint32_t slowdown_q10[BF_MAX_TOOLS + 1];  /* f[k], k=1..n, 1024 = isolated speed */
} bf_scenario_desc;

/* Result of a search: the argmin mapping and its makespan. */
typedef struct bf_result {
  uint64_t index;                  /* canonical mapping index */
  uint32_t makespan_us;            /* 0xFFFFFFFF if feasible == 0 */
  uint32_t feasible;               /* 1 if a feasible mapping was found in the searched range */
  uint8_t mode[BF_MAX_TOOLS];      /* decoded digits of `index` (bf_mode), 0 beyond n */
} bf_result;

/* Opaque handle: validated scenario, its device-format tables and a small
 * device/pinned scratch area.  Owned by the library. */
typedef struct bf_scenario bf_scenario;

/* Validate a desc without touching the GPU.  BF_OK or BF_EINVAL. */
BF_API int bf_validate_desc(const bf_scenario_desc* desc);

/* The problem instance of §2.1 -- the tool DAG G=(V,E), each tool's profile
 * (Table 1 / §3.1: CPU and GPU latency, load-in, VRAM) plus its transfer time,
 * the VRAM budget M -- with the contention table of §2.3 Factor A.
 * Validate `desc`, copy it, allocate the handle's scratch (8-byte device key,
 * 8-byte pinned host key) on the current device and return it in *out.
 * The caller releases it with bf_destroy_scenario.  BF_EINVAL, BF_ENOMEM,
 * BF_ECUDA. */
BF_API int bf_create_scenario(const bf_scenario_desc* desc, bf_scenario** out);

/* Release a handle (NULL is accepted).  Synchronises with nothing: the caller
 * must make sure no work using it is still in flight. */
BF_API int bf_destroy_scenario(bf_scenario* scn);

/* Evaluate mappings [first, first+count) (§2.1's T_e2e under the model):
 * d_makespan[j] = makespan of mapping first+j (0xFFFFFFFF if infeasible),
 * d_feasible[j] = 1/0.  Both are caller-owned device arrays of >= count
 * elements.  Asynchronous on `cuda_stream`.  count == 0 is a no-op.
 * BF_ERANGE if first+count > 3^n; BF_EINVAL on NULL pointers. */
BF_API int bf_eval_mappings(const bf_scenario* scn, uint64_t first, uint64_t count,
                     uint32_t* d_makespan, uint8_t* d_feasible, void* cuda_stream);

/* Brute-force oracle of §2.3/§4.1 under the model: the feasible mapping of
 * lowest makespan over all 3^n, ties to the lowest index.  Blocks until the
 * result is on the host (bounded wait).  Writes *out on BF_OK. */
BF_API int bf_search_best(const bf_scenario* scn, bf_result* out, void* cuda_stream);

/* As bf_search_best over mappings [first, first+count) only; out->feasible is
 * 0 (and index = first) when no mapping in the range is feasible.  Range
 * searches compose: the best of the parts' results (lowest makespan, then
 * lowest index) is the result of their union -- used to split one search
 * across devices or to resume it piecewise.  BF_ERANGE if outside [0, 3^n);
 * count == 0 gives feasible = 0. */
BF_API int bf_search_range(const bf_scenario* scn, uint64_t first, uint64_t count,
                    bf_result* out, void* cuda_stream);

/* Full search of `count` independent scenarios in one call (one launch per
 * group of scenarios of similar size, four at most): out[i] is the
 * brute-force oracle of §2.3/§4.1 (as bf_search_best) for descs[i].  The paper
 * searches one workflow at a time; running many per launch is this library's
 * addition, for callers that score many workflows or many candidate
 * contention tables (the calibration of Table 2's S5 latencies) together.  All descs are validated
 * before any GPU work; the first invalid one (lowest position) fails the call with BF_EINVAL naming
 * its position.  Allocates its device scratch (packed tables + one key per scenario) from the
 * device's default stream-ordered memory pool on cuda_stream and frees it there after its kernels,
 * also when the wait times out (BF_ETIMEOUT).  A large batch launches part of its work on a stream
 * the call creates and destroys; that work starts after the work already enqueued on cuda_stream,
 * and work enqueued on cuda_stream after the call starts after it.  Blocks until the results are
 * on the host. */
BF_API int bf_search_batch(const bf_scenario_desc* descs, uint32_t count, bf_result* out,
                    void* cuda_stream);

/* Same result as bf_search_best (the feasible mapping of lowest makespan over
 * all 3^n, ties to the lowest index), found by branch and bound instead of
 * full enumeration.  An incumbent is taken from a few mappings (hint_index if
 * < 3^n, all-cpu, all-gpu_now, all-gpu_queue, each tool on its isolated-faster
 * device); a prefix (or a mid combination) is skipped when the time at which
 * its remaining tools can first start, plus the longest path through them in
 * minimum isolated durations min(c, g + x), exceeds the incumbent's makespan
 * -- no mode, contention or queueing makes a tool faster than that.  When
 * that first pass keeps more than 1/64 of the prefixes (a DAG without cut
 * points), the call continues as bf_search_tree over the full space, whose
 * bound is stronger.  Exact either way: the optimum and all its ties are
 * never skipped.  Allocates a 4-byte-per-prefix buffer (and, when it hands
 * over, the tree search's level buffers) in the handle on first use.  Blocks
 * until the result is on the host. */
BF_API int bf_search_pruned(const bf_scenario* scn, uint64_t hint_index, bf_result* out, void* cuda_stream);

/* Decision spaces of bf_search_tree: the full space (each tool on cpu,
 * gpu_now or gpu_queue; 3^n mappings) or the binary space the paper's S1-S10
 * use (§4.1: each tool on the CPU or the GPU, i.e. cpu or gpu_now; 2^n
 * mappings).  The value is the number of modes per tool. */
#define BF_SPACE_BINARY 2u
#define BF_SPACE_FULL 3u
/* bf_search_tree flag: simulate every mapping of the space (no pruning). */
#define BF_TREE_NO_PRUNE 1u

/* What a tree search did (bf_search_tree, optional). */
typedef struct bf_tree_stats {
  uint64_t nodes;         /* prefix nodes created (tools assigned in the search's order), root included */
  uint64_t leaf_nodes;    /* nodes whose last leaf_depth tools were enumerated */
  uint64_t leaves;        /* mappings simulated to the end (at most leaf_nodes * modes^leaf_depth) */
  uint32_t launches;      /* kernel launches */
  uint32_t leaf_depth;    /* tools enumerated below each leaf node */
  uint32_t incumbent_us;  /* the starting bound (0xFFFFFFFF with BF_TREE_NO_PRUNE) */
  uint32_t pad;
} bf_tree_stats;

/* The optimum of a decision space -- the feasible mapping of lowest makespan,
 * ties to the lowest canonical index, exactly as full enumeration would give
 * it -- for scenarios of up to 32 tools (3^32 ~ 1.9e15 mappings), by depth-
 * first branch and bound over the modes of the tools in a topological order:
 * the sources (tools without predecessors) first, then the others, each group
 * in index order (the model's results do not depend on that order; the index
 * returned is the canonical one).  A node (the modes of the first d tools of
 * that order) carries the simulation state at the first instant a later tool
 * could become ready, shared by all its mappings.
 * A node is dropped when a lower bound on all of its mappings' makespans
 * exceeds the best makespan known (strictly, so the optimum and its ties
 * survive): running tools end no earlier than their remaining work at
 * isolated speed allows, every other tool ends no earlier than the latest of
 * the node's time and its predecessors' earliest ends plus its duration in
 * its mode (or min(c, g + x) if open), and queued tools run one at a time.
 * The first bound is the best of a few mappings of the space (hint_index if
 * it lies in it, all-cpu, all-gpu_now, each tool on its isolated-faster
 * device, all-gpu_queue); when the tree is large, a narrow dive to the leaves
 * (8192 nodes per level) tightens it before the search restarts from the root;
 * better bounds are found as the search proceeds.  space: BF_SPACE_FULL or
 * BF_SPACE_BINARY.
 * flags: 0 or BF_TREE_NO_PRUNE (every mapping of the space is simulated:
 * full enumeration).  `stats` may be NULL.  Allocates level buffers in the
 * handle on first use (about 1.7 GB for 32 tools in the full space).  Blocks
 * until the result is on the host.  The whole search, not only each level
 * step, is held to the wait limit (bf_set_wait_timeout_ms): past it the call
 * returns BF_ETIMEOUT (an unpruned full space of 28 or more tools takes
 * hours). */
BF_API int bf_search_tree(const bf_scenario* scn, uint32_t space, uint32_t flags, uint64_t hint_index,
                   bf_result* out, bf_tree_stats* stats, void* cuda_stream);

/* Makespans and feasibility of an arbitrary list of mappings: d_makespan[j] and
 * d_feasible[j] for mapping d_indices[j] (all three caller-owned device arrays
 * of >= count elements).  An index >= 3^n yields makespan 0xFFFFFFFF and
 * d_feasible = 0xFF.  Asynchronous on `cuda_stream`; count == 0 is a no-op.
 * Used to score neighbourhoods of a mapping (bf_whatif) or any caller-chosen
 * candidate set. */
BF_API int bf_eval_indices(const bf_scenario* scn, const uint64_t* d_indices, uint64_t count,
                    uint32_t* d_makespan, uint8_t* d_feasible, void* cuda_stream);

/* One probe of the runtime monitor's bounded what-if exploration. */
typedef struct bf_probe {
  uint64_t index;        /* canonical index of the probed mapping */
  uint32_t makespan_us;  /* 0xFFFFFFFF if infeasible */
  uint32_t feasible;     /* 0 = exceeds the VRAM budget ("exceed") */
  uint8_t kind;          /* 0 = single-tool reprobe, 1 = swap reprobe */
  uint8_t tool;          /* i: the tool moved (swap: the tool moved to gpu_now) */
  uint8_t mode;          /* the new mode of tool i (bf_mode) */
  uint8_t other;         /* swap: j, the gpu_now tool moved to gpu_queue; single: 0xFF */
} bf_probe;

#define BF_MAX_PROBES (2 * BF_MAX_TOOLS + BF_MAX_TOOLS * BF_MAX_TOOLS)

/* The what-if probes of Algorithm 1's exploration step (§3.2) around mapping
 * base_index, scored on the model in one launch: for each tool i in index
 * order and each alternative mode a != d_i (in the order cpu, gpu_now,
 * gpu_queue), the single-tool reprobe d[i := a]; when that reprobe moves i to
 * gpu_now and exceeds the budget (infeasible), then for each tool j on
 * gpu_now in d (index order) the swap reprobe d[i := gpu_now, j := gpu_queue].
 * Writes the probes in that order to out[0 .. *count) (at most
 * BF_MAX_PROBES); BF_EINVAL if capacity is smaller than the number of probes,
 * BF_ERANGE if base_index >= 3^n.  Blocks until the results are on the host. */
BF_API int bf_whatif(const bf_scenario* scn, uint64_t base_index, bf_probe* out, uint32_t capacity,
              uint32_t* count, void* cuda_stream);

/* Largest batch bf_search_batch_noalloc accepts. */
#define BF_NOALLOC_MAX_SCENARIOS 1024

/* The batched search of bf_search_batch without any memory allocation.  The
 * paper has no counterpart: this exists for callers that cannot allocate
 * device memory at the moment they search -- e.g. a scheduler loop whose
 * process has handed all GPU memory to another allocator's pool, or one that
 * must not let cudaMalloc/cudaFree synchronise the device between rounds.
 * The caller passes the inputs (descs) and outputs (out) as for
 * bf_search_batch; the scratch (packed scenario records and one key per
 * scenario, about 0.84 MiB for BF_NOALLOC_MAX_SCENARIOS) is a fixed array in
 * the library's device image, held on every GPU that loads the library until
 * the process exits.  count > BF_NOALLOC_MAX_SCENARIOS fails with BF_EINVAL.
 * The first call on a device (and the first after a device reset) resolves
 * that array's device address; make it before any stream capture.
 * All calls share the one array, which keeps the last call's contents (each
 * call resets its keys), so two calls whose GPU work overlapped would race.
 * The library prevents that: calls on one device are serialised by a host
 * lock, and after a call returns BF_ETIMEOUT its kernel may still be using
 * the array, so the next call first waits (bounded) for that call's stream to
 * finish and returns BF_ETIMEOUT if it does not; keep that stream alive until
 * then.  Blocks until the results are on the host. */
BF_API int bf_search_batch_noalloc(const bf_scenario_desc* descs, uint32_t count, bf_result* out,
                            void* cuda_stream);

/* Time limit of blocking waits, in milliseconds (default 600000; 0 = none).
 * Process-wide. */
BF_API void bf_set_wait_timeout_ms(uint32_t ms);

/* Description of the last failure on this thread ("" if none). */
BF_API const char* bf_last_error(void);

/* Library version string, e.g. "bf 1.0 (model v1)". */
BF_API const char* bf_version(void);

#ifdef __cplusplus
}
#endif

#endif /* BF_H_ */
