#!/usr/bin/env python3
"""Benchmark: brute-force optimal device-mapping search on GB300.

One step = one full search of the N=19 workload (scenarios.config3(): a spine
plus two fan-outs, tools from all four scheduling zones of §2.2, 32 GiB VRAM
budget, contention f[k] = 1 + 0.35(k-1)): all 3^19 = 1,162,261,467 mappings
enumerated, simulated and reduced to the argmin in one bf_search_best call.

Prints ONE JSON line (rank 0).  Metric: mappings evaluated per second (whole
job).  Also reported: the per-step wall time to the optimum, the kernel's
integer-issue roofline, the oracle timed on the host cores on a bounded sample
(cpu_baseline), and the end-to-end rate through the host-buffer API (create
scenario from host tables, search, result back on the host, release).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl bf|reference]

With --impl reference the CPU oracle is timed instead (rank 0 only), on
bounded samples of the same workload.  Under torchrun (N > 1) one step is
still one search of all 3^19 mappings, split into N contiguous index ranges
(bf_search_range on each rank's GPU) and reduced by one all-gather of an
8-byte key per rank; the step time is the max over ranks and `value` counts
the 3^19 mappings once (strong scaling).
"""
from __future__ import annotations

import argparse
import ctypes
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "mappings evaluated/sec on 1 GB300; wall time to optimum at N=19; % of issue peak"
UNIT = "mappings/s"
WORKLOAD = ("config3: N=19 tools (spine of 7 + two fan-outs of 6; 11 GPU-preferred, 4 ambiguous, "
            "1 CPU-preferred, 3 neutral), 32 GiB VRAM budget, f[k]=1+0.35(k-1), seed 3; full 3^19 search")
# Algorithmic integer operations per simulated mapping: N events, each with an
# N-wide next-completion scan and an N-wide readiness scan (2 N^2).
N_TOOLS = 19
OPS_PER_MAPPING = 2 * N_TOOLS * N_TOOLS
INT_LANES_PER_SM = 128  # 4 SMSPs x 32 lanes: one thread instruction each per clock at full issue

# Committed ncu summaries of the enumerating kernels, one per standard workload.
PROFILES = {"config0": "search_kernel_config0_n8.md", "config1": "search_kernel_config1_n12.md",
            "config2": "lanetree_single_kernel_config2_n16.md", "config3": "search_kernel_config3_n19.md",
            "config4_batch": "lanetree_kernel_config4.md"}
# Translation unit each summary's fingerprint covers (_build.kernel_fingerprint): the full search of
# the 16-tool workload and the batch run the lane-tree kernels.
PROFILE_UNITS = {"config2": "LANETREE_UNIT", "config4_batch": "LANETREE_UNIT"}
PROFILE_KEYS = ("source_fingerprint", "dram_bytes_per_launch", "thread_instructions_per_mapping", "issue_active",
                "warp_efficiency", "kernel_ms")


def profiled_fields(workload: str = "config3"):
    """Fields of the committed ncu summary of `workload`'s kernel (DRAM bytes per launch, executed
    thread instructions per mapping, issue-slot utilisation, warp execution efficiency), or {} when
    the summary is missing or the enumerating kernels' translation unit changed since that capture."""
    from paper_2607_22242_gb300 import _build
    try:
        text = open(os.path.join(ROOT, "profiles", PROFILES[workload])).read()
    except OSError:
        return {}
    fields = dict(line.split(": ", 1) for line in text.splitlines()
                  if line.startswith(tuple(k + ": " for k in PROFILE_KEYS)))
    unit = getattr(_build, PROFILE_UNITS.get(workload, "KERNEL_UNIT"))
    if fields.get("source_fingerprint", "").strip() != _build.kernel_fingerprint(unit=unit):
        return {}
    return {k: v.strip() for k, v in fields.items()}


def issue_roofline(fields, mappings_per_s: float, peak_ops: float):
    """The instruction-issue roofline of one workload: executed thread instructions per mapping (ncu) x
    mappings/s against SMs x 128 lanes x clock, with the ncu issue-slot share and warp efficiency."""
    if "thread_instructions_per_mapping" not in fields:
        return {}
    inst = float(fields["thread_instructions_per_mapping"])
    out = {"thread_instructions_per_mapping": inst, "issue_frac": inst * mappings_per_s / peak_ops}
    for key, name in (("issue_active", "issue_active_frac"), ("warp_efficiency", "warp_efficiency")):
        if key in fields:
            out[name] = float(fields[key])
    return out


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", str(rank)))
    return rank, world, local


def emit(obj):
    print(json.dumps(obj), flush=True)


# --------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi samples every 200 ms while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_id: str):
        self.device_id = device_id
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200",
                 "-i", self.device_id], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            time.sleep(0.3)
        except (OSError, ValueError):
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.thread.join(timeout=2)

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def device_id_for_smi(torch, dev: int) -> str:
    try:
        return "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        return str(dev)


# --------------------------------------------------------------------------- CPU oracle timing

def oracle_sample_time(scn, budget_mappings: int, threads: int):
    """Time the oracle on `budget_mappings` indices in 16 evenly spaced contiguous chunks."""
    import oracle
    total = 3 ** scn.n
    chunks = 16
    per = budget_mappings // chunks
    t0 = time.perf_counter()
    for c in range(chunks):
        oracle.search_range(scn, (total // chunks) * c, per, threads)
    dt = time.perf_counter() - t0
    return per * chunks, dt


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    import oracle
    from paper_2607_22242_gb300 import scenarios as S
    oracle.build()
    scn = S.config3()
    threads = oracle.default_threads()
    per_step = args.ref_sample
    for _ in range(args.warmup):
        oracle_sample_time(scn, per_step, threads)
    times = []
    for _ in range(args.steps):
        n, dt = oracle_sample_time(scn, per_step, threads)
        times.append(dt)
    ms = 1e3 * statistics.mean(times)
    value = per_step / (ms / 1e3)
    sample = (f"{per_step} mappings per step: 16 contiguous chunks spread evenly over [0, 3^19), "
              f"oracle search over {threads} host threads")
    emit({"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
          "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
          "scaling": "weak", "vs_baseline": None, "dtype": "u64", "data": "synthetic",
          "config": {"workload": WORKLOAD, "mappings_per_step": per_step},
          "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "cpu_model": cpu_model(), "kind": "oracle", "sample": sample},
          "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}})
    return 0


# --------------------------------------------------------------------------- GPU arm

def tree_search_times(torch, bf, S, stream, reps: int = 3):
    """bf_search_tree on the 28- and 32-tool workloads: CUDA-event time of the call to the exact optimum
    (median of `reps` after one warm-up), each result checked against the oracle's stored optimum."""
    with open(os.path.join(ROOT, "tests", "golden", "wide_results.json")) as fh:
        golden = json.load(fh)["workloads"]
    cases = (("wide32", bf.SPACE_FULL, True), ("wide28", bf.SPACE_FULL, True), ("wide32", bf.SPACE_BINARY, True),
             ("wide28", bf.SPACE_BINARY, False))
    out = {}
    for name, space, prune in cases:
        scn = getattr(S, name)()
        want = tuple(golden[name]["ternary" if space == bf.SPACE_FULL else "binary"])
        times, stats = [], {}
        with bf.create_scenario(scn) as h:
            for rep in range(reps + 1):
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(stream)
                r, stats = bf.search_tree(h, space, prune, None, stream)
                b.record(stream)
                b.synchronize()
                assert (r.index, r.makespan_us) == want, (name, space, prune, r, want)
                if rep:
                    times.append(a.elapsed_time(b))
        ms = statistics.median(times)
        key = f"{name}_{'full' if space == bf.SPACE_FULL else 'binary'}{'' if prune else '_unpruned'}"
        out[key] = {"ms": ms, "mappings_in_space": space ** scn.n, "leaves_simulated": stats["leaves"],
                    "nodes": stats["nodes"], "leaves_per_s": stats["leaves"] / (ms / 1e3)}
    out["note"] = ("bf_search_tree: exact optimum (lowest makespan, lowest index) by branch and bound; "
                   "'unpruned' simulates every mapping of the space")
    return out


def per_config_times(torch, bf, S, stream, reps: int = 5):
    """Exhaustive search of each standard workload (the 4096-scenario batch as one call): median CUDA-event
    time of the call and mappings/s, each optimum checked against the oracle's stored results."""
    with open(os.path.join(ROOT, "tests", "golden", "config_results.json")) as fh:
        golden = json.load(fh)["configs"]
    out = {}
    for cfg in range(4):
        scn = S.config(cfg)
        summ = golden[str(cfg)]["summary"]
        times = []
        with bf.create_scenario(scn) as h:
            for rep in range(reps + 1):
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(stream)
                r = bf.search_best(h, stream)
                b.record(stream)
                b.synchronize()
                assert (r.index, r.makespan_us) == (summ["best_index"], summ["best_makespan"]), (cfg, r)
                if rep:
                    times.append(a.elapsed_time(b))
        ms = statistics.median(times)
        out[f"config{cfg}"] = {"ms": ms, "mappings": 3 ** scn.n, "mappings_per_s": 3 ** scn.n / (ms / 1e3)}
    import ctypes
    batch = S.config4()
    packed = bf.pack_descs(batch)  # the C caller's array of bf_scenario_desc
    descs = packed.ctypes.data_as(ctypes.POINTER(bf.Desc))
    results = (bf.CResult * len(batch))()
    want = list(zip(golden["4"]["best_index"], golden["4"]["best_makespan"]))
    times = []
    for rep in range(4):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        rc = bf.load().bf_search_batch(descs, len(batch), results, ctypes.c_void_p(stream.cuda_stream))
        b.record(stream)
        b.synchronize()
        assert rc == bf.BF_OK, bf.last_error()
        assert [(r.index, r.makespan_us) for r in results] == want
        if rep:
            times.append(a.elapsed_time(b))
    ms = statistics.median(times)
    total = len(batch) * 3 ** 10
    out["config4_batch"] = {"ms": ms, "mappings": total, "mappings_per_s": total / (ms / 1e3),
                            "note": "one bf_search_batch C call on an array of 4096 descs: per-scenario "
                                    "tables and plans on the host, allocation, copies and the kernel"}
    return out


def cpu_model() -> str:
    """Host CPU model name (lscpu, else /proc/cpuinfo, else the machine type)."""
    import platform
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as fh:
            for line in fh:
                if line.startswith("model name"):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    return platform.machine()


def oracle_single_core(S, seconds_per_config: float = 1.5):
    """The oracle on one host thread: mappings/s per standard workload on a timed slice of its index space."""
    import oracle
    out = {}
    for cfg in range(4):
        scn = S.config(cfg)
        total = 3 ** scn.n
        count = min(total, 1 << 14)
        n_done, t0 = 0, time.perf_counter()
        while time.perf_counter() - t0 < seconds_per_config and n_done < total:
            first = (n_done * 7919) % max(1, total - count)
            oracle.search_range(scn, first, count, 1)
            n_done += count
        dt = time.perf_counter() - t0
        out[f"config{cfg}"] = n_done / dt
    return out


def sharded_step(search_range, total: int):
    """The multi-GPU step: this rank searches its contiguous share of [0, total) with
    ``search_range(first, count) -> (index, makespan, feasible)``, then one all-gather of one 8-byte key
    per rank gives the optimum (index, makespan) of the whole space on every rank."""
    from paper_2607_22242_gb300 import shard
    idx, ms, _ = shard.sharded_search(search_range, total)
    return idx, ms


def run_gpu(args):
    import torch
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    dev = torch.cuda.current_device()

    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_22242_gb300 import bf
    from paper_2607_22242_gb300 import scenarios as S
    from paper_2607_22242_gb300 import shard

    scn = S.config3()
    total = 3 ** scn.n
    with open(os.path.join(ROOT, "tests", "golden", "config_results.json")) as fh:
        summ = json.load(fh)["configs"]["3"]["summary"]
    want = (summ["best_index"], summ["best_makespan"])
    stream = torch.cuda.current_stream()
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.int32, device="cuda")  # > 129 MB L2

    def search_step(handle):
        """One search of all 3^19 mappings: on one GPU the whole space (bf_search_best); on N ranks
        each searches its contiguous index range (bf_search_range) and one all-gather of 8-byte keys
        gives every rank the optimum."""
        if world == 1:
            r = bf.search_best(handle, stream)
            return r.index, r.makespan_us
        return sharded_step(shard.gpu_search_range(handle, stream), total)

    def barrier():
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()

    h = bf.create_scenario(scn)
    for _ in range(args.warmup):
        res = search_step(h)
    assert res == want, (res, want)

    # ---- timed region: K full searches, L2 flushed between them -------------
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    sampler = ClockSampler(device_id_for_smi(torch, dev))
    results = []
    with sampler:
        barrier()
        wall0 = time.perf_counter()
        for i in range(args.steps):
            flush.zero_()
            starts[i].record(stream)
            results.append(search_step(h))
            ends[i].record(stream)
        barrier()
        wall = time.perf_counter() - wall0
    assert all(r == want for r in results), results
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    mean_ms = statistics.mean(step_ms)
    worst_ms = shard.max_over_ranks(mean_ms) if world > 1 else mean_ms
    value = total / (worst_ms / 1e3)  # the 3^19 mappings of one search, counted once
    clocks = sampler.summary()

    # ---- end to end through the host-buffer API ------------------------------
    e2e_times = []
    barrier()
    for _ in range(max(3, args.steps // 4)):
        t0 = time.perf_counter()
        with bf.create_scenario(scn) as h2:       # host tables in, validated, scratch allocated
            r2 = search_step(h2)                   # tables travel with the launch; 8-byte key back
        e2e_times.append(time.perf_counter() - t0)
        assert r2 == want
    e2e_mean = statistics.mean(e2e_times)
    if world > 1:
        e2e_mean = shard.max_over_ranks(e2e_mean)
    e2e_value = total / e2e_mean

    extras = {}
    if world == 1:
        # ---- the same optimum by branch and bound (reported beside, not as `value`) ---
        pruned_ms = []
        for _ in range(max(3, args.steps // 4)):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            rp = bf.search_pruned(h, None, stream)
            b.record(stream)
            b.synchronize()
            pruned_ms.append(a.elapsed_time(b))
            assert (rp.index, rp.makespan_us) == want
        # ---- host wall time of the blocking call, scenario already created ----------
        host_ms = []
        for _ in range(10):
            t0 = time.perf_counter()
            bf.search_best(h, stream)
            host_ms.append((time.perf_counter() - t0) * 1e3)
        extras = {"pruned_ms": pruned_ms, "host_ms": host_ms,
                  # ---- every standard workload, and beyond 20 tools the tree search ---------
                  "per_config": per_config_times(torch, bf, S, stream),
                  "tree": tree_search_times(torch, bf, S, stream),
                  "modes": bf.search_best(h, stream).modes}
    h.close()

    if rank != 0:
        torch.distributed.destroy_process_group()
        return 0

    sm_count = torch.cuda.get_device_properties(dev).multi_processor_count
    clk_mhz = clocks["sm_mhz"] or 2070.0
    peak_ops = sm_count * INT_LANES_PER_SM * clk_mhz * 1e6
    per_gpu = value / world  # mappings/s of one GPU's kernel
    prof = profiled_fields("config3")
    issue = issue_roofline(prof, per_gpu, peak_ops)
    roofline = {"bound": "alu",
                "achieved": issue["thread_instructions_per_mapping"] * per_gpu / 1e12 if issue else None,
                "peak": peak_ops / 1e12, "unit": "T thread-instructions/s",
                "frac": issue.get("issue_frac"),
                "traffic": int(prof["dram_bytes_per_launch"]) if "dram_bytes_per_launch" in prof else None,
                "peak_basis": f"{sm_count} SMs x {INT_LANES_PER_SM} lanes (4 SMSPs x 32) x "
                              f"{clk_mhz:.0f} MHz ({'sampled median under load' if clocks['sm_mhz'] else 'max clock, no samples'}); "
                              "derived from unit counts and the sampled clock (no integer peak is measured)",
                "executed_thread_instructions_per_mapping": issue.get("thread_instructions_per_mapping"),
                "issue_active_frac": issue.get("issue_active_frac"),
                "warp_efficiency": issue.get("warp_efficiency"),
                "algorithmic_ops_per_mapping": OPS_PER_MAPPING,
                "algorithmic_frac": OPS_PER_MAPPING * per_gpu / peak_ops,
                "note": ("frac = executed thread instructions per mapping (ncu, committed summary whose kernel "
                         "fingerprint matches the built kernels; null when stale) x mappings/s / peak; "
                         "algorithmic_frac counts 2 N^2 integer ops per mapping (a from-scratch simulation), "
                         "which the checkpointed enumeration does not execute")}

    out = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": worst_ms, "higher_is_better": True,
           "scaling": "strong" if world > 1 else "weak",
           "vs_baseline": None, "dtype": "u32", "data": "synthetic",
           "config": {"workload": WORKLOAD, "mappings_per_step": total,
                      "parallelism": f"index-range shards x{world}" if world > 1 else "single GPU",
                      "l2": "flushed between steps (256 MiB write, outside the timed events)"},
           "wall_time_to_optimum_ms": {"median": statistics.median(step_ms), "min": min(step_ms),
                                       "max": max(step_ms)},
           "result": {"index": want[0], "makespan_us": want[1], "checked": "equals the oracle's stored optimum"},
           "roofline": roofline,
           "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": ctypes.sizeof(bf.Desc),
                   "d2h_bytes_per_step": 8,
                   "path": "bf_create_scenario(host desc) + " + ("bf_search_best" if world == 1 else
                           "bf_search_range on each rank's index range + all-gather of 8-byte keys") +
                           " + bf_destroy_scenario",
                   "bytes_note": "in: the step's input, one bf_scenario_desc per GPU (its derived tables reach "
                                 "the GPU as kernel parameters); out: the 8-byte result key"},
           "gpu_launches": args.steps,  # one search kernel per timed step (per GPU)
           "clocks": clocks, "timed_wall_s": wall, "sm_count": sm_count}
    if world == 1:
        for name, entry in extras["per_config"].items():
            entry.update(issue_roofline(profiled_fields(name), entry["mappings_per_s"], peak_ops))
        out["wall_time_to_optimum_ms"].update(
            host_median=statistics.median(extras["host_ms"]),
            host_note="bf_search_best call as seen by the host (blocks until the result is in pinned host "
                      "memory), median of 10")
        out["per_config"] = extras["per_config"]
        out["pruned_wall_time_to_optimum_ms"] = {
            "median": statistics.median(extras["pruned_ms"]), "min": min(extras["pruned_ms"]),
            "note": "bf_search_pruned: exact branch and bound, same optimum; not a full enumeration"}
        out["tree_search"] = extras["tree"]
        out["result"]["modes"] = extras["modes"]
    if world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        threads = oracle.default_threads()
        n, dt = oracle_sample_time(scn, args.cpu_sample, threads)
        out["cpu_baseline"] = {"value": n / dt, "unit": UNIT, "cores": threads, "kind": "oracle",
                               "sample": f"{n} mappings of the same workload in 16 contiguous chunks spread "
                                         f"evenly over [0, 3^19), oracle search, {dt:.1f} s",
                               "single_core_per_config": oracle_single_core(S),
                               "cpu_model": cpu_model()}
    emit(out)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=("bf", "reference"), default="bf")
    ap.add_argument("--cpu-sample", type=int, default=1 << 25, help="mappings for the oracle CPU baseline")
    ap.add_argument("--ref-sample", type=int, default=1 << 23, help="mappings per --impl reference step")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        return run_reference(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())
