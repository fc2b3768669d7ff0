"""Classical scheduling baselines on the model, scored against the brute-force optimum.

The paper compares its scheduler with All-GPU, HEFT, UCB1, StarPU and, under
VRAM pressure, a memory-aware greedy policy (§4.1, §4.4).  Three of them are
deterministic policies that map a scenario to one mapping; this module states
them, scores their mappings with ``bf_eval_indices`` and the optimum with
``bf_search_best`` (both on the GPU), and reports the gap.

* All-GPU (§4.1): every tool on the GPU, i.e. gpu_now everywhere.
* Memory-aware greedy (§4.4): tools in decreasing GPU speedup c/(g+x) (ties to
  the lower index) go to gpu_now while the sum of their footprints fits the
  budget; the first tool that does not fit exhausts the budget, and it and
  every later tool run on the CPU.
* HEFT (Topcuoglu, Hariri and Wu, IEEE TPDS 2002): tasks in decreasing upward
  rank (mean of CPU and GPU cost plus the largest rank of a successor; no
  communication costs, transfers being part of GPU time), each placed on the
  processor giving the earliest finish time.  Processors: the CPU pool
  (unlimited cores, so a CPU task starts when its predecessors finish) and the
  GPU as one exclusive processor with insertion into idle gaps.  A task placed
  on the GPU becomes gpu_now.  HEFT sees neither contention nor VRAM, which is
  exactly the gap the model exposes.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List

from .scenarios import CPU, GPU_NOW, Scenario, mapping_index


def all_gpu(scn: Scenario) -> List[int]:
    return [GPU_NOW] * scn.n


def memory_aware_greedy(scn: Scenario) -> List[int]:
    order = sorted(range(scn.n), key=lambda i: (-scn.cpu_us[i] / (scn.gpu_us[i] + scn.xfer_us[i]), i))
    modes = [CPU] * scn.n
    used = 0
    for i in order:
        if used + scn.vram_mib[i] > scn.vram_budget_mib:
            break  # budget exhausted: this tool and all later ones stay on the CPU
        used += scn.vram_mib[i]
        modes[i] = GPU_NOW
    return modes


def heft(scn: Scenario) -> List[int]:
    n = scn.n
    succ = [[v for v in range(n) if (scn.pred_mask[v] >> u) & 1] for u in range(n)]
    preds = [[u for u in range(n) if (scn.pred_mask[v] >> u) & 1] for v in range(n)]
    gpu_cost = [scn.gpu_us[i] + scn.xfer_us[i] for i in range(n)]
    mean = [(scn.cpu_us[i] + gpu_cost[i]) / 2.0 for i in range(n)]
    rank = [0.0] * n
    for v in reversed(range(n)):  # topological numbering: successors have larger indices
        rank[v] = mean[v] + max((rank[s] for s in succ[v]), default=0.0)
    order = sorted(range(n), key=lambda v: (-rank[v], v))
    finish = [0] * n
    gpu_busy: List[tuple] = []  # (start, end) intervals, kept sorted
    modes = [CPU] * n
    for v in order:
        ready = max((finish[u] for u in preds[v]), default=0)
        cpu_eft = ready + scn.cpu_us[v]
        # earliest GPU slot of length gpu_cost[v] starting at or after `ready`
        start = ready
        for a, b in gpu_busy:
            if start + gpu_cost[v] <= a:
                break
            start = max(start, b)
        gpu_eft = start + gpu_cost[v]
        if gpu_eft < cpu_eft:
            modes[v] = GPU_NOW
            finish[v] = gpu_eft
            gpu_busy.append((start, gpu_eft))
            gpu_busy.sort()
        else:
            finish[v] = cpu_eft
    return modes


POLICIES = {"all_gpu": all_gpu, "memory_aware_greedy": memory_aware_greedy, "heft": heft}


@dataclasses.dataclass
class Gap:
    policy: str
    index: int
    makespan_us: int       # 0xFFFFFFFF when the policy's mapping is infeasible
    feasible: bool
    gap: float             # makespan / optimum - 1 (inf when infeasible)


def gaps(handle, stream=None) -> Dict[str, Gap]:
    """Each policy's mapping scored on the GPU, against the optimum of the same scenario."""
    import torch
    from . import bf
    scn = handle.scenario
    best = bf.search_best(handle, stream)
    names = list(POLICIES)
    idx = [mapping_index(POLICIES[p](scn)) for p in names]
    ms, fe = bf.eval_indices(handle, torch.tensor(idx, dtype=torch.int64, device="cuda"), stream=stream)
    ms = [int(v) & 0xFFFFFFFF for v in ms.cpu().tolist()]
    fe = [int(v) for v in fe.cpu().tolist()]
    out = {}
    for p, i, m, f in zip(names, idx, ms, fe):
        feasible = f == 1
        out[p] = Gap(p, i, m, feasible, m / best.makespan_us - 1.0 if feasible else float("inf"))
    out["optimum"] = Gap("optimum", best.index, best.makespan_us, True, 0.0)
    return out
