"""Algorithm 1's bounded what-if exploration on the model -- TEST INFRASTRUCTURE.

The exploration step of Algorithm 1 (runtime monitor, §3.2) for a base mapping d: for
each tool i and each alternative mode a != d_i, the single-tool reprobe
d[i := a]; if that reprobe exceeds the VRAM budget and a is gpu_now, a swap
reprobe d[i := gpu_now, j := gpu_queue] for each tool j currently on gpu_now.
"Exceeds" is the model's infeasibility (only VRAM makes a mapping
infeasible).  Reprobes are scored with the C++ oracle; alternative modes are
tried in the order cpu, gpu_now, gpu_queue (the paper gives no order).
"""
from __future__ import annotations

from typing import List, Tuple

from . import INFEASIBLE, evaluate

CPU, GPU_NOW, GPU_QUEUE = 0, 1, 2


def _index(modes) -> int:
    return sum(a * 3 ** i for i, a in enumerate(modes))


def whatif(scn, base_index: int, evaluate=evaluate) -> List[Tuple[str, int, int, object, int, int, bool]]:
    """[(kind, tool, mode, other, index, makespan, feasible), ...] in Algorithm 1's order.

    `evaluate(scn, idx)` scores one mapping (the C++ oracle by default)."""
    d = []
    v = base_index
    for _ in range(scn.n):
        d.append(v % 3)
        v //= 3
    probes = []
    for i in range(scn.n):
        for a in (CPU, GPU_NOW, GPU_QUEUE):
            if a == d[i]:
                continue
            moved = list(d)
            moved[i] = a
            idx = _index(moved)
            ms = evaluate(scn, idx)
            probes.append(("single", i, a, None, idx, ms, ms != INFEASIBLE))
            if ms == INFEASIBLE and a == GPU_NOW:  # r.status = exceed and a = gpu_now
                for j in range(scn.n):
                    if d[j] != GPU_NOW:
                        continue
                    swapped = list(d)
                    swapped[i] = GPU_NOW
                    swapped[j] = GPU_QUEUE
                    sidx = _index(swapped)
                    sms = evaluate(scn, sidx)
                    probes.append(("swap", i, GPU_NOW, j, sidx, sms, sms != INFEASIBLE))
    return probes
