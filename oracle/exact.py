"""The latency model in exact rational arithmetic -- TEST INFRASTRUCTURE.

Processor sharing (Factor A, §2.3) without any rounding: while k GPU tools run,
each progresses at exactly 1024/f[k] isolated microseconds per microsecond, and
event times are exact fractions.  Everything else (admission, the FIFO GPU
queue, the VRAM rules of §2.1 and Factor B) is as in the integer model.

Used only to bound the integer model's rounding: on mappings without
gpu_queue whose feasibility is the same in both, the integer makespan lies
within a small number of microseconds of this one.
"""
from __future__ import annotations

from fractions import Fraction
from typing import List, Sequence, Tuple

CPU, GPU_NOW, GPU_QUEUE = 0, 1, 2


def simulate(scn, modes: Sequence[int]) -> Tuple[Fraction, bool, int]:
    """(exact makespan, feasible, number of events)."""
    n = scn.n
    preds = [{u for u in range(n) if (scn.pred_mask[v] >> u) & 1} for v in range(n)]
    f = scn.slowdown_q10
    budget = scn.vram_budget_mib
    done, pending = set(), set(range(n))
    cpu_end = {}
    remaining = {}            # isolated microseconds of work left, exact
    fifo: List[int] = []
    queued_running = None
    now = Fraction(0)
    events = 0

    def admit() -> bool:
        nonlocal queued_running
        for v in sorted(v for v in pending if preds[v] <= done):
            pending.discard(v)
            if modes[v] == CPU:
                cpu_end[v] = now + scn.cpu_us[v]
            elif modes[v] == GPU_NOW:
                remaining[v] = Fraction(scn.gpu_us[v] + scn.xfer_us[v])
            else:
                fifo.append(v)
        if sum(scn.vram_mib[v] for v in remaining) > budget:
            return False
        if fifo:
            head = fifo[0]
            if scn.vram_mib[head] > budget:
                return False
            if queued_running is None and sum(scn.vram_mib[v] for v in remaining) + scn.vram_mib[head] <= budget:
                fifo.pop(0)
                remaining[head] = Fraction(scn.load_us[head] + scn.gpu_us[head] + scn.xfer_us[head])
                queued_running = head
        return True

    if not admit():
        return Fraction(-1), False, 0
    while len(done) < n:
        events += 1
        k = len(remaining)
        rate = Fraction(1024, f[k]) if k else None
        candidates = list(cpu_end.values())
        if k:
            candidates.append(now + min(remaining.values()) / rate)
        t = min(candidates)
        if k:
            for v in remaining:
                remaining[v] -= (t - now) * rate
        now = t
        for v in [v for v, r in remaining.items() if r == 0]:
            del remaining[v]
            done.add(v)
            if v == queued_running:
                queued_running = None
        for v in [v for v, e in cpu_end.items() if e == now]:
            del cpu_end[v]
            done.add(v)
        if not admit():
            return Fraction(-1), False, events
    return now, True, events
