"""Second restatement of the integer latency model -- TEST INFRASTRUCTURE.

Structurally different from ``bf_oracle.cpp`` on purpose, so that a slip in one
shows up as a disagreement:

* GPU progress is kept as per-tool *remaining* work (decremented by every
  advance) instead of a global virtual clock with per-tool end stamps;
* the serialised GPU queue of §2.1 / Factor B (§2.3) is an explicit FIFO list
  (tools that become ready at the same instant are appended in index order)
  instead of a min-search over (ready time, index);
* readiness uses set arithmetic over successor lists instead of predecessor
  bitmasks.

Same model, same integer rounding: a GPU completion is rounded up to a whole
microsecond, and the work done by running GPU tools while a CPU tool ends first
is rounded down to whole 1/1024-microsecond units.  Pure Python; small N only.
"""
from __future__ import annotations

from typing import List, Sequence, Tuple

INFEASIBLE = 0xFFFFFFFF
CPU, GPU_NOW, GPU_QUEUE = 0, 1, 2


def _decode(idx: int, n: int) -> List[int]:
    modes = []
    for _ in range(n):
        idx, d = divmod(idx, 3)
        modes.append(d)
    return modes


def simulate(scn, modes: Sequence[int]) -> Tuple[int, bool]:
    """(makespan, feasible) of one mapping given as a list of modes."""
    n = scn.n
    preds = [{u for u in range(n) if (scn.pred_mask[v] >> u) & 1} for v in range(n)]
    f = scn.slowdown_q10
    budget = scn.vram_budget_mib

    done = set()
    pending = set(range(n))
    cpu_running = {}        # tool -> real end time
    gpu_remaining = {}      # tool -> remaining work, 1/1024 us units
    fifo: List[int] = []    # waiting gpu_queue tools, in arrival order
    queued_running = None   # the queued tool currently on the GPU
    now = 0

    def vram_in_use():
        return sum(scn.vram_mib[v] for v in gpu_remaining)

    def admit() -> bool:
        nonlocal queued_running
        newly = sorted(v for v in pending if preds[v] <= done)
        for v in newly:
            pending.discard(v)
            if modes[v] == CPU:
                cpu_running[v] = now + scn.cpu_us[v]
            elif modes[v] == GPU_NOW:
                gpu_remaining[v] = 1024 * (scn.gpu_us[v] + scn.xfer_us[v])
            else:
                fifo.append(v)
        if vram_in_use() > budget:
            return False
        if fifo:
            head = fifo[0]
            if scn.vram_mib[head] > budget:
                return False
            if queued_running is None and vram_in_use() + scn.vram_mib[head] <= budget:
                fifo.pop(0)
                gpu_remaining[head] = 1024 * (scn.load_us[head] + scn.gpu_us[head] + scn.xfer_us[head])
                queued_running = head
        return True

    if not admit():
        return INFEASIBLE, False
    while len(done) < n:
        k = len(gpu_remaining)
        next_cpu = min(cpu_running.values()) if cpu_running else None
        if k:
            least = min(gpu_remaining.values())
            gpu_dt = -((-least * f[k]) // (1 << 20))          # ceil
        if k and (next_cpu is None or now + gpu_dt <= next_cpu):
            dt, dwork = gpu_dt, least
        else:
            dt = next_cpu - now
            dwork = (dt * (1 << 20)) // f[k] if k else 0        # floor
        now += dt
        for v in list(gpu_remaining):
            gpu_remaining[v] -= dwork
            if gpu_remaining[v] == 0:
                del gpu_remaining[v]
                done.add(v)
                if v == queued_running:
                    queued_running = None
        for v, end in list(cpu_running.items()):
            if end == now:
                del cpu_running[v]
                done.add(v)
        if not admit():
            return INFEASIBLE, False
    return now, True


def evaluate(scn, idx: int) -> Tuple[int, bool]:
    return simulate(scn, _decode(idx, scn.n))


def search(scn) -> Tuple[int, int]:
    best = None
    for idx in range(3 ** scn.n):
        ms, ok = evaluate(scn, idx)
        if ok and (best is None or ms < best[1]):
            best = (idx, ms)
    return best
