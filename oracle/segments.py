"""Optimum of a scenario with serialisation points, segment by segment -- TEST INFRASTRUCTURE.

A serialisation point is a tool s such that every other tool is an ancestor or
a descendant of s.  With tools numbered topologically, the ancestors are
exactly the tools below s and the descendants the tools above it.  Under the
latency model (stated at the top of ``bf_oracle.cpp``) the instant s becomes
ready is the instant the last tool below it ends; nothing runs or waits then,
so s starts at once in every mode and no VRAM is held.  Everything from there
on is a fresh run of the tools >= s, and the model's arithmetic depends only
on differences of T and of V, so that run takes the same time as the
sub-scenario of those tools started at T = 0.

Hence, splitting [0, n) at the serialisation points s_1 < ... < s_k into
segments [0, s_1), [s_1, s_2), ..., [s_k, n): the makespan of a mapping is the
sum of its segments' makespans (infeasible if any segment is), the optimum is
the sum of the segments' optima, and, since segment j owns the digits
[s_j, s_{j+1}) of the index, the lowest optimal index is the sum of the
segments' lowest optimal indices times 3^{s_j}.  Each segment is searched by
the plain oracle (full enumeration), so a workload of 32 tools made of short
segments gets its exact optimum in seconds.

Pinned in ``tests/test_oracle_pins.py`` against full enumeration (random
segmented DAGs, and the 19-tool workload's stored brute-force optimum).
"""
from __future__ import annotations

from typing import List, NamedTuple, Tuple

from . import INFEASIBLE, default


class SubScenario(NamedTuple):
    """The oracle's own record of a segment: the fields its flat record reads."""
    n: int
    pred_mask: List[int]
    cpu_us: List[int]
    gpu_us: List[int]
    xfer_us: List[int]
    load_us: List[int]
    vram_mib: List[int]
    vram_budget_mib: int
    slowdown_q10: List[int]


def serialisation_points(pred_mask: List[int], n: int) -> List[int]:
    """Tools s >= 1 whose ancestors are all tools < s and descendants all tools > s."""
    anc = [0] * n
    for v in range(n):
        a = pred_mask[v]
        for u in range(v):
            if (pred_mask[v] >> u) & 1:
                a |= anc[u]
        anc[v] = a
    desc = [0] * n
    for v in range(n):
        for u in range(v):
            if (anc[v] >> u) & 1:
                desc[u] |= 1 << v
    full = (1 << n) - 1
    pts = []
    for s in range(1, n):
        below = (1 << s) - 1
        if anc[s] == below and desc[s] == full & ~((1 << (s + 1)) - 1):
            pts.append(s)
    return pts


def segment(scn, lo: int, hi: int):
    """The sub-scenario of tools [lo, hi), renumbered from 0 (edges from below lo dropped)."""
    m = hi - lo
    return SubScenario(m, [(scn.pred_mask[v] >> lo) & ((1 << m) - 1) for v in range(lo, hi)],
                       scn.cpu_us[lo:hi], scn.gpu_us[lo:hi], scn.xfer_us[lo:hi], scn.load_us[lo:hi],
                       scn.vram_mib[lo:hi], scn.vram_budget_mib, scn.slowdown_q10)


def bounds(scn) -> List[Tuple[int, int]]:
    cuts = [0] + serialisation_points(scn.pred_mask, scn.n) + [scn.n]
    return list(zip(cuts[:-1], cuts[1:]))


def search(scn, binary: bool = False, threads: int = 1, lib=None) -> Tuple[int, int]:
    """(index, makespan) of the optimum over all 3^n mappings (or the binary
    cpu/gpu_now space), combined from the segments' optima."""
    o = lib or default()
    idx = total = 0
    for lo, hi in bounds(scn):
        sub = segment(scn, lo, hi)
        i, ms = o.search_binary(sub, threads) if binary else o.search(sub, threads)
        if ms == INFEASIBLE:
            return -1, INFEASIBLE
        idx += i * 3 ** lo
        total += ms
    return idx, total


def evaluate(scn, index: int, lib=None) -> int:
    """Makespan of one mapping as the sum of its segments' makespans."""
    o = lib or default()
    total = 0
    for lo, hi in bounds(scn):
        sub_index = (index // 3 ** lo) % 3 ** (hi - lo)
        ms = o.evaluate(segment(scn, lo, hi), sub_index)
        if ms == INFEASIBLE:
            return INFEASIBLE
        total += ms
    return total
