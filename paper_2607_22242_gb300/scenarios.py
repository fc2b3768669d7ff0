"""Seeded synthetic scenario generator (inputs only).

This module draws the workflow DAGs and per-tool tables that both the CUDA
search and the CPU oracle consume.  It holds none of the latency model's
arithmetic: it only produces numbers (latencies, transfers, load-in times,
VRAM footprints, budgets, contention tables, edges) and serialises them.

A scenario follows the problem statement of §2.1: a DAG G=(V,E) of N tool
invocations numbered 0..N-1 in a topological order (every edge u->v has u<v),
per-tool profiles as in Table 1 (CPU time, GPU time, load-in time, VRAM
footprint, §3.1) plus a host<->device transfer time, a VRAM budget M, and a
GPU-contention slowdown table f[k] (Factor A, §2.3) in 1/1024 units.

Units: integer microseconds for times, MiB for memory ("GB" in the workload
recipes means GiB).  Draws use numpy's PCG64 ``default_rng(seed)``; values are
rounded half-to-even.  The five standard workloads are ``config(0..4)``.
"""
from __future__ import annotations

import dataclasses
import hashlib
import json
from typing import List, Sequence

import numpy as np

MAX_TOOLS = 32          # largest scenario the library takes (32-bit tool masks)
ENUM_MAX_TOOLS = 20     # largest scenario of the full-enumeration searches (3^20 < 2^32 indices)
CPU, GPU_NOW, GPU_QUEUE = 0, 1, 2
MODE_NAMES = ("cpu", "gpu_now", "gpu_queue")


@dataclasses.dataclass
class Scenario:
    """One workflow: DAG plus per-tool tables (§2.1, Table 1 columns)."""

    n: int
    pred_mask: List[int]      # bit u of pred_mask[v] set iff edge u->v (u < v)
    cpu_us: List[int]         # c_i: CPU latency
    gpu_us: List[int]         # g_i: GPU compute latency (isolated)
    xfer_us: List[int]        # x_i: host<->device transfer, paid in GPU modes
    load_us: List[int]        # l_i: gpu_queue load-in cost
    vram_mib: List[int]       # m_i: VRAM footprint
    vram_budget_mib: int      # M
    slowdown_q10: List[int]   # f[k], k=1..n (or more) at [k]; [0] unused; 1024 = no slowdown

    def __post_init__(self):
        for name in ("pred_mask", "cpu_us", "gpu_us", "xfer_us", "load_us", "vram_mib"):
            setattr(self, name, [int(v) for v in getattr(self, name)])
        self.slowdown_q10 = [int(v) for v in self.slowdown_q10]
        self.n = int(self.n)
        self.vram_budget_mib = int(self.vram_budget_mib)

    @property
    def num_mappings(self) -> int:
        return 3 ** self.n

    def to_dict(self) -> dict:
        return dataclasses.asdict(self)

    @staticmethod
    def from_dict(d: dict) -> "Scenario":
        return Scenario(**d)

    def canonical_bytes(self) -> bytes:
        return json.dumps(self.to_dict(), sort_keys=True, separators=(",", ":")).encode()


def sha256_of(scenarios: Sequence[Scenario]) -> str:
    h = hashlib.sha256()
    for s in scenarios:
        h.update(s.canonical_bytes())
    return h.hexdigest()


def mapping_index(modes: Sequence[int]) -> int:
    """Canonical index of a mapping: sum_i a_i * 3**i (tool 0 least significant)."""
    idx = 0
    for i, a in enumerate(modes):
        idx += int(a) * 3 ** i
    return idx


def mapping_modes(index: int, n: int) -> List[int]:
    """Inverse of :func:`mapping_index`."""
    out = []
    for _ in range(n):
        out.append(index % 3)
        index //= 3
    return out


# ---------------------------------------------------------------------------
# Contention tables (inputs).  f[k] is the slowdown of each of k concurrently
# running GPU tools, in 1/1024 units (Factor A, §2.3: concurrent GPU tools
# slow each other; CPU tools are unaffected).
# ---------------------------------------------------------------------------

def slowdown_flat(kmax: int = ENUM_MAX_TOOLS) -> List[int]:
    """No contention: f[k] = 1024 for k = 1..kmax."""
    return [0] + [1024] * kmax


def slowdown_linear(pct_per_extra_tool: int = 35, kmax: int = ENUM_MAX_TOOLS) -> List[int]:
    """f[k] = round-half-up(1024 * (1 + pct/100 * (k-1))) for k = 1..kmax."""
    return [0] + [(1024 * (100 + pct_per_extra_tool * (k - 1)) + 50) // 100
                  for k in range(1, kmax + 1)]


# ---------------------------------------------------------------------------
# Per-tool draws shared by the standard workloads.
# ---------------------------------------------------------------------------

G_MEDIAN_US = 40000.0
G_SIGMA = 0.8
G_MAX_US = 2_000_000
C_MAX_US = 40_000_000


def _rint(v: float) -> int:
    return int(np.rint(v))


def _draw_tool(rng: np.random.Generator, m_lo: int, m_hi: int):
    """Draw (g, ratio, x, m) in that order for one ordinary tool."""
    g = min(max(_rint(rng.lognormal(np.log(G_MEDIAN_US), G_SIGMA)), 1), G_MAX_US)
    ratio = rng.uniform(0.5, 20.0)
    x = _rint(rng.uniform(1000.0, 30000.0))
    m = int(rng.integers(m_lo, m_hi, endpoint=True))
    c = min(max(_rint(g * ratio), 1), C_MAX_US)
    return c, g, x, m


def _load_from_vram(m: int) -> int:
    # Load-in time for gpu_queue: 40 us per MiB (about 26 GB/s of weight upload).
    return 40 * m


def _layered_edges(rng: np.random.Generator, layer_sizes: Sequence[int], p: float) -> List[int]:
    """Edges between consecutive layers, each present with probability p."""
    starts = np.cumsum([0] + list(layer_sizes))
    n = int(starts[-1])
    pred = [0] * n
    for li in range(len(layer_sizes) - 1):
        for u in range(starts[li], starts[li + 1]):
            for v in range(starts[li + 1], starts[li + 2]):
                if rng.uniform() < p:
                    pred[v] |= 1 << u
    return pred


def _ordinary(rng, n, m_lo, m_hi):
    cols = [_draw_tool(rng, m_lo, m_hi) for _ in range(n)]
    c, g, x, m = (list(t) for t in zip(*cols))
    return c, g, x, m


# ---------------------------------------------------------------------------
# The five standard workloads.
# ---------------------------------------------------------------------------

def config0() -> Scenario:
    """N=8 serial chain, no VRAM pressure (80 GiB), no contention; seed 0."""
    rng = np.random.default_rng(0)
    c, g, x, m = _ordinary(rng, 8, 512, 6144)
    pred = [0] + [1 << (i - 1) for i in range(1, 8)]
    return Scenario(8, pred, c, g, x, [_load_from_vram(v) for v in m], m,
                    81920, slowdown_flat())


def config1() -> Scenario:
    """N=12 fan-out/fan-in: tool 0 -> tools 1..10 -> tool 11; seed 1."""
    rng = np.random.default_rng(1)
    c, g, x, m = _ordinary(rng, 12, 512, 6144)
    pred = [0] + [1] * 10 + [((1 << 11) - 1) & ~1]
    return Scenario(12, pred, c, g, x, [_load_from_vram(v) for v in m], m,
                    81920, slowdown_linear())


def config2() -> Scenario:
    """N=16 random layered DAG (4 layers of 4, p=0.4), 2..16 GiB tools vs 24 GiB; seed 2."""
    rng = np.random.default_rng(2)
    c, g, x, m = _ordinary(rng, 16, 2048, 16384)
    pred = _layered_edges(rng, [4, 4, 4, 4], 0.4)
    return Scenario(16, pred, c, g, x, [_load_from_vram(v) for v in m], m,
                    24576, slowdown_linear())


# Tool layout of config 3 (topological numbering):
#   spine s0..s6 = 0,1,2,9,10,11,18; fan-out F1 = 3..8 (pred s1, all -> s3);
#   fan-out F2 = 12..17 (pred s4, all -> s6); s2 follows s1 and precedes s3.
CONFIG3_SPINE = (0, 1, 2, 9, 10, 11, 18)
CONFIG3_F1 = tuple(range(3, 9))
CONFIG3_F2 = tuple(range(12, 18))
GPU_PREFERRED, AMBIGUOUS, CPU_PREFERRED, NEUTRAL = range(4)


def _zoned_tool(rng: np.random.Generator, cat: int):
    """Draw one tool of a scheduling zone (§2.2): g, then the zone's c, x, m."""
    gi = min(max(_rint(rng.lognormal(np.log(G_MEDIAN_US), G_SIGMA)), 1), G_MAX_US)
    if cat == GPU_PREFERRED:
        ci = gi * rng.uniform(5.0, 70.0)
        xi = _rint(rng.uniform(1000.0, 30000.0))
        mi = int(rng.integers(512, 6144, endpoint=True))
    elif cat == AMBIGUOUS:
        ci = gi * rng.uniform(0.8, 1.5)
        xi = _rint(rng.uniform(1000.0, 30000.0))
        mi = int(rng.integers(512, 6144, endpoint=True))
    elif cat == CPU_PREFERRED:
        xi = _rint(gi * rng.uniform(1.5, 3.0))
        ci = (gi + xi) * rng.uniform(0.3, 0.5)
        mi = int(rng.integers(512, 6144, endpoint=True))
    else:
        ci = gi * rng.uniform(0.95, 1.05)
        xi = _rint(rng.uniform(0.0, 1000.0))
        mi = int(rng.integers(16, 128, endpoint=True))
    return min(max(_rint(ci), 1), C_MAX_US), gi, xi, mi


def _zoned_tools(rng: np.random.Generator, zone_counts: Sequence[int]):
    """Zones assigned to tools by a seeded permutation, then each tool's draws in index order."""
    cats = rng.permutation(sum(([z] * k for z, k in enumerate(zone_counts)), []))
    cols = [_zoned_tool(rng, int(cat)) for cat in cats]
    return [list(t) for t in zip(*cols)]


def config3() -> Scenario:
    """N=19 mixed DAG with the four scheduling zones of §2.2; 32 GiB budget; seed 3.

    Categories (11 GPU-preferred, 4 ambiguous, 1 CPU-preferred, 3 neutral, as in
    the Table 1 census) are assigned to tools by a seeded permutation.
    """
    rng = np.random.default_rng(3)
    n = 19
    c, g, x, m = _zoned_tools(rng, (11, 4, 1, 3))
    pred = [0] * n
    s0, s1, s2, s3, s4, s5, s6 = CONFIG3_SPINE
    pred[s1] = 1 << s0
    pred[s2] = 1 << s1
    for v in CONFIG3_F1:
        pred[v] = 1 << s1
    pred[s3] = (1 << s2) | sum(1 << v for v in CONFIG3_F1)
    pred[s4] = 1 << s3
    pred[s5] = 1 << s4
    for v in CONFIG3_F2:
        pred[v] = 1 << s4
    pred[s6] = (1 << s5) | sum(1 << v for v in CONFIG3_F2)
    return Scenario(n, pred, c, g, x, [_load_from_vram(v) for v in m], m,
                    32768, slowdown_linear())


def config3_categories() -> List[int]:
    rng = np.random.default_rng(3)
    return [int(v) for v in rng.permutation(
        [GPU_PREFERRED] * 11 + [AMBIGUOUS] * 4 + [CPU_PREFERRED] + [NEUTRAL] * 3)]


def config4(count: int = 4096) -> List[Scenario]:
    """Batch of independent N=10 layered scenarios ([3,3,2,2], p=0.3); seed 4.

    Each scenario draws its tools (2..16 GiB footprints), then its edges, then its
    budget uniform over [16, 48] GiB.  ``count`` < 4096 returns a prefix.
    """
    rng = np.random.default_rng(4)
    out = []
    for _ in range(count):
        c, g, x, m = _ordinary(rng, 10, 2048, 16384)
        pred = _layered_edges(rng, [3, 3, 2, 2], 0.3)
        budget = int(rng.integers(16384, 49152, endpoint=True))
        out.append(Scenario(10, pred, c, g, x, [_load_from_vram(v) for v in m], m,
                            budget, slowdown_linear()))
    return out


# ---------------------------------------------------------------------------
# Workloads beyond 20 tools (the tree search, bf_search_tree).  The config-3
# recipe grown by one more spine segment and wider fan-outs: spine
# s0 -> s1 -> s2 -> s3 -> ... ; fan-out j (width w) hangs off spine tool
# s(3j+1) and joins at s(3j+3), beside s(3j+2).  Zones in config 3's
# proportions (11 : 4 : 1 : 3 of 19), seeded permutation; 32 GiB budget;
# f = 1 + 0.35 (k-1) up to k = n.
# ---------------------------------------------------------------------------

def spine_fanout_layout(fanouts: int, width: int, tail: int):
    """(n, pred) of the spine/fan-out DAG in topological numbering, ``tail`` spine tools after the last join."""
    pred: List[int] = []
    prev = None

    def add(mask):
        pred.append(mask)
        return len(pred) - 1

    prev = add(0)                      # s0
    for _ in range(fanouts):
        head = add(1 << prev)          # s(3j+1): the fan-out's source
        side = add(1 << head)          # s(3j+2)
        fan = [add(1 << head) for _ in range(width)]
        prev = add((1 << side) | sum(1 << v for v in fan))  # s(3j+3): the join
    for _ in range(tail):
        prev = add(1 << prev)
    return len(pred), pred


def _wide(fanouts: int, width: int, tail: int, zones, seed: int) -> Scenario:
    n, pred = spine_fanout_layout(fanouts, width, tail)
    assert sum(zones) == n
    rng = np.random.default_rng(seed)
    c, g, x, m = _zoned_tools(rng, zones)
    return Scenario(n, pred, c, g, x, [_load_from_vram(v) for v in m], m,
                    32768, slowdown_linear(kmax=n))


def wide28() -> Scenario:
    """N=28: spine of 10, three fan-outs of 6; zones 16/6/2/4; seed 5 (the full 3^28 space)."""
    return _wide(3, 6, 0, (16, 6, 2, 4), 5)


def wide32() -> Scenario:
    """N=32: spine of 11, three fan-outs of 7; zones 18/7/2/5; seed 6 (the binary 2^32 space)."""
    return _wide(3, 7, 1, (18, 7, 2, 5), 6)


def layered24() -> Scenario:
    """N=24 random layered DAG (6 layers of 4, p=0.4), 2..16 GiB tools vs 40 GiB; seed 7.
    No serialisation point: its binary space (2^24) is searched whole by the oracle."""
    rng = np.random.default_rng(7)
    c, g, x, m = _ordinary(rng, 24, 2048, 16384)
    pred = _layered_edges(rng, [4] * 6, 0.4)
    return Scenario(24, pred, c, g, x, [_load_from_vram(v) for v in m], m,
                    40960, slowdown_linear(kmax=24))


WIDE_NAMES = {
    "wide28": "N=28 spine+3 fan-outs of 6, 4 zones, 32 GiB (3^28 mappings)",
    "wide32": "N=32 spine+3 fan-outs of 7, 4 zones, 32 GiB (3^32 mappings; binary space 2^32)",
    "layered24": "N=24 layered 6x4 p=0.4, 2-16 GiB vs 40 GiB (binary space, 2^24 mappings)",
}


def config(i: int):
    return (config0, config1, config2, config3, config4)[i]()


CONFIG_NAMES = (
    "N=8 serial chain, 80 GiB, no contention",
    "N=12 fan-out/fan-in, 80 GiB, f=1+0.35(k-1)",
    "N=16 layered 4x4 p=0.4, 2-16 GiB vs 24 GiB",
    "N=19 spine+2 fan-outs, 4 zones, 32 GiB",
    "4096 x N=10 layered [3,3,2,2] p=0.3, 16-48 GiB",
)


# ---------------------------------------------------------------------------
# Small random scenarios for tests: small integers so that ties between event
# times, VRAM-blocked queues and infeasible starts all occur often.
# ---------------------------------------------------------------------------

def random_small(rng: np.random.Generator, n: int, *, edge_p: float = 0.4,
                 tight: bool = True, contention: bool = True,
                 max_time: int = 40) -> Scenario:
    pred = [0] * n
    for v in range(n):
        for u in range(v):
            if rng.uniform() < edge_p:
                pred[v] |= 1 << u
    c = [int(rng.integers(1, max_time + 1)) for _ in range(n)]
    g = [int(rng.integers(1, max_time + 1)) for _ in range(n)]
    x = [int(rng.integers(0, max_time // 4 + 1)) for _ in range(n)]
    load = [int(rng.integers(0, max_time // 2 + 1)) for _ in range(n)]
    m = [int(rng.integers(1, 11)) for _ in range(n)]
    budget = int(rng.integers(5, 16)) if tight else 10 * n + 10
    if contention:
        f = [0, 1024]
        for _ in range(2, max(ENUM_MAX_TOOLS, n) + 1):
            f.append(f[-1] + int(rng.integers(0, 700)))
    else:
        f = slowdown_flat(max(ENUM_MAX_TOOLS, n))
    return Scenario(n, pred, c, g, x, load, m, budget, f)


def random_segmented(rng: np.random.Generator, n: int, *, seg_max: int = 6, edge_p: float = 0.4,
                     **kw) -> Scenario:
    """A ``random_small`` scenario whose DAG is a row of segments joined at
    serialisation points: each segment's first tool has every tool of the
    previous segment as a predecessor, and every other tool of a segment has at
    least one predecessor inside it (random edges with probability ``edge_p``,
    else the segment's first tool).  Segment lengths are uniform in 1..seg_max."""
    base = random_small(rng, n, edge_p=0.0, **kw)
    cuts = [0]
    while cuts[-1] < n:
        cuts.append(min(n, cuts[-1] + int(rng.integers(1, seg_max + 1))))
    pred = [0] * n
    for j in range(len(cuts) - 1):
        lo, hi = cuts[j], cuts[j + 1]
        pred[lo] = ((1 << lo) - 1) & ~((1 << cuts[j - 1]) - 1) if j else 0
        for v in range(lo + 1, hi):
            m = sum(1 << u for u in range(lo, v) if rng.uniform() < edge_p)
            pred[v] = m or (1 << lo)
    return Scenario(**{**base.to_dict(), "pred_mask": pred})
