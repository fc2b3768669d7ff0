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

MAX_TOOLS = 20
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
    slowdown_q10: List[int]   # f[k], k=1..20 at [k]; [0] unused; 1024 = no slowdown

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

def slowdown_flat() -> List[int]:
    """No contention: f[k] = 1024 for every k."""
    return [0] + [1024] * MAX_TOOLS


def slowdown_linear(pct_per_extra_tool: int = 35) -> List[int]:
    """f[k] = round-half-up(1024 * (1 + pct/100 * (k-1))) for k = 1..20."""
    return [0] + [(1024 * (100 + pct_per_extra_tool * (k - 1)) + 50) // 100
                  for k in range(1, MAX_TOOLS + 1)]


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


def config3() -> Scenario:
    """N=19 mixed DAG with the four scheduling zones of §2.2; 32 GiB budget; seed 3.

    Categories (11 GPU-preferred, 4 ambiguous, 1 CPU-preferred, 3 neutral, as in
    the Table 1 census) are assigned to tools by a seeded permutation.
    """
    rng = np.random.default_rng(3)
    n = 19
    cats = rng.permutation([GPU_PREFERRED] * 11 + [AMBIGUOUS] * 4 + [CPU_PREFERRED] + [NEUTRAL] * 3)
    c, g, x, m = [], [], [], []
    for i in range(n):
        gi = min(max(_rint(rng.lognormal(np.log(G_MEDIAN_US), G_SIGMA)), 1), G_MAX_US)
        cat = int(cats[i])
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
        c.append(min(max(_rint(ci), 1), C_MAX_US))
        g.append(gi)
        x.append(xi)
        m.append(mi)
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
        for _ in range(2, MAX_TOOLS + 1):
            f.append(f[-1] + int(rng.integers(0, 700)))
    else:
        f = slowdown_flat()
    return Scenario(n, pred, c, g, x, load, m, budget, f)
