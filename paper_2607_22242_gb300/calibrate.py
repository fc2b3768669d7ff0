"""Contention-table calibration on the paper's scenario S5 with the batched search.

The latency model takes GPU contention as a slowdown table f[k] (processor
sharing, Factor A of §2.3).  The paper measures S5 (§4.3; Table 2): four
amplified tools in a fan-out, ocr_x2 || whisper_x4 || vector_search_x15 ||
image_resize_x30, with a binary CPU/GPU decision space.  Its measured oracle
mapping offloads vector_search_x15 to the CPU (Table 2, Table 3: GPU, GPU,
CPU, GPU), with end-to-end latencies 988 ms for All-GPU and 812 ms for the
oracle mapping (Table 2).

This module builds S5 under a family of candidate tables
f[k] = 1024 (1 + a (k-1)^b), runs the brute-force search of every candidate in
one bf_search_batch launch, scores the two measured mappings of every
candidate with bf_eval_indices, and keeps the candidates under which the
paper's oracle mapping is optimal (its makespan equals the optimum; with
vector_search_x15 on the CPU for 706 ms, moving image_resize_x30 to the CPU as
well ties it, and the search reports the tie's lower index); among those, the
best fit minimises the squared error to the two measured end-to-end
latencies.

Inputs (milliseconds converted to microseconds): isolated GPU times from
Table 2 (370, 136, 277, 145); CPU times = the isolated GPU time times the
tool's CPU/GPU ratio (Table 1 for ocr and whisper; 3.7x for image_resize as
stated in §4.3), except vector_search_x15, whose CPU time is measured in
Table 2 (706 ms); footprints from Table 1 (248, 442, 3106, 340 MB; Table 3
total 4136).  GPU time includes transfer (x = 0).  The decision space is
binary, so gpu_queue is priced out with a 3 s load-in (never optimal), and
the budget is unconstrained (80 GiB).
"""
from __future__ import annotations

import dataclasses
from typing import List, Sequence, Tuple

from .scenarios import CPU, GPU_NOW, MAX_TOOLS, Scenario, mapping_index

S5_TOOLS = ("ocr_x2", "whisper_x4", "vector_search_x15", "image_resize_x30")
S5_GPU_MS = (370, 136, 277, 145)
S5_CPU_MS = (370 * 1386 / 176, 136 * 473 / 35, 706, 145 * 3.7)
S5_VRAM_MB = (248, 442, 3106, 340)
S5_ALL_GPU = (GPU_NOW, GPU_NOW, GPU_NOW, GPU_NOW)
S5_ORACLE = (GPU_NOW, GPU_NOW, CPU, GPU_NOW)
S5_MEASURED_US = {"all_gpu": 988_000, "oracle": 812_000}
QUEUE_PRICED_OUT_US = 3_000_000


def table(a: float, b: float) -> List[int]:
    """f[k] = round(1024 (1 + a (k-1)^b)) for k = 1..MAX_TOOLS (the desc's 32 slots); f[0] unused."""
    return [0] + [int(round(1024 * (1 + a * (k - 1) ** b))) for k in range(1, MAX_TOOLS + 1)]


def s5(f: Sequence[int]) -> Scenario:
    us = lambda v: int(round(v * 1000))
    return Scenario(4, [0, 0, 0, 0], [us(v) for v in S5_CPU_MS], [us(v) for v in S5_GPU_MS], [0] * 4,
                    [QUEUE_PRICED_OUT_US - us(v) for v in S5_GPU_MS], list(S5_VRAM_MB), 81920, list(f))


def candidates(a_steps: int = 301, a_max: float = 3.0, bs: Sequence[float] = (0.5, 0.75, 1.0, 1.5, 2.0)):
    """(a, b) pairs of the candidate family; a in [0, a_max]."""
    return [(a_max * i / (a_steps - 1), b) for b in bs for i in range(a_steps)]


@dataclasses.dataclass
class Fit:
    a: float
    b: float
    f: List[int]
    argmin: int
    optimum_us: int
    all_gpu_us: int
    oracle_us: int
    error_us2: float

    @property
    def paper_oracle_optimal(self) -> bool:
        return self.oracle_us == self.optimum_us


def calibrate(stream=None, grid=None) -> Tuple[Fit, List[Fit]]:
    """(best fit, every candidate) -- each candidate's optimum from one batched search."""
    import torch
    from . import bf
    grid = grid or candidates()
    scns = [s5(table(a, b)) for a, b in grid]
    optima = bf.search_batch(scns, stream)
    pair = torch.tensor([mapping_index(S5_ALL_GPU), mapping_index(S5_ORACLE)], dtype=torch.int64, device="cuda")
    fits = []
    for (a, b), scn, opt in zip(grid, scns, optima):
        with bf.create_scenario(scn) as h:
            ms, _ = bf.eval_indices(h, pair, stream=stream)
        e_all, e_or = [int(v) & 0xFFFFFFFF for v in ms.cpu().tolist()]
        err = float(e_all - S5_MEASURED_US["all_gpu"]) ** 2 + float(e_or - S5_MEASURED_US["oracle"]) ** 2
        fits.append(Fit(a, b, scn.slowdown_q10, opt.index, opt.makespan_us, e_all, e_or, err))
    matching = [f for f in fits if f.paper_oracle_optimal]
    best = min(matching or fits, key=lambda f: f.error_us2)
    return best, fits
