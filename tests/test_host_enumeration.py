"""The search kernels' enumeration logic, built for the host, against the oracle (no GPU).

tests/host_enum.cpp compiles bf_plan.h, bf_enum.cuh and bf_sim.cuh -- the code the kernels run --
with g++ and executes each plan's warp tasks lane by lane.  Every mapping's makespan, stored at its
canonical index, must equal the oracle's: in the scenario's numbering over whole spaces and index
ranges, and over whole spaces renumbered with the sources first.  This checks splits, windows, the
closed-form last tool, the renumbering and the canonical index arithmetic on every CPU test run;
the GPU tests check the same on the hardware.  The lane-tree kernels' code (bf_lanetree.cuh) is
run the same way, lane by lane, by the lanetree tests below.
"""
import ctypes
import os
import subprocess
import tempfile

import numpy as np
import pytest

import oracle
from paper_2607_22242_gb300 import bf
from paper_2607_22242_gb300 import scenarios as S
from tie_cases import tie_order_scenarios

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
THREADS = oracle.default_threads()


@pytest.fixture(scope="module")
def host():
    out = os.path.join(tempfile.mkdtemp(prefix="bf_host_enum_"), "host_enum.so")
    subprocess.run(["g++", "-O2", "-std=c++17", "-shared", "-fPIC", "-I", os.path.join(ROOT, "include"), "-o", out,
                    os.path.join(HERE, "host_enum.cpp")], check=True)
    lib = ctypes.CDLL(out)
    lib.host_eval.argtypes = [ctypes.POINTER(bf.Desc), ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint32,
                              ctypes.c_void_p, ctypes.c_void_p]
    lib.host_eval.restype = ctypes.c_int
    lib.host_pruned.argtypes = [ctypes.POINTER(bf.Desc), ctypes.c_uint32]
    lib.host_pruned.restype = ctypes.c_uint64

    def run(scn, first, count, mode):
        d = bf.to_desc(scn)
        ms = np.zeros(count, np.uint32)
        info = np.zeros(6, np.uint32)
        assert lib.host_eval(ctypes.byref(d), first, count, mode, ms.ctypes.data, info.ctypes.data) == 0
        return ms.astype(np.uint64), info
    run.pruned = lambda scn, bound: lib.host_pruned(ctypes.byref(bf.to_desc(scn)), bound)
    lib.host_lanetree.argtypes = [ctypes.POINTER(bf.Desc), ctypes.c_uint32, ctypes.c_uint64, ctypes.c_int,
                                  ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p]
    lib.host_lanetree.restype = ctypes.c_int

    def lanetree(scn, lanes, min_roots=0, sampled=False, wide=False):
        ms = np.zeros(3 ** scn.n, np.uint32)
        info = np.zeros(3, np.uint32)
        assert lib.host_lanetree(ctypes.byref(bf.to_desc(scn)), lanes, min_roots, int(sampled), int(wide),
                                 ms.ctypes.data, info.ctypes.data) == 0
        return ms.astype(np.uint64), info
    run.lanetree = lanetree
    return run


def _same(host, scn, first, count, mode):
    got, info = host(scn, first, count, mode)
    want, _ = oracle.eval_range(scn, first, count, THREADS)
    bad = np.flatnonzero(got != want)
    assert bad.size == 0, (f"mode {mode}, plan {info.tolist()}: {bad.size} mismatches, first at index "
                           f"{first + int(bad[0])}: {int(got[bad[0]])} vs {int(want[bad[0]])}")
    return info


def test_random_dags_every_mode(host):
    """Random DAGs of 1-9 tools with small integer times (ties, blocked queues, infeasible
    starts), some with late sources or a last tool that waits for all others: every mapping in both
    modes, and random index ranges in the scenario's numbering."""
    rng = np.random.default_rng(90)
    flags = 0
    for t in range(240):
        n = int(rng.integers(1, 10))
        base = S.random_small(rng, n, edge_p=float(rng.choice([0.0, 0.25, 0.5, 0.8])), tight=bool(t % 3),
                              contention=bool(t % 4), max_time=int(rng.choice([3, 7, 40, 2000])))
        pred = list(base.pred_mask)
        if t % 3 == 0 and n > 3:
            pred[int(rng.integers(n // 2, n))] = 0
        if t % 4 == 1 and n > 2:
            pred[n - 1] = (1 << (n - 1)) - 1
        scn = S.Scenario(n, pred, base.cpu_us, base.gpu_us, base.xfer_us, base.load_us, base.vram_mib,
                         base.vram_budget_mib, base.slowdown_q10)
        total = 3 ** n
        for mode in (0, 1):
            flags |= int(_same(host, scn, 0, total, mode)[5])
        if total > 3:
            a = int(rng.integers(0, total - 2))
            _same(host, scn, a, int(rng.integers(1, total - a + 1)), 0)
    assert flags == 3, flags  # renumbered and last tool apart both exercised


def test_standard_workloads_host(host):
    """The 8- and 12-tool workloads over their whole spaces in every mode; head, middle and tail
    ranges of the 16-tool one."""
    for cfg in (0, 1):
        scn = S.config(cfg)
        for mode in (0, 1):
            _same(host, scn, 0, 3 ** scn.n, mode)
    scn = S.config2()
    total = 3 ** scn.n
    for first in (0, total // 2 - 1000, total - 60_001):
        _same(host, scn, first, 60_001, 0)


def test_branch_and_bound_host(host):
    """bf_search_pruned's two passes (checkpoint bound, then the survivors' mappings with the
    bound at the inner checkpoint) with incumbents at the optimum, above it and absent: always
    the oracle's optimum, ties to the lowest index."""
    rng = np.random.default_rng(91)
    for t in range(150):
        n = int(rng.integers(1, 10))
        base = S.random_small(rng, n, edge_p=float(rng.choice([0.0, 0.3, 0.6])), tight=bool(t % 3),
                              max_time=int(rng.choice([5, 40, 2000])))
        pred = list(base.pred_mask)
        if t % 3 == 0 and n > 3:
            pred[int(rng.integers(n // 2, n))] = 0
        scn = S.Scenario(n, pred, base.cpu_us, base.gpu_us, base.xfer_us, base.load_us, base.vram_mib,
                         base.vram_budget_mib, base.slowdown_q10)
        want = oracle.search(scn)
        for bound in (want[1], want[1] + int(rng.integers(0, 60)), 0xFFFFFFFF):
            key = host.pruned(scn, bound)
            assert (key & 0xFFFFFFFF, key >> 32) == tuple(want), (t, bound)
    for cfg in (1, 2):
        scn = S.config(cfg)
        want = oracle.search(scn, THREADS)
        key = host.pruned(scn, want[1])
        assert (key & 0xFFFFFFFF, key >> 32) == tuple(want)


def test_tie_order_scenarios_host(host):
    """Queue-heavy tiny DAGs with late sources, some with tied optima whose lowest member differs
    between the canonical and the renumbered order: every mapping in both modes at its
    canonical index, and bf_search_pruned's optimum (ties to the lowest canonical index) from the
    optimum's makespan and from no incumbent."""
    for t, scn in enumerate(tie_order_scenarios()):
        for mode in (0, 1):
            _same(host, scn, 0, 3 ** scn.n, mode)
        want = oracle.search(scn)
        for bound in (want[1], 0xFFFFFFFF):
            key = host.pruned(scn, bound)
            got = (key & 0xFFFFFFFF, key >> 32) if key != 2 ** 64 - 1 else (-1, 0xFFFFFFFF)
            assert got == tuple(want), (t, bound, got, want)


def _same_lanetree(host, scn, lanes, min_roots=0, sampled=False, wide=False):
    got, info = host.lanetree(scn, lanes, min_roots, sampled, wide)
    want, _ = oracle.eval_range(scn, 0, 3 ** scn.n, THREADS)
    bad = np.flatnonzero(got != want)
    assert bad.size == 0, (f"levels x={int(info[0])} y={int(info[1])}, {int(info[2])} blocks: {bad.size} "
                           f"mismatches, first at index {int(bad[0])}: {int(got[bad[0]])} vs {int(want[bad[0]])}")
    return info


def test_lanetree_random_dags(host):
    """The lane-tree batch search (roots, then up to two levels of checkpoints per lane) on random DAGs of
    1-12 tools with small integer times, late sources and last tools that wait for all others: every
    feasible mapping reported once, at its canonical index, with the oracle's makespan; infeasible ones
    never; with 1, 3 and 32 lanes."""
    rng = np.random.default_rng(92)
    levels = set()
    for t in range(200):
        n = int(rng.integers(1, 13)) if t % 5 else int(rng.integers(8, 13))
        base = S.random_small(rng, n, edge_p=float(rng.choice([0.0, 0.25, 0.5, 0.8])), tight=bool(t % 3),
                              contention=bool(t % 4), max_time=int(rng.choice([3, 7, 40, 2000])))
        pred = list(base.pred_mask)
        if t % 3 == 0 and n > 3:
            pred[int(rng.integers(n // 2, n))] = 0
        if t % 4 == 1 and n > 2:
            pred[n - 1] = (1 << (n - 1)) - 1
        scn = S.Scenario(n, pred, base.cpu_us, base.gpu_us, base.xfer_us, base.load_us, base.vram_mib,
                         base.vram_budget_mib, base.slowdown_q10)
        info = _same_lanetree(host, scn, (1, 3, 32)[t % 3])
        levels.add(1 + (int(info[0]) < n) + (int(info[1]) < n))
    assert levels == {1, 2, 3}, levels


def test_lanetree_workloads_and_ties(host):
    """The 8- and 12-tool workloads (the latter over several blocks), the first 48 scenarios of the
    4096-scenario batch workload and the tie-order scenarios: every mapping against the oracle."""
    for cfg in (0, 1):
        info = _same_lanetree(host, S.config(cfg), 32)
    assert int(info[2]) > 1  # the 12-tool workload's roots span several blocks
    for scn in S.config4(48):
        _same_lanetree(host, scn, 32)
    for scn in tie_order_scenarios():
        _same_lanetree(host, scn, 3)


def test_lanetree_whole_space_records(host):
    """The one-scenario lane-tree search (three 6-bit table chunks, roots of up to 16 tools, levels for
    a given number of roots, from the closed-form or the sampled estimate) on random DAGs of 10-14 tools -- queued tools numbered up to 13, late
    sources, last tools that wait for all others -- and on the 16-tool layered workload's first 13
    tools: every mapping against the oracle, with roots from 3^(n-8) up to the whole space."""
    rng = np.random.default_rng(93)
    xs = set()
    for t in range(24):
        n = int(rng.integers(10, 13)) if t % 6 else 14
        base = S.random_small(rng, n, edge_p=float(rng.choice([0.0, 0.25, 0.5])), tight=bool(t % 3),
                              contention=bool(t % 4), max_time=int(rng.choice([3, 7, 40, 2000])))
        pred = list(base.pred_mask)
        if t % 3 == 0:
            pred[int(rng.integers(n // 2, n))] = 0
        if t % 4 == 1:
            pred[n - 1] = (1 << (n - 1)) - 1
        scn = S.Scenario(n, pred, base.cpu_us, base.gpu_us, base.xfer_us, base.load_us, base.vram_mib,
                         base.vram_budget_mib, base.slowdown_q10)
        min_roots = 3 ** int(rng.integers(n - 8, n + 1))
        info = _same_lanetree(host, scn, (1, 3, 32)[t % 3], min_roots, sampled=bool(t % 2))
        assert int(info[2]) == 1 and 3 ** int(info[0]) >= min_roots
        xs.add(int(info[0]) == n)
    assert xs == {False, True}
    full = S.config(2)
    m = 13
    cut = S.Scenario(m, [p & ((1 << m) - 1) for p in full.pred_mask[:m]], full.cpu_us[:m], full.gpu_us[:m],
                     full.xfer_us[:m], full.load_us[:m], full.vram_mib[:m], full.vram_budget_mib,
                     full.slowdown_q10)
    info = _same_lanetree(host, cut, 32, 3 ** 10, sampled=True)
    assert int(info[0]) >= 10 and int(info[1]) < m


def test_lanetree_wide_queue_form(host):
    """The wide form of the one-scenario lane tree (four table chunks, 5-bit queue entries in two words,
    eleven state words per checkpoint), run at small sizes so that every mapping is checked: random DAGs
    of 8-13 tools with small integer times, and 13 tools without edges whose all-queue mapping holds 13
    waiting tools (the second queue word holds the 13th), each against the oracle."""
    rng = np.random.default_rng(94)
    for t in range(16):
        n = int(rng.integers(8, 14))
        base = S.random_small(rng, n, edge_p=float(rng.choice([0.0, 0.2, 0.4])), tight=bool(t % 3),
                              contention=bool(t % 4), max_time=int(rng.choice([3, 7, 40])))
        _same_lanetree(host, base, (1, 3, 32)[t % 3], 3 ** int(rng.integers(n - 6, n)), sampled=bool(t % 2),
                       wide=True)
    for tight in (False, True):
        flat = S.random_small(rng, 13, edge_p=0.0, tight=tight, contention=True, max_time=9)
        assert all(p == 0 for p in flat.pred_mask)
        _same_lanetree(host, flat, 32, 3 ** 9, wide=True)


def test_lanetree_batch_records_of_larger_scenarios(host):
    """The batch's records of scenarios of 13 and 14 tools (the lane-tree batch kernel's three-chunk group; at
    most 1,024 blocks per scenario) and, in the wide form, of 9-12 tools: every mapping against the
    oracle."""
    rng = np.random.default_rng(95)
    for t in range(6):
        n = 13 + t % 2 if t < 4 else int(rng.integers(9, 13))
        base = S.random_small(rng, n, edge_p=float(rng.choice([0.2, 0.35])), tight=bool(t % 3),
                              contention=True, max_time=int(rng.choice([5, 40])))
        info = _same_lanetree(host, base, 32, 0, wide=t >= 4)
        assert int(info[2]) >= 1
