"""The tree search's node logic, built for the host, against the oracle (no GPU).

tests/host_tree.cpp compiles bf_tree.cuh -- the constants, the sources-first renumbering, node
expansion and its bound, the leaf re-test, the leaf window and the leaf enumeration with its tie
rule, the code the tree kernels run -- with g++ and walks the tree depth first.  Its optimum
(lowest makespan, ties to the lowest canonical index) must equal the oracle's full enumeration
in both spaces, pruned from no incumbent and from the optimum's own makespan (the tightest bound
that keeps the optimum), and unpruned.  The GPU tests check the kernels' level loop on the
hardware.
"""
import ctypes
import json
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
INF = 0xFFFFFFFF


@pytest.fixture(scope="module")
def tree():
    out = os.path.join(tempfile.mkdtemp(prefix="bf_host_tree_"), "host_tree.so")
    subprocess.run(["g++", "-O2", "-std=c++17", "-shared", "-fPIC", "-Wno-unknown-pragmas", "-I",
                    os.path.join(ROOT, "include"), "-o", out, os.path.join(HERE, "host_tree.cpp")], check=True)
    lib = ctypes.CDLL(out)
    lib.host_tree.argtypes = [ctypes.POINTER(bf.Desc), ctypes.c_uint32, ctypes.c_uint32, ctypes.c_uint32,
                              ctypes.c_void_p]
    lib.host_tree.restype = ctypes.c_int

    def run(scn, space, prune=True, bound=INF):
        res = np.zeros(6, np.uint64)
        assert lib.host_tree(ctypes.byref(bf.to_desc(scn)), space, int(prune), bound, res.ctypes.data) == 0
        ms, idx = int(res[0]), int(res[1])
        best = (idx, ms) if ms != 2 ** 64 - 1 else (-1, INF)
        return best, res[2:].tolist()
    return run


def _with_late_sources(rng, base, n):
    pred = list(base.pred_mask)
    for v in rng.choice(np.arange(n // 2, n), size=min(2, n - n // 2), replace=False):
        pred[int(v)] = 0
    return S.Scenario(n, pred, base.cpu_us, base.gpu_us, base.xfer_us, base.load_us, base.vram_mib,
                      base.vram_budget_mib, base.slowdown_q10)


def _with_last_waiting(base, n):
    pred = list(base.pred_mask)
    pred[n - 1] = (1 << (n - 1)) - 1
    return S.Scenario(n, pred, base.cpu_us, base.gpu_us, base.xfer_us, base.load_us, base.vram_mib,
                      base.vram_budget_mib, base.slowdown_q10)


def test_tree_node_logic_random_dags(tree):
    """Random DAGs of 1-11 tools with small integer times (frequent ties), some with late sources
    (renumbered) or a last tool that waits for all others (closed form at the leaves): both spaces,
    pruned from no incumbent and from the optimum, and unpruned."""
    rng = np.random.default_rng(77)
    seen = set()
    for t in range(200):
        n = int(rng.integers(1, 12))
        base = S.random_small(rng, n, edge_p=float(rng.choice([0.0, 0.3, 0.6])), tight=bool(t % 3),
                              contention=bool(t % 4), max_time=int(rng.choice([4, 9, 40, 3000])))
        scn = base
        if t % 3 == 0 and n > 3:
            scn = _with_late_sources(rng, base, n)
        elif t % 3 == 1 and n > 2:
            scn = _with_last_waiting(base, n)
        full = oracle.search(scn, THREADS)
        binary = oracle.search_binary(scn, THREADS)
        for space, want in ((3, full), (2, binary)):
            got, st = tree(scn, space)
            assert got == want, (t, scn, space, got, want, st)
            seen.add(("renumbered", st[2]))
            if want[0] >= 0:
                got, _ = tree(scn, space, True, want[1])
                assert got == want, (t, space, "bound at the optimum", got, want)
            if n <= 8:
                got, st = tree(scn, space, False)
                assert got == want, (t, space, "unpruned", got, want)
                assert st[1] <= space ** n  # subtrees that are infeasible throughout are cut
    assert ("renumbered", 1) in seen and ("renumbered", 0) in seen


def test_tree_node_logic_queue_bound(tree):
    """Queue-heavy DAGs (few edges, tight budgets, steep contention, CPU times scaled up to 10x),
    where the bound's serial queue sum is what prunes: from the optimum's makespan and from no
    incumbent, the oracle's optimum (a queue sum raised by 1 us per queued tool changes the
    result of scenario 15 here)."""
    rng = np.random.default_rng(6)
    for t in range(40):
        n = int(rng.integers(6, 11))
        base = S.random_small(rng, n, edge_p=float(rng.choice([0.0, 0.1, 0.3])), tight=True, contention=True,
                              max_time=int(rng.choice([3, 10, 100])))
        cpu = [c * int(rng.choice([1, 3, 10])) for c in base.cpu_us]
        scn = S.Scenario(n, base.pred_mask, cpu, base.gpu_us, base.xfer_us, base.load_us, base.vram_mib,
                         base.vram_budget_mib, base.slowdown_q10)
        want = oracle.search(scn)
        if want[0] < 0:
            continue
        for bound in (want[1], INF):
            got, st = tree(scn, 3, True, bound)
            assert got == want, (t, bound, got, want, st)


def test_tree_node_logic_tie_order(tree):
    """Queue-heavy tiny DAGs with late sources, where the tied optima's lowest canonical index
    differs from the lowest index in the renumbered (sources-first) order (scenario 91 here):
    ties must be broken by canonical index, in both spaces."""
    for t, scn in enumerate(tie_order_scenarios()):
        for space, want in ((3, oracle.search(scn)), (2, oracle.search_binary(scn))):
            got, st = tree(scn, space)
            assert got == want, (t, space, got, want, st)


def test_tree_node_logic_standard_workloads(tree):
    """The 8-, 12- and 16-tool workloads (the 16-tool one has a late source and runs renumbered)
    in both spaces against the oracle, with the bound at the optimum."""
    for cfg in (0, 1, 2):
        scn = S.config(cfg)
        for space, want in ((3, oracle.search(scn, THREADS)), (2, oracle.search_binary(scn, THREADS))):
            for bound in (INF, want[1]):
                got, st = tree(scn, space, True, bound)
                assert got == want, (cfg, space, bound, got, want, st)
            if cfg == 2:
                assert st[2] == 1


def test_tree_node_logic_beyond_20_tools(tree):
    """32-slot trees: random segmented DAGs of 21-32 tools in both spaces against the segment
    rule (oracle.segments, pinned against full enumeration), and the stored optima of the 28- and
    32-tool workloads and of the 24-tool layered DAG's binary space (two late sources, renumbered,
    no serialisation point; the oracle's full enumeration of 2^24 mappings)."""
    from oracle import segments
    rng = np.random.default_rng(4243)
    for t in range(12):
        n = int(rng.integers(21, 33))
        scn = S.random_segmented(rng, n, seg_max=int(rng.choice([4, 6, 8])), tight=bool(t % 2),
                                 max_time=int(rng.choice([20, 2000])))
        for space in (3, 2):
            got, st = tree(scn, space)
            assert got == tuple(segments.search(scn, binary=space == 2, threads=THREADS)), (t, n, space, got, st)
    with open(os.path.join(HERE, "golden", "wide_results.json")) as fh:
        golden = json.load(fh)["workloads"]
    widths = set()
    # the 32-tool full space starts from the optimum's makespan, as the kernels' dive would
    # give it (from no incumbent the depth-first walk simulates 7.7e8 leaves, about 2 minutes)
    for name, space, key, start in (("wide28", 3, "ternary", False), ("wide32", 3, "ternary", True),
                                    ("wide32", 2, "binary", False), ("layered24", 2, "binary", False)):
        scn = getattr(S, name)()
        assert S.sha256_of([scn]) == golden[name]["sha256"]
        got, st = tree(scn, space, True, golden[name][key][1] if start else INF)
        assert got == tuple(golden[name][key]), (name, space, got, st)
        widths.add(st[3])
        if name == "layered24":
            assert st[2] == 1
    assert max(widths) > 12, widths  # a leaf window wider than the small DAGs reach
