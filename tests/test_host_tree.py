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
import os
import subprocess
import tempfile

import numpy as np
import pytest

import oracle
from paper_2607_22242_gb300 import bf
from paper_2607_22242_gb300 import scenarios as S

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
