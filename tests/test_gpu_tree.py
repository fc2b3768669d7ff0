"""Parity of the tree search (bf_search_tree) and of the 32-slot index lists with the CPU oracle.

The tree search must return exactly the oracle's optimum -- lowest makespan,
ties to the lowest index -- of the full space or the binary cpu/gpu_now space,
with and without pruning.  Up to 10 tools the oracle enumerates every mapping
in the test; beyond 20 tools the reference is the segment rule
(oracle.segments, pinned against full enumeration) on DAGs with serialisation
points, or the oracle's full enumeration of a binary space stored in
golden/wide_results.json.
"""
import json
import os

import numpy as np
import pytest

import oracle
from oracle import segments
from paper_2607_22242_gb300 import bf
from paper_2607_22242_gb300 import scenarios as S

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
INF = 0xFFFFFFFF
THREADS = oracle.default_threads()


@pytest.fixture(scope="module", autouse=True)
def cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)
    return torch


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as fh:
        return json.load(fh)


def _pair(res):
    return (res.index, res.makespan_us) if res.feasible else (-1, INF)


def test_tree_matches_oracle_small():
    """Every mode of the search against full enumeration on random DAGs of 1..10 tools."""
    rng = np.random.default_rng(2024)
    for t in range(120):
        n = int(rng.integers(1, 11))
        scn = S.random_small(rng, n, edge_p=float(rng.choice([0.0, 0.3, 0.6])), tight=bool(t % 3),
                             contention=bool(t % 4), max_time=int(rng.choice([7, 40, 3000])))
        full = oracle.search(scn, THREADS)
        binary = oracle.search_binary(scn, THREADS)
        with bf.create_scenario(scn) as h:
            for space, want in ((bf.SPACE_FULL, full), (bf.SPACE_BINARY, binary)):
                for prune in (True, False):
                    res, st = bf.search_tree(h, space, prune)
                    assert _pair(res) == want, (t, scn, space, prune, res, want)
                    assert st["leaves"] <= space ** n, st
            # a hint (the optimum itself, or one outside the binary space) changes nothing
            res, _ = bf.search_tree(h, bf.SPACE_FULL, True, hint_index=full[0])
            assert _pair(res) == full
            res, _ = bf.search_tree(h, bf.SPACE_BINARY, True, hint_index=2 * 3 ** (n - 1))
            assert _pair(res) == binary


def test_tree_matches_standard_workloads():
    """The stored brute-force optima of the 8-, 12-, 16- and 19-tool workloads."""
    g = _golden("config_results.json")["configs"]
    for cfg in range(4):
        scn = S.config(cfg)
        want = (g[str(cfg)]["summary"]["best_index"], g[str(cfg)]["summary"]["best_makespan"])
        res, st = bf.search_tree(scn, bf.SPACE_FULL, True)
        assert _pair(res) == want, (cfg, res, st)
        assert st["leaves"] < 3 ** scn.n or scn.n <= 8


def test_tree_agrees_with_exhaustive_kernels():
    """Full enumeration through the tree (no pruning) and the enumerating search, random DAGs up to 14 tools."""
    rng = np.random.default_rng(77)
    for t in range(12):
        n = int(rng.integers(11, 15))
        scn = S.random_small(rng, n, edge_p=0.25, tight=bool(t % 2), max_time=int(rng.choice([30, 3000])))
        with bf.create_scenario(scn) as h:
            want = _pair(bf.search_best(h))
            for prune in (True, False):
                res, _ = bf.search_tree(h, bf.SPACE_FULL, prune)
                assert _pair(res) == want, (t, scn, prune)


def test_tree_segmented_beyond_20_tools():
    """Random segmented DAGs of 21..32 tools: both spaces against the segment rule."""
    rng = np.random.default_rng(4242)
    for t in range(16):
        n = int(rng.integers(21, 33))
        scn = S.random_segmented(rng, n, seg_max=int(rng.choice([4, 6, 8])), tight=bool(t % 2),
                                 max_time=int(rng.choice([20, 2000])))
        with bf.create_scenario(scn) as h:
            for space, binary in ((bf.SPACE_FULL, False), (bf.SPACE_BINARY, True)):
                want = segments.search(scn, binary=binary, threads=THREADS)
                res, st = bf.search_tree(h, space, True)
                assert _pair(res) == want, (t, n, space, res, st, want)
                assert segments.evaluate(scn, res.index) == res.makespan_us


@pytest.mark.parametrize("name", ["wide28", "wide32"])
def test_tree_wide_workloads(name):
    g = _golden("wide_results.json")["workloads"][name]
    scn = getattr(S, name)()
    assert S.sha256_of([scn]) == g["sha256"]
    with bf.create_scenario(scn) as h:
        for space, key in ((bf.SPACE_FULL, "ternary"), (bf.SPACE_BINARY, "binary")):
            res, st = bf.search_tree(h, space, True)
            assert _pair(res) == tuple(g[key]), (name, space, res, st)
            assert res.modes == S.mapping_modes(res.index, scn.n)


def test_tree_full_enumeration_of_32_tool_binary_space():
    """Every binary mapping of the 32-tool workload (2^32, less those under infeasible prefixes)
    simulated: the same optimum as the pruned search."""
    g = _golden("wide_results.json")["workloads"]["wide32"]
    res, st = bf.search_tree(S.wide32(), bf.SPACE_BINARY, False)
    assert _pair(res) == tuple(g["binary"])
    assert 2 ** 31 < st["leaves"] <= 2 ** 32, st


def test_tree_layered24_binary():
    """No serialisation point: the oracle's full enumeration of 2^24 binary mappings."""
    g = _golden("wide_results.json")["workloads"]["layered24"]
    scn = S.layered24()
    assert S.sha256_of([scn]) == g["sha256"]
    with bf.create_scenario(scn) as h:
        for prune in (True, False):
            res, st = bf.search_tree(h, bf.SPACE_BINARY, prune)
            assert _pair(res) == tuple(g["binary"]), (prune, res, st)


def test_tree_21_tools_without_cut_points():
    """A 21-tool layered DAG with no serialisation point: the pruned full-space search equals the
    unpruned one (every one of the 3^21 mappings simulated), and the binary space equals the
    oracle's full enumeration of its 2^21 mappings."""
    rng = np.random.default_rng(21)
    c, g, x, m = S._ordinary(rng, 21, 2048, 16384)
    pred = S._layered_edges(rng, [4, 4, 4, 4, 5], 0.4)
    scn = S.Scenario(21, pred, c, g, x, [40 * v for v in m], m, 40960, S.slowdown_linear(kmax=21))
    assert segments.bounds(scn) == [(0, 21)]
    with bf.create_scenario(scn) as h:
        pruned, _ = bf.search_tree(h, bf.SPACE_FULL, True)
        full, st = bf.search_tree(h, bf.SPACE_FULL, False)
        assert _pair(pruned) == _pair(full), (pruned, full)
        assert st["leaves"] <= 3 ** 21
        assert oracle.evaluate(scn, pruned.index) == pruned.makespan_us
        binary, _ = bf.search_tree(h, bf.SPACE_BINARY, True)
        assert _pair(binary) == oracle.search_binary(scn, THREADS)


def test_wide_eval_indices_and_whatif_match_oracle():
    """The 32-slot index-list kernel: random mappings of the 28- and 32-tool workloads, and the what-if probes."""
    import torch
    from oracle import whatif as W
    rng = np.random.default_rng(5)
    for name in ("wide28", "wide32"):
        scn = getattr(S, name)()
        total = 3 ** scn.n
        idx = [int(v) % total for v in rng.integers(0, 2 ** 62, 3000)] + [0, total - 1, total]
        with bf.create_scenario(scn) as h:
            ms, fe = bf.eval_indices(h, torch.tensor(idx, dtype=torch.int64, device="cuda"))
            ms = [int(v) & 0xFFFFFFFF for v in ms.cpu().tolist()]
            fe = fe.cpu().tolist()
            for j, x in enumerate(idx[:-1]):
                want = oracle.evaluate(scn, x)
                assert (ms[j], fe[j]) == (want, int(want != INF)), (name, x)
            assert (ms[-1], fe[-1]) == (INF, 0xFF)
            best = _golden("wide_results.json")["workloads"][name]["ternary"][0]
            for base in (best, 0, int(idx[7])):
                got = [(p.kind, p.tool, p.mode, p.other, p.index, p.makespan_us, p.feasible)
                       for p in bf.whatif(h, base)]
                assert got == W.whatif(scn, base), (name, base)


def test_empty_and_single_inputs():
    """Empty index lists and batches, and one-tool scenarios, on every path that takes them."""
    import torch
    one = S.Scenario(1, [0], [50], [5], [3], [4], [10], 20, S.slowdown_flat())
    with bf.create_scenario(one) as h:
        ms, fe = bf.eval_indices(h, torch.empty(0, dtype=torch.int64, device="cuda"))
        assert ms.numel() == 0 and fe.numel() == 0
        want = oracle.search(one)
        assert _pair(bf.search_best(h)) == want == (1, 8)
        assert _pair(bf.search_pruned(h)) == want
        for space in (bf.SPACE_FULL, bf.SPACE_BINARY):
            for prune in (True, False):
                assert _pair(bf.search_tree(h, space, prune)[0]) == want
        assert [p.index for p in bf.whatif(h, 0)] == [1, 2]
    assert bf.search_batch([]) == [] and bf.search_batch_noalloc([]) == []


def test_tree_argument_errors():
    scn = S.config0()
    with bf.create_scenario(scn) as h:
        with pytest.raises(bf.BfError) as ei:
            bf.search_tree(h, 4, True)
        assert ei.value.code == bf.BF_EINVAL
        r = bf.CResult()
        st = bf.CTreeStats()
        import ctypes
        assert bf.load().bf_search_tree(h.ptr, 3, 2, 0, ctypes.byref(r), ctypes.byref(st), None) == bf.BF_EINVAL
        assert bf.load().bf_search_tree(h.ptr, 3, 0, 0, None, None, None) == bf.BF_EINVAL
    wide = S.wide28()
    with bf.create_scenario(wide) as h:
        for call in (lambda: bf.search_best(h), lambda: bf.search_range(h, 0, 10), lambda: bf.search_pruned(h),
                     lambda: bf.eval_mappings(h, 0, 10)):
            with pytest.raises(bf.BfError) as ei:
                call()
            assert ei.value.code == bf.BF_EINVAL and "n <= 20" in ei.value.message


def test_tree_search_time_limit():
    """A search that would run for hours (every one of the 3^28 mappings of the 28-tool workload,
    no pruning) returns BF_ETIMEOUT once the wait limit has passed, and the library works
    afterwards."""
    import time
    import torch
    scn = S.wide28()
    bf.set_wait_timeout_ms(300)
    try:
        with bf.create_scenario(scn) as h:
            t = time.time()
            with pytest.raises(bf.BfError) as ei:
                bf.search_tree(h, bf.SPACE_FULL, False)
            assert ei.value.code == bf.BF_ETIMEOUT, ei.value.message
            assert time.time() - t < 30
            torch.cuda.synchronize()  # the last steps are still in flight
    finally:
        bf.set_wait_timeout_ms(600000)
        torch.cuda.synchronize()
    want = _golden("wide_results.json")["workloads"]["wide28"]["ternary"]
    res, _ = bf.search_tree(scn, bf.SPACE_FULL, True)
    assert _pair(res) == tuple(want)


def test_tie_order_scenarios_every_search():
    """Queue-heavy tiny DAGs with late sources, among them tied optima whose lowest member differs
    between the sources-first order the searches may run in and the canonical order (the first is
    scenario 91): the tree search in both spaces, pruned and unpruned, the exhaustive search, the
    branch and bound and the batched search (lane-tree kernel) must all return the lowest
    canonical index among the oracle's optima."""
    from tie_cases import tie_order_scenarios
    scns = tie_order_scenarios()
    want = [oracle.search(s) for s in scns]
    for t, (scn, w) in enumerate(zip(scns, want)):
        binary = oracle.search_binary(scn)
        with bf.create_scenario(scn) as h:
            for prune in (True, False):
                assert _pair(bf.search_tree(h, bf.SPACE_FULL, prune)[0]) == w, (t, prune)
                assert _pair(bf.search_tree(h, bf.SPACE_BINARY, prune)[0]) == binary, (t, prune)
            assert _pair(bf.search_best(h)) == w, t
            assert _pair(bf.search_pruned(h)) == w, t
    assert [_pair(r) for r in bf.search_batch(scns)] == want
