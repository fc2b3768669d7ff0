"""Parity of the CUDA search (through the C ABI) with the CPU oracle.

Makespans, feasibility flags and argmin indices must match bit for bit.
Small and mid-size cases are compared element by element with the oracle run
in the test; full-size cases (3^19 mappings, 4096-scenario batch) against the
oracle's results committed in golden/config_results.json, plus sampled
chunks computed by the oracle here.
"""
import json
import os

import numpy as np
import pytest

import oracle
import pins
from batch_cases import mixed_group_batch
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


@pytest.fixture(scope="module")
def golden():
    path = os.path.join(GOLDEN, "config_results.json")
    with open(path) as fh:
        return json.load(fh)["configs"]


def gpu_eval(h, first, count):
    import torch
    ms, fe = bf.eval_mappings(h, first, count)
    torch.cuda.synchronize()
    return ms.cpu().numpy().view(np.uint32).astype(np.uint64), fe.cpu().numpy()


def assert_same(h, scn, first, count):
    g_ms, g_fe = gpu_eval(h, first, count)
    o_ms, o_fe = oracle.eval_range(scn, first, count, THREADS)
    bad = np.flatnonzero((g_ms != o_ms) | (g_fe != o_fe))
    assert bad.size == 0, (f"{bad.size} mismatches, first at index {first + int(bad[0])}: "
                           f"gpu {int(g_ms[bad[0]])}/{int(g_fe[bad[0]])} oracle {int(o_ms[bad[0]])}/{int(o_fe[bad[0]])}")


# --------------------------------------------------------------------------- small cases

def test_hand_examples():
    for ex in pins._load("hand_examples.json")["examples"]:
        scn = S.Scenario.from_dict(ex["scenario"])
        with bf.create_scenario(scn) as h:
            ms, fe = gpu_eval(h, 0, 3 ** scn.n)
            for idx, want in ex["expected"].items():
                assert int(ms[int(idx)]) == want, (ex["name"], idx)
                assert bool(fe[int(idx)]) == (want != INF)
            if "argmin" in ex:
                r = bf.search_best(h)
                assert [r.index, r.makespan_us] == ex["argmin"], ex["name"]


@pytest.mark.parametrize("seed", range(6))
def test_random_small_exhaustive(seed):
    """Every mapping of small random DAGs: ties, VRAM-blocked queues, infeasible starts."""
    rng = np.random.default_rng(1000 + seed)
    for t in range(60):
        n = int(rng.integers(1, 8))
        scn = S.random_small(rng, n, edge_p=float(rng.choice([0.0, 0.3, 0.7])), tight=bool(t % 3),
                             contention=bool(t % 5), max_time=int(rng.choice([6, 30, 2000])))
        with bf.create_scenario(scn) as h:
            assert_same(h, scn, 0, 3 ** n)
            r = bf.search_best(h)
        assert (r.index, r.makespan_us) == oracle.search(scn)
        assert r.modes == S.mapping_modes(r.index, n)


@pytest.mark.parametrize("n", [1, 2, 9, 11, 13, 15, 17])
def test_every_bucket_edge(n):
    """Scenarios of several sizes (windows across the compiled widths), realistic magnitudes."""
    rng = np.random.default_rng(50 + n)
    base = S.random_small(rng, n, edge_p=0.3, tight=True, max_time=50)
    scale = lambda v: [x * 997 + 1 for x in v]
    scn = S.Scenario(n, base.pred_mask, scale(base.cpu_us), scale(base.gpu_us), scale(base.xfer_us),
                     scale(base.load_us), [m * 300 for m in base.vram_mib], base.vram_budget_mib * 300,
                     S.slowdown_linear())
    total = 3 ** n
    with bf.create_scenario(scn) as h:
        count = min(total, 200_003)
        assert_same(h, scn, 0, count)
        assert_same(h, scn, total - min(total, 4099), min(total, 4099))
        r = bf.search_best(h)
    if total <= 2_000_000:
        assert (r.index, r.makespan_us) == oracle.search(scn, THREADS)


@pytest.mark.parametrize("n", [5, 6, 8, 9, 10, 12, 14])
def test_last_tool_waiting_for_all(n):
    """A last tool that every other tool precedes: the kernels leave it out of the window when
    that narrows the compiled width, and end it in closed form.  Full space (n <= 12) or head,
    tail and middle ranges element by element, ranges that cut the last tool's modes apart, and
    the exhaustive and branch-and-bound searches, against the oracle."""
    rng = np.random.default_rng(700 + n)
    base = S.random_small(rng, n, edge_p=0.25, tight=bool(n % 2), max_time=60)
    pred = list(base.pred_mask)
    pred[n - 1] = (1 << (n - 1)) - 1
    scn = S.Scenario(n, pred, base.cpu_us, base.gpu_us, base.xfer_us, base.load_us, base.vram_mib,
                     base.vram_budget_mib, base.slowdown_q10)
    total = 3 ** n
    third = 3 ** (n - 1)
    with bf.create_scenario(scn) as h:
        if total <= 600_000:
            assert_same(h, scn, 0, total)
        else:
            for first in (0, total // 2 - 77_777, total - 150_001):
                assert_same(h, scn, first, 150_001)
        for first, count in ((third - 5, 11), (2 * third - 1, 2), (third + 1, third - 2)):
            if count <= 600_000:
                assert_same(h, scn, first, count)
        want = oracle.search(scn, THREADS)
        r = bf.search_best(h)
        assert (r.index, r.makespan_us) == want
        rp = bf.search_pruned(h)
        assert (rp.index, rp.makespan_us) == want


@pytest.mark.parametrize("n", [8, 12])
def test_magnitudes_at_the_validation_bounds(n):
    """Durations near the validated limits: GPU work of almost 2^32 units per tool (the virtual
    clock wraps modulo 2^32 about once per GPU tool), slowdowns up to 64x, CPU times of up to
    a minute, makespans up to about 10^8 microseconds.  Every mapping element by element, and
    every search path, against the oracle's 64-bit arithmetic."""
    rng = np.random.default_rng(900 + n)
    base = S.random_small(rng, n, edge_p=0.3, tight=True, max_time=50)
    big = (1 << 22) - 1
    g = [int(v) for v in rng.integers(big // 2, big // 2 + big // 4, n)]
    x = [int(v) for v in rng.integers(0, big // 8, n)]
    l = [int(v) for v in rng.integers(0, big // 8, n)]
    c = [int(v) for v in rng.integers(1, 300_000_000 // n, n)]
    f = [0, 1024] + [min(65536, 1024 + (65536 - 1024) * (k - 1) // (n - 1)) for k in range(2, 21)]
    scn = S.Scenario(n, base.pred_mask, c, g, x, l, base.vram_mib, base.vram_budget_mib, f)
    bf.validate_desc(scn)
    with bf.create_scenario(scn) as h:
        assert_same(h, scn, 0, 3 ** n)
        want = oracle.search(scn, THREADS)
        for res in (bf.search_best(h), bf.search_pruned(h), bf.search_tree(h, bf.SPACE_FULL, True)[0],
                    bf.search_tree(h, bf.SPACE_FULL, False)[0]):
            assert (res.index, res.makespan_us) == want
        binary = bf.search_tree(h, bf.SPACE_BINARY, True)[0]
        assert (binary.index, binary.makespan_us) == oracle.search_binary(scn, THREADS)


def test_late_sources_renumbered_searches():
    """DAGs with sources late in the scenario's numbering, which the whole-space searches may
    renumber (sources first), with small integer times so that queue ties are frequent: the
    exhaustive search, the branch and bound, the batched search and the tree search (which always
    renumbers; both spaces) against the oracle."""
    rng = np.random.default_rng(31)
    scns = []
    for t in range(160):
        n = int(rng.integers(6, 13))
        base = S.random_small(rng, n, edge_p=float(rng.choice([0.3, 0.5])), tight=bool(t % 2),
                              contention=bool(t % 3), max_time=int(rng.choice([4, 9, 40])))
        pred = list(base.pred_mask)
        for v in rng.choice(np.arange(n // 2, n), size=2, replace=False):
            pred[int(v)] = 0
        scns.append(S.Scenario(n, pred, base.cpu_us, base.gpu_us, base.xfer_us, base.load_us, base.vram_mib,
                               base.vram_budget_mib, base.slowdown_q10))
    want = [oracle.search(scn, THREADS) for scn in scns]
    for scn, w in zip(scns, want):
        with bf.create_scenario(scn) as h:
            r = bf.search_best(h)
            assert (r.index, r.makespan_us) == w, scn
            rp = bf.search_pruned(h)
            assert (rp.index, rp.makespan_us) == w, scn
            rt, _ = bf.search_tree(h, bf.SPACE_FULL, True)
            assert (rt.index, rt.makespan_us) == w, scn
            rb, _ = bf.search_tree(h, bf.SPACE_BINARY, True)
            assert (rb.index, rb.makespan_us) == oracle.search_binary(scn, THREADS), scn
    assert [(r.index, r.makespan_us) for r in bf.search_batch(scns)] == want


def test_lanetree_whole_space_search():
    """Full searches of 10 to 16 tools run the one-scenario lane-tree kernel (every lane of the GPU on
    one scenario's roots, a shared tail of roots, the result written by the last block): random DAGs
    with small integer times (queue ties, VRAM-blocked queues, infeasible starts), late sources and
    last tools that wait for all others, up to 16 tools with queued tools numbered up to 15; each
    searched twice on one handle (every launch resets its state), against the oracle."""
    rng = np.random.default_rng(77)
    for t in range(14):
        n = 10 + t % 7
        base = S.random_small(rng, n, edge_p=float(rng.choice([0.2, 0.35])), tight=bool(t % 3 != 2),
                              contention=bool(t % 4), max_time=int(rng.choice([5, 9, 40])))
        pred = list(base.pred_mask)
        if t % 3 == 0:
            pred[int(rng.integers(n // 2, n))] = 0
        if t % 4 == 1:
            pred[n - 1] = (1 << (n - 1)) - 1
        scn = S.Scenario(n, pred, base.cpu_us, base.gpu_us, base.xfer_us, base.load_us, base.vram_mib,
                         base.vram_budget_mib, base.slowdown_q10)
        want = oracle.search(scn, THREADS)
        with bf.create_scenario(scn) as h:
            for _ in range(2):
                r = bf.search_best(h)
                assert (r.index, r.makespan_us) == want, (t, n)
        assert r.modes == S.mapping_modes(r.index, n)


def test_lanetree_full_queue_of_16():
    """Sixteen tools without edges (every tool is ready at time 0) with small integer times: the
    mapping that queues all of them fills the lane tree's 16-entry queue word, and ties between
    tools ready at the same instant go by index.  Full searches against the oracle, with a loose
    and a tight VRAM budget."""
    rng = np.random.default_rng(16)
    for tight in (False, True):
        base = S.random_small(rng, 16, edge_p=0.0, tight=tight, contention=True, max_time=9)
        assert all(p == 0 for p in base.pred_mask)
        want = oracle.search(base, THREADS)
        with bf.create_scenario(base) as h:
            r = bf.search_best(h)
        assert (r.index, r.makespan_us) == want, tight


def _layered_scn(seed, sizes, budget):
    rng = np.random.default_rng(seed)
    n = sum(sizes)
    c, g, x, m = S._ordinary(rng, n, 2048, 16384)
    pred = S._layered_edges(rng, sizes, 0.4)
    return S.Scenario(n, pred, c, g, x, [S._load_from_vram(v) for v in m], m, budget, S.slowdown_linear(kmax=n))


def test_lanetree_wide_search():
    """Full searches of 17 to 20 tools on the wide form of the one-scenario lane tree (four table chunks,
    5-bit queue entries in two words): a 17-tool layered DAG and 17 tools without edges (all seventeen
    queued at once in the all-queue mapping) against the oracle, and 18- and 20-tool layered DAGs
    against the search kernel run as two half-range searches (range searches always take it)."""
    for scn in (_layered_scn(61, [4, 4, 3, 3, 3], 24576),
                S.random_small(np.random.default_rng(17), 17, edge_p=0.0, tight=True, contention=True, max_time=9)):
        want = oracle.search(scn, THREADS)
        with bf.create_scenario(scn) as h:
            r = bf.search_best(h)
        assert (r.index, r.makespan_us) == want
    for scn in (_layered_scn(62, [4, 4, 4, 3, 3], 32768), _layered_scn(63, [4] * 5, 40960)):
        total = 3 ** scn.n
        with bf.create_scenario(scn) as h:
            r = bf.search_best(h)
            halves = [bf.search_range(h, 0, total // 2), bf.search_range(h, total // 2, total - total // 2)]
        best = min((x.makespan_us, x.index) for x in halves if x.feasible)
        assert (r.index, r.makespan_us) == (best[1], best[0]), scn.n


def test_batch_of_larger_scenarios():
    """Batches run scenarios of 13-16 tools and of 17-20 tools on the lane-tree batch kernel's larger
    forms (three table chunks; four and the wide queue): a batch of layered DAGs of 10 and 13 to 19
    tools, each result equal to that scenario's own full search (itself checked against the oracle)."""
    scns = [_layered_scn(70 + k, sizes, 24576 + 8192 * (k % 2))
            for k, sizes in enumerate([[4, 3, 3], [4, 4, 3, 2], [4, 4, 4, 3], [4, 4, 4, 4], [4, 4, 3, 3, 3],
                                       [4, 4, 4, 4, 3], [3, 3, 4]])]
    assert sorted(s.n for s in scns) == [10, 10, 13, 15, 16, 17, 19]
    want = []
    for scn in scns:
        with bf.create_scenario(scn) as h:
            r = bf.search_best(h)
        want.append((r.index, r.makespan_us))
    assert [(r.index, r.makespan_us) for r in bf.search_batch(scns)] == want


def test_degenerate_budgets_all_paths():
    """Zero VRAM budget (only all-cpu feasible) and maximal contention, through the exhaustive search,
    the batch, the branch and bound and the tree search, against the oracle."""
    rng = np.random.default_rng(2222)
    scns = []
    for _ in range(12):
        n = int(rng.integers(2, 9))
        base = S.random_small(rng, n, max_time=300)
        scns.append(S.Scenario(**{**base.to_dict(), "vram_budget_mib": 0}))
        scns.append(S.Scenario(**{**base.to_dict(), "vram_budget_mib": sum(base.vram_mib),
                                  "slowdown_q10": [0, 1024] + [65536] * (len(base.slowdown_q10) - 2)}))
    batch = bf.search_batch(scns)
    for scn, rb in zip(scns, batch):
        want = oracle.search(scn)
        with bf.create_scenario(scn) as h:
            assert_same(h, scn, 0, 3 ** scn.n)
            for r in (bf.search_best(h), bf.search_pruned(h), rb, bf.search_tree(h)[0]):
                assert (r.index, r.makespan_us) == want, (scn, r, want)
        if scn.vram_budget_mib == 0:
            assert want[0] == 0


# --------------------------------------------------------------------------- standard workloads

@pytest.mark.parametrize("cfg", [0, 1, 2])
def test_config_full_arrays(cfg, golden):
    scn = S.config(cfg)
    assert S.sha256_of([scn]) == golden[str(cfg)]["sha256"]
    with bf.create_scenario(scn) as h:
        assert_same(h, scn, 0, 3 ** scn.n)
        r = bf.search_best(h)
    g = golden[str(cfg)]["summary"]
    assert (r.index, r.makespan_us, r.feasible) == (g["best_index"], g["best_makespan"], True)


def test_config3_argmin(golden):
    """The full 3^19 search in the benchmark's launch configuration."""
    scn = S.config3()
    assert S.sha256_of([scn]) == golden["3"]["sha256"]
    g = golden["3"]["summary"]
    with bf.create_scenario(scn) as h:
        for _ in range(2):
            r = bf.search_best(h)
            assert (r.index, r.makespan_us, r.feasible) == (g["best_index"], g["best_makespan"], True)
        assert oracle.evaluate(scn, r.index) == r.makespan_us


def test_config3_sampled_chunks():
    scn = S.config3()
    total = 3 ** scn.n
    rng = np.random.default_rng(7)
    starts = [0, total - 70_001] + [int(v) for v in rng.integers(0, total - 70_001, 10)]
    with bf.create_scenario(scn) as h:
        for s in starts:
            assert_same(h, scn, s, 70_001)


def test_config3_full_stream_summary(golden):
    """Every makespan of the 3^19 stream, compared through the oracle's summary."""
    import torch
    scn = S.config3()
    total = 3 ** scn.n
    g = golden["3"]["summary"]
    # torch's int64 products wrap modulo 2^64 like the oracle's uint64: check on a sample first.
    sample = np.random.default_rng(3).integers(0, 2 ** 32, 1000, dtype=np.uint64)
    t = torch.from_numpy(sample.astype(np.int64)).cuda()
    idx = torch.arange(5, 1005, dtype=torch.int64, device="cuda")
    th = int((t * (idx * 2654435761 + 1)).sum().item()) & (2 ** 64 - 1)
    assert th == oracle.stream_hash(sample, 5)
    piece = 1 << 27
    feasible = ms_sum = hsum = 0
    with bf.create_scenario(scn) as h:
        ms = torch.empty(piece, dtype=torch.int32, device="cuda")
        fe = torch.empty(piece, dtype=torch.uint8, device="cuda")
        for first in range(0, total, piece):
            cnt = min(piece, total - first)
            bf.eval_mappings(h, first, cnt, ms, fe)
            m64 = ms[:cnt].to(torch.int64) & 0xFFFFFFFF
            f = fe[:cnt].to(torch.bool)
            feasible += int(f.sum().item())
            ms_sum += int(m64[f].sum().item())
            idx = torch.arange(first, first + cnt, dtype=torch.int64, device="cuda")
            hsum += int((m64 * (idx * 2654435761 + 1)).sum().item())
    assert feasible == g["feasible"]
    assert ms_sum == g["makespan_sum"]
    assert hsum & (2 ** 64 - 1) == g["hash"]


def test_config4_batch(golden):
    batch = S.config4()
    assert S.sha256_of(batch) == golden["4"]["sha256"]
    res = bf.search_batch(batch)
    want_i, want_m = golden["4"]["best_index"], golden["4"]["best_makespan"]
    bad = [i for i, r in enumerate(res) if (r.index, r.makespan_us, r.feasible) != (want_i[i], want_m[i], True)]
    assert not bad, f"{len(bad)} scenarios differ, first {bad[0]}: {res[bad[0]]} vs {(want_i[bad[0]], want_m[bad[0]])}"


def test_batch_mixed_sizes():
    rng = np.random.default_rng(77)
    scns = [S.random_small(rng, int(rng.integers(1, 9)), max_time=int(rng.choice([8, 500]))) for _ in range(40)]
    res = bf.search_batch(scns)
    o_i, o_m = oracle.search_batch(scns, THREADS)
    assert [(r.index, r.makespan_us) for r in res] == list(zip(o_i.tolist(), o_m.tolist()))


# --------------------------------------------------------------------------- ranges and edge cases

def test_search_ranges_compose():
    scn = S.config2()
    total = 3 ** scn.n
    cuts = [0, 1, 12345, 3 ** 10, 20_000_000, total - 1, total]
    with bf.create_scenario(scn) as h:
        parts = [bf.search_range(h, a, b - a) for a, b in zip(cuts, cuts[1:])]
        full = bf.search_best(h)
    best = min((p.makespan_us, p.index) for p in parts if p.feasible)
    assert best == (full.makespan_us, full.index)
    for (a, b), p in zip(zip(cuts, cuts[1:]), parts):
        if b - a <= 2_000_000:
            oi, om = oracle.search_range(scn, a, b - a, THREADS)
            assert (p.index, p.makespan_us) == ((oi, om) if oi >= 0 else (a, INF))


def test_n20_sampled():
    rng = np.random.default_rng(20)
    base = S.random_small(rng, 20, edge_p=0.15, tight=True, max_time=60)
    scn = S.Scenario(20, base.pred_mask, [c * 1000 for c in base.cpu_us], [g * 1000 for g in base.gpu_us],
                     [x * 1000 for x in base.xfer_us], [l * 1000 for l in base.load_us],
                     [m * 1000 for m in base.vram_mib], base.vram_budget_mib * 1000, S.slowdown_linear())
    total = 3 ** 20
    with bf.create_scenario(scn) as h:
        for first in (0, total // 3, total - 50_000):
            assert_same(h, scn, first, 50_000)
        r = bf.search_range(h, total - 1_000_000, 1_000_000)
    oi, om = oracle.search_range(scn, total - 1_000_000, 1_000_000, THREADS)
    assert (r.index, r.makespan_us, r.feasible) == ((oi, om, True) if oi >= 0 else (total - 1_000_000, INF, False))


def test_all_infeasible_range():
    # a single tool larger than the budget: only the cpu mapping is feasible
    scn = S.Scenario(1, [0], [50], [5], [0], [0], [10], 5, S.slowdown_flat())
    with bf.create_scenario(scn) as h:
        r = bf.search_range(h, 1, 2)
        assert not r.feasible and r.makespan_us == INF and r.index == 1
        r = bf.search_best(h)
        assert (r.index, r.makespan_us, r.feasible) == (0, 50, True)
        r = bf.search_range(h, 0, 0)
        assert not r.feasible


def test_range_errors():
    scn = S.config0()
    lib = bf.load()
    with bf.create_scenario(scn) as h:
        for first, count in ((0, 3 ** 8 + 1), (3 ** 8, 1), (3 ** 8 + 1, 0), (2 ** 63, 2 ** 63), (1, 2 ** 64 - 1)):
            with pytest.raises(bf.BfError) as ei:
                bf.search_range(h, first, count)
            assert ei.value.code == bf.BF_ERANGE
            # the range is checked before the output pointers
            assert lib.bf_eval_mappings(h.ptr, first, count, None, None, None) == bf.BF_ERANGE
        bf.eval_mappings(h, 3 ** 8, 0)  # empty range at the end is fine


def test_ragged_eval_ranges():
    scn = S.config1()
    with bf.create_scenario(scn) as h:
        for first, count in ((1, 255), (255, 257), (100_000, 1), (3 ** 12 - 513, 513), (7, 33_333)):
            assert_same(h, scn, first, count)


def test_non_default_stream():
    import torch
    scn = S.config1()
    s = torch.cuda.Stream()
    with bf.create_scenario(scn) as h:
        with torch.cuda.stream(s):
            r = bf.search_best(h, stream=s)
            ms, fe = bf.eval_mappings(h, 0, 3 ** 12, stream=s)
        s.synchronize()
    assert (r.index, r.makespan_us) == oracle.search(scn, THREADS)
    o_ms, _ = oracle.eval_range(scn, 0, 3 ** 12, THREADS)
    assert np.array_equal(ms.cpu().numpy().view(np.uint32).astype(np.uint64), o_ms)


def test_concurrent_handles_on_host_threads(golden):
    """Calls on different handles may run at once: five host threads, each with its own handle
    (or batch) and its own CUDA stream, repeat full searches, a tree search and a batched search
    concurrently; every result equals the stored oracle optimum."""
    import threading
    import torch
    with open(os.path.join(GOLDEN, "wide_results.json")) as fh:
        wide = json.load(fh)["workloads"]["wide28"]
    batch = S.config4(256)
    want_batch = [(i, m) for i, m in zip(golden["4"]["best_index"][:256], golden["4"]["best_makespan"][:256])]

    def full(cfg):
        g = golden[str(cfg)]["summary"]
        return lambda h, st: (bf.search_best(h, st), (g["best_index"], g["best_makespan"]))

    jobs = [(S.config0(), full(0)), (S.config1(), full(1)), (S.config2(), full(2)),
            (S.wide28(), lambda h, st: (bf.search_tree(h, bf.SPACE_FULL, True, None, st)[0], tuple(wide["ternary"]))),
            (None, None)]
    errors = []

    def worker(scn, call):
        try:
            torch.cuda.set_device(0)
            st = torch.cuda.Stream()
            if scn is None:
                for _ in range(4):
                    got = [(r.index, r.makespan_us) for r in bf.search_batch(batch, st)]
                    if got != want_batch:
                        errors.append("batch")
                return
            with bf.create_scenario(scn) as h:
                for _ in range(4):
                    res, want = call(h, st)
                    if (res.index, res.makespan_us) != want:
                        errors.append((scn.n, res.index, res.makespan_us, want))
        except Exception as exc:  # reported below; a thread's exception would otherwise vanish
            errors.append(repr(exc))

    threads = [threading.Thread(target=worker, args=job) for job in jobs]
    for t in threads:
        t.start()
    for t in threads:
        t.join(timeout=300)
    assert not any(t.is_alive() for t in threads)
    assert errors == []


def test_wait_timeout_is_reported():
    """The host wait is bounded: a 1 ms limit on a 16 ms search returns BF_ETIMEOUT, the GPU
    work finishes normally, and the library works afterwards."""
    import torch
    scn = S.config3()
    with bf.create_scenario(scn) as h:
        bf.set_wait_timeout_ms(1)
        try:
            with pytest.raises(bf.BfError) as ei:
                bf.search_best(h)
            assert ei.value.code == bf.BF_ETIMEOUT
        finally:
            bf.set_wait_timeout_ms(600000)
            torch.cuda.synchronize()
        r = bf.search_best(h)
    assert r.feasible


def test_pipelined_batch_with_both_groups(golden):
    """A batch large enough to be pipelined (its first eighth of lane-tree scenarios launched while the
    rest are built, the rest on a second stream), with 30 random scenarios of 1-14 tools interleaved
    (those of 13 and 14 tools run the lane-tree batch kernel's three-chunk form, also on the second
    stream): every result at its position against the oracle."""
    small = S.config4(1200)
    extra = mixed_group_batch(seed=99, count=30)
    scns, origin = [], []  # origin: index into small, or -1 for an interleaved scenario
    for i, scn in enumerate(small):
        scns.append(scn)
        origin.append(i)
        if i % 40 == 0:
            scns.append(extra[i // 40])
            origin.append(-1)
    assert sum(s.n <= 12 for s in scns) >= 1024 and any(s.n > 12 for s in scns)
    o_i, o_m = oracle.search_batch(extra, THREADS)
    want_extra = iter(zip(o_i.tolist(), o_m.tolist()))
    res = bf.search_batch(scns)
    for pos, (k, r) in enumerate(zip(origin, res)):
        want = (golden["4"]["best_index"][k], golden["4"]["best_makespan"][k]) if k >= 0 else next(want_extra)
        assert (r.index, r.makespan_us) == want, pos


def test_batch_wait_timeout_then_next_call(golden):
    """A batch call whose host wait runs out returns BF_ETIMEOUT; its scratch is freed in stream order
    after its kernels, and the next call on the same stream gives the oracle's optima."""
    import torch
    batch = S.config4(1024)
    want = list(zip(golden["4"]["best_index"][:1024], golden["4"]["best_makespan"][:1024]))
    bf.set_wait_timeout_ms(1)
    try:
        with pytest.raises(bf.BfError) as ei:
            bf.search_batch(batch)
        assert ei.value.code == bf.BF_ETIMEOUT
    finally:
        bf.set_wait_timeout_ms(600000)
    got = [(r.index, r.makespan_us) for r in bf.search_batch(batch)]
    torch.cuda.synchronize()
    assert got == want


def test_shards_combine_to_full_search(golden):
    """The per-rank pieces of a sharded search (shard.gpu_search_range on each
    rank's range), combined by packed key, give the full N=19 optimum."""
    from paper_2607_22242_gb300 import shard
    scn = S.config3()
    total = 3 ** scn.n
    g = golden["3"]["summary"]
    with bf.create_scenario(scn) as h:
        search = shard.gpu_search_range(h)
        for world in (2, 3, 8):
            keys = [shard.pack_key(*search(*shard.shard_range(total, r, world))) for r in range(world)]
            assert shard.unpack_key(min(keys)) == (g["best_index"], g["best_makespan"], True)


def test_batch_shards_combine_to_full_batch(golden):
    """The per-rank blocks of a sharded batch (shard.gpu_search_batch on each rank's block of the
    4096 scenarios), concatenated in rank order, give every scenario's optimum."""
    from paper_2607_22242_gb300 import shard
    batch = S.config4()
    want = [(i, m, True) for i, m in zip(golden["4"]["best_index"], golden["4"]["best_makespan"])]
    search = shard.gpu_search_batch()
    for world in (2, 3, 8):
        got = []
        for r in range(world):
            first, count = shard.shard_range(len(batch), r, world)
            got += search(batch[first:first + count])
        assert got == want, world


# --------------------------------------------------------------------------- what-if and index lists

def _same_probes(got, want):
    return [(p.kind, p.tool, p.mode, p.other, p.index, p.makespan_us, p.feasible) for p in got] == want


def test_whatif_matches_algorithm1_oracle():
    from oracle import whatif as W
    rng = np.random.default_rng(314)
    for t in range(80):
        n = int(rng.integers(1, 9))
        scn = S.random_small(rng, n, tight=bool(t % 2), max_time=int(rng.choice([9, 900])))
        with bf.create_scenario(scn) as h:
            for base in rng.integers(0, 3 ** n, 4):
                assert _same_probes(bf.whatif(h, int(base)), W.whatif(scn, int(base))), (scn, int(base))


def test_whatif_fig7_and_config3():
    from oracle import whatif as W
    f7 = pins._load("paper_fig7.json")
    tools = [dict(cpu_ms=t["cpu"], gpu_ms=t["gpu"], load_ms=t["load"], vram_mb=t["mem"]) for t in f7["tools"]]
    scn = pins._fanout(tools, f7["budget_mb"])
    base = S.mapping_index([1, 1, 2, 0])
    with bf.create_scenario(scn) as h:
        assert _same_probes(bf.whatif(h, base), W.whatif(scn, base))
    scn = S.config3()
    rng = np.random.default_rng(3)
    with bf.create_scenario(scn) as h:
        for base in [575638191, 0, 3 ** 19 - 1] + [int(v) for v in rng.integers(0, 3 ** 19, 5)]:
            got = bf.whatif(h, base)
            assert len(got) <= bf.MAX_PROBES
            assert _same_probes(got, W.whatif(scn, base)), base


def test_eval_indices_matches_oracle():
    import torch
    rng = np.random.default_rng(99)
    for cfg in (1, 2, 3):
        scn = S.config(cfg)
        total = 3 ** scn.n
        idx = rng.integers(0, total, 20_000).astype(np.int64)
        idx[:3] = [0, total - 1, total]          # includes one index past the end
        with bf.create_scenario(scn) as h:
            ms, fe = bf.eval_indices(h, torch.from_numpy(idx).cuda())
            torch.cuda.synchronize()
        ms = ms.cpu().numpy().view(np.uint32)
        fe = fe.cpu().numpy()
        assert fe[2] == 0xFF and ms[2] == INF
        for j in list(range(3)) + [int(v) for v in rng.integers(3, idx.size, 400)]:
            if idx[j] >= total:
                continue
            want = oracle.evaluate(scn, int(idx[j]))
            assert (int(ms[j]), int(fe[j])) == (want, int(want != INF)), (cfg, int(idx[j]))


def test_whatif_range_error():
    scn = S.config0()
    with bf.create_scenario(scn) as h:
        with pytest.raises(bf.BfError) as ei:
            bf.whatif(h, 3 ** 8)
        assert ei.value.code == bf.BF_ERANGE


# --------------------------------------------------------------------------- branch and bound

def test_pruned_search_equals_exhaustive_small():
    rng = np.random.default_rng(2718)
    for t in range(120):
        n = int(rng.integers(1, 10))
        scn = S.random_small(rng, n, edge_p=float(rng.choice([0.0, 0.3, 0.7])), tight=bool(t % 3),
                             max_time=int(rng.choice([6, 30, 2000])))
        want = oracle.search(scn)
        with bf.create_scenario(scn) as h:
            for hint in (None, int(rng.integers(0, 3 ** n)), want[0]):
                r = bf.search_pruned(h, hint)
                assert (r.index, r.makespan_us, r.feasible) == (want[0], want[1], True), (scn, hint)


@pytest.mark.parametrize("cfg", [0, 1, 2, 3])
def test_pruned_search_standard_workloads(cfg, golden):
    scn = S.config(cfg)
    g = golden[str(cfg)]["summary"]
    with bf.create_scenario(scn) as h:
        for hint in (None, 0, g["best_index"]):
            r = bf.search_pruned(h, hint)
            assert (r.index, r.makespan_us, r.feasible) == (g["best_index"], g["best_makespan"], True)


def test_pruned_search_batch_scenarios(golden):
    batch = S.config4(64)
    want_i, want_m = golden["4"]["best_index"], golden["4"]["best_makespan"]
    for k, scn in enumerate(batch):
        with bf.create_scenario(scn) as h:
            r = bf.search_pruned(h)
        assert (r.index, r.makespan_us) == (want_i[k], want_m[k]), k


# --------------------------------------------------------------------------- the batch's two groups

def test_batch_two_groups():
    """Scenarios of up to 12 tools interleaved with scenarios of 13 and 14 tools (the lane-tree batch
    kernel's two- and three-chunk groups) in one call: every result at its position, equal to the
    oracle's."""
    scns = mixed_group_batch()
    assert {s.n > 12 for s in scns} == {True, False}
    o_i, o_m = oracle.search_batch(scns, THREADS)
    res = bf.search_batch(scns)
    assert [(r.index, r.makespan_us) for r in res] == list(zip(o_i.tolist(), o_m.tolist()))


@pytest.mark.parametrize("which", ["fanout12", "layered13"])
def test_search_launch_state_across_calls(which):
    """A search call is one launch whose last block writes the result to the handle's host mirror and
    resets the launch state: every kind of search, and empty and partial ranges, on one handle and on
    two streams in turn, must each give the oracle's answer.  The 12-tool workload runs its full
    search on the search kernel; the 16-tool workload's first 13 tools run theirs on the lane-tree
    kernel, which shares the launch state with the range searches of the same handle."""
    import torch
    if which == "fanout12":
        scn = S.config1()
    else:
        full, m = S.config2(), 13
        scn = S.Scenario(m, [p & ((1 << m) - 1) for p in full.pred_mask[:m]], full.cpu_us[:m], full.gpu_us[:m],
                         full.xfer_us[:m], full.load_us[:m], full.vram_mib[:m], full.vram_budget_mib,
                         full.slowdown_q10)
    total = 3 ** scn.n
    want = oracle.search(scn, THREADS)
    part = (total // 3, total // 5)
    want_part = oracle.search_range(scn, part[0], part[1], THREADS)
    streams = [torch.cuda.current_stream(), torch.cuda.Stream()]
    with bf.create_scenario(scn) as h:
        for k in range(3):
            st = streams[k % 2]
            r = bf.search_best(h, st)
            assert (r.index, r.makespan_us) == want
            empty = bf.search_range(h, 17, 0, st)
            assert not empty.feasible and empty.index == 17
            r = bf.search_range(h, part[0], part[1], st)
            assert (r.index, r.makespan_us) == want_part
            r = bf.search_best(h, st)
            assert (r.index, r.makespan_us) == want
            r = bf.search_pruned(h, None, st)
            assert (r.index, r.makespan_us) == want
            rt, _ = bf.search_tree(h, bf.SPACE_FULL, True, None, st)
            assert (rt.index, rt.makespan_us) == want
            streams[1 - k % 2].wait_stream(st)
