"""bf_search_batch_noalloc: the batched search for callers that cannot allocate.

Some callers cannot allocate device memory at the moment they search -- their
process has given all GPU memory to another allocator's pool, or a
cudaMalloc/cudaFree pair would synchronise the device inside a latency-critical
scheduling loop.  This entry point keeps its scratch in a fixed array inside the
library's device image.  The tests call it through the C ABI twice in a row,
with batches of different sizes and contents (the second on a stream of its
own), and check each result against the allocating entry point bf_search_batch
and against the oracle (exact: makespans and indices are integers).  Collected
last so that a run stopping at the first failure has already run every other
test.
"""
import json
import os

import numpy as np
import pytest

import oracle
from paper_2607_22242_gb300 import bf
from paper_2607_22242_gb300 import scenarios as S

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "config_results.json")


@pytest.fixture(scope="module", autouse=True)
def cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def _same(a, b):
    return [(r.index, r.makespan_us, r.feasible, r.modes) for r in a] == \
           [(r.index, r.makespan_us, r.feasible, r.modes) for r in b]


def _batches():
    first = S.config4(bf.NOALLOC_MAX_SCENARIOS)          # the largest batch it accepts
    rng = np.random.default_rng(2024)
    second = [S.random_small(rng, int(rng.integers(1, 12)), max_time=int(rng.choice([9, 700])))
              for _ in range(301)]                           # smaller, mixed sizes: stale keys must not leak
    return first, second


def _oracle_optima(first, second):
    with open(GOLDEN) as fh:
        g = json.load(fh)["configs"]["4"]
    want_first = list(zip(g["best_index"][:len(first)], g["best_makespan"][:len(first)]))
    idx, ms = oracle.search_batch(second, oracle.default_threads())
    return want_first, [(int(i), int(m)) for i, m in zip(idx, ms)]


def test_noalloc_matches_allocating_batch_and_oracle_on_two_calls():
    import torch
    first, second = _batches()
    want_first, want_second = _oracle_optima(first, second)
    side = torch.cuda.Stream()
    for batch, stream, want in ((first, None, want_first), (second, side, want_second)):
        got = bf.search_batch_noalloc(batch, stream)
        assert [(r.index, r.makespan_us) for r in got] == want
        assert _same(got, bf.search_batch(batch, stream))


def test_noalloc_waits_for_a_timed_out_call():
    """A call that times out leaves its kernel reading the shared array; the next call must not reuse it
    until that kernel has finished.  64 copies of the 16-tool layered workload (about 0.2 s of kernel)
    outlast a 1 ms wait limit."""
    import torch
    with open(GOLDEN) as fh:
        g = json.load(fh)["configs"]["2"]["summary"]
    heavy = [S.config2()] * 64
    want_heavy = [(g["best_index"], g["best_makespan"])] * len(heavy)
    _, second = _batches()
    _, want_second = _oracle_optima([], second)
    busy = torch.cuda.Stream()
    torch.cuda.synchronize()
    try:
        bf.set_wait_timeout_ms(1)
        with pytest.raises(bf.BfError) as ei:
            bf.search_batch_noalloc(heavy, busy)
        assert ei.value.code == bf.BF_ETIMEOUT
        with pytest.raises(bf.BfError) as ei:               # the earlier call's kernel is still running
            bf.search_batch_noalloc(second)
        assert ei.value.code == bf.BF_ETIMEOUT and "earlier call" in ei.value.message
    finally:
        bf.set_wait_timeout_ms(600000)
    got = bf.search_batch_noalloc(second)                   # waits for the timed-out call, then runs
    assert [(r.index, r.makespan_us) for r in got] == want_second
    got = bf.search_batch_noalloc(heavy, busy)
    assert [(r.index, r.makespan_us) for r in got] == want_heavy


def test_noalloc_rejects_oversized_batch():
    batch = S.config4(bf.NOALLOC_MAX_SCENARIOS + 1)
    with pytest.raises(bf.BfError) as ei:
        bf.search_batch_noalloc(batch)
    assert ei.value.code == bf.BF_EINVAL
    assert str(bf.NOALLOC_MAX_SCENARIOS) in ei.value.message


def test_noalloc_two_groups():
    """Scenarios of up to 12 tools and of 13 and 14 tools interleaved in one call: two groups of the
    lane-tree batch kernel over the fixed scratch, every result at its position, equal to the
    oracle's."""
    from batch_cases import mixed_group_batch
    scns = mixed_group_batch()
    o_i, o_m = oracle.search_batch(scns, oracle.default_threads())
    got = bf.search_batch_noalloc(scns)
    assert [(r.index, r.makespan_us) for r in got] == list(zip(o_i.tolist(), o_m.tolist()))


def test_noalloc_all_three_groups():
    """A batch with scenarios of every lane-tree group -- up to 12 tools, 13 to 16, and 17 to 20 (the
    wide form) -- interleaved in one call: every result at its position, equal to bf_search_batch's
    (whose groups are checked against the oracle and against each scenario's full search)."""
    def layered(seed, sizes, budget):
        rng = np.random.default_rng(seed)
        n = sum(sizes)
        c, g, x, m = S._ordinary(rng, n, 2048, 16384)
        pred = S._layered_edges(rng, sizes, 0.4)
        return S.Scenario(n, pred, c, g, x, [S._load_from_vram(v) for v in m], m, budget,
                          S.slowdown_linear(kmax=n))
    scns = list(S.config4(6))
    scns.insert(2, layered(81, [4, 4, 3, 3, 3], 32768))   # 17 tools
    scns.insert(4, layered(82, [4, 4, 3, 2], 24576))      # 13 tools
    scns.append(layered(83, [4, 4, 4, 3, 3], 24576))      # 18 tools
    assert {0, 1, 2} == {0 if s.n <= 12 else (1 if s.n <= 16 else 2) for s in scns}
    got = bf.search_batch_noalloc(scns)
    assert _same(got, bf.search_batch(scns))
