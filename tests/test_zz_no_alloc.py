"""bf_search_batch_noalloc: the batched search for callers that cannot allocate.

Some callers cannot allocate device memory at the moment they search -- their
process has given all GPU memory to another allocator's pool, or a
cudaMalloc/cudaFree pair would synchronise the device inside a latency-critical
scheduling loop.  This entry point keeps its scratch in a fixed array inside the
library's device image.  The test calls it through the C ABI twice in a row,
with batches of different sizes and contents, and checks each result against
the allocating entry point bf_search_batch (exact: makespans and indices are
integers).  Collected last so that a run stopping at the first failure has
already run every other test.
"""
import numpy as np
import pytest

from paper_2607_22242_gb300 import bf
from paper_2607_22242_gb300 import scenarios as S

pytestmark = pytest.mark.gpu


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


def test_noalloc_matches_allocating_batch_on_two_calls():
    first = S.config4(bf.NOALLOC_MAX_SCENARIOS)          # the largest batch it accepts
    rng = np.random.default_rng(2024)
    second = [S.random_small(rng, int(rng.integers(1, 12)), max_time=int(rng.choice([9, 700])))
              for _ in range(301)]                           # smaller, mixed sizes: stale keys must not leak
    for batch in (first, second):
        got = bf.search_batch_noalloc(batch)
        want = bf.search_batch(batch)
        assert _same(got, want)


def test_noalloc_rejects_oversized_batch():
    batch = S.config4(bf.NOALLOC_MAX_SCENARIOS + 1)
    with pytest.raises(bf.BfError) as ei:
        bf.search_batch_noalloc(batch)
    assert ei.value.code == bf.BF_EINVAL
    assert str(bf.NOALLOC_MAX_SCENARIOS) in ei.value.message
