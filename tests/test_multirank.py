"""Multi-rank path on CPU: world_size-2 gloo process groups (no GPU).

A search split over ranks (contiguous index ranges, one 8-byte key exchanged
per rank) must equal the single-process search; the per-rank step-time
reduction must be the maximum.  The CPU oracle stands in for each rank's GPU
range search.
"""
import os
import socket

import pytest
import torch.multiprocessing as mp

from paper_2607_22242_gb300 import shard


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, cfg, out):
    import torch.distributed as dist
    import oracle
    from paper_2607_22242_gb300 import scenarios as S
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        scn = S.config(cfg) if cfg >= 0 else S.Scenario(1, [0], [50], [5], [0], [0], [10], 5, S.slowdown_flat())
        total = 3 ** scn.n

        def search_range(first, count):
            idx, ms = oracle.search_range(scn, first, count)
            return (idx, ms, True) if idx >= 0 else (first, shard.INFEASIBLE, False)
        got = shard.sharded_search(search_range, total)
        step = shard.max_over_ranks(10.0 * (rank + 1))
        out.put((rank, got, step))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("cfg,world", [(0, 2), (1, 2), (0, 3), (-1, 2)])
def test_sharded_search_equals_single_process(cfg, world):
    import oracle
    from paper_2607_22242_gb300 import scenarios as S
    oracle.build()
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, cfg, out)) for r in range(world)]
    for p in procs:
        p.start()
    results = [out.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    scn = S.config(cfg) if cfg >= 0 else S.Scenario(1, [0], [50], [5], [0], [0], [10], 5, S.slowdown_flat())
    want = oracle.search(scn)
    for rank, (idx, ms, feasible), step in results:
        assert feasible and (idx, ms) == want, (rank, idx, ms, want)
        assert step == 10.0 * world


def test_shard_ranges_partition():
    for total in (1, 2, 3, 81, 6561, 3 ** 19):
        for world in (1, 2, 3, 8):
            spans = [shard.shard_range(total, r, world) for r in range(world)]
            assert spans[0][0] == 0
            assert sum(c for _, c in spans) == total
            for (f0, c0), (f1, _) in zip(spans, spans[1:]):
                assert f0 + c0 == f1


def test_key_order_is_makespan_then_index():
    a = shard.pack_key(7, 100, True)
    b = shard.pack_key(3, 100, True)
    c = shard.pack_key(0, 101, True)
    assert min(a, b, c) == b
    assert shard.unpack_key(min(a, b, c)) == (3, 100, True)
    assert shard.unpack_key(shard.pack_key(5, 0, False)) == (-1, shard.INFEASIBLE, False)


def _batch_worker(rank, world, port, count, out):
    import torch.distributed as dist
    import oracle
    from paper_2607_22242_gb300 import scenarios as S
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        scns = S.config4(count)

        def search_batch(block):
            idx, ms = oracle.search_batch(block)
            return [(int(i), int(m), int(m) != shard.INFEASIBLE) for i, m in zip(idx, ms)]
        out.put((rank, shard.sharded_batch(search_batch, scns)))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("count,world", [(9, 2), (7, 3), (2, 3)])
def test_sharded_batch_equals_single_process(count, world):
    """Scenarios split into contiguous blocks per rank (one with none when count < world):
    every rank gets every scenario's optimum, in order."""
    import oracle
    from paper_2607_22242_gb300 import scenarios as S
    oracle.build()
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_batch_worker, args=(r, world, port, count, out)) for r in range(world)]
    for p in procs:
        p.start()
    results = [out.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    idx, ms = oracle.search_batch(S.config4(count))
    want = [(int(i), int(m), True) for i, m in zip(idx, ms)]
    for rank, got in results:
        assert got == want, rank


def _bench_worker(rank, world, port, out):
    import torch.distributed as dist
    import oracle
    import bench
    from paper_2607_22242_gb300 import scenarios as S
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        scn = S.config(1)
        total = 3 ** scn.n
        seen = []

        def search_range(first, count):
            seen.append((first, count))
            idx, ms = oracle.search_range(scn, first, count)
            return (idx, ms, True) if idx >= 0 else (first, shard.INFEASIBLE, False)
        out.put((rank, bench.sharded_step(search_range, total), seen))
    finally:
        dist.destroy_process_group()


def test_bench_sharded_step_two_ranks():
    """The benchmark's multi-GPU step with the oracle standing in for each rank's GPU range search:
    two ranks search the two halves of the 12-tool workload's index space, once each, and both get
    the single-process optimum."""
    import oracle
    from paper_2607_22242_gb300 import scenarios as S
    oracle.build()
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_bench_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    results = sorted(out.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    scn = S.config(1)
    want = oracle.search(scn)
    total = 3 ** scn.n
    assert [seen for _, _, seen in results] == [[shard.shard_range(total, r, 2)] for r in range(2)]
    for rank, got, _ in results:
        assert got == want, rank
