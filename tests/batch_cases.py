"""Seeded batches shared by the GPU tests (input generation only, no arithmetic of the method).

mixed_group_batch(): scenarios of 1-12 tools interleaved with scenarios of 13 and 14 tools, which a
batch call searches in two groups (the lane-tree batch kernel's two- and three-chunk forms), so that
its results must come back to their positions from both groups.
"""
import numpy as np

from paper_2607_22242_gb300 import scenarios as S


def mixed_group_batch(seed=4242, count=18):
    rng = np.random.default_rng(seed)
    scns = []
    for t in range(count):
        n = int(rng.integers(13, 15)) if t % 3 == 0 else int(rng.integers(1, 13))
        scns.append(S.random_small(rng, n, edge_p=float(rng.choice([0.2, 0.5])),
                                   max_time=int(rng.choice([9, 400]))))
    return scns
