"""Seeded scenarios shared by the host-built tests (input generation only, no arithmetic of the
method).

tie_order_scenarios(): queue-heavy tiny DAGs (tight budgets, steep contention, CPU times scaled
up to 10x) with sources late in the numbering, so that the searches that renumber with the
sources first run renumbered; among them are tied optima whose lowest member differs between the
canonical and the renumbered order (scenario 91 of the default list is the first).
"""
import numpy as np

from paper_2607_22242_gb300 import scenarios as S


def tie_order_scenarios(count=120, seed=1):
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(count):
        n = int(rng.integers(3, 8))
        base = S.random_small(rng, n, edge_p=float(rng.choice([0.1, 0.3, 0.6])), tight=True, contention=True,
                              max_time=int(rng.choice([2, 3, 10])))
        cpu = [c * int(rng.choice([1, 3, 10])) for c in base.cpu_us]
        pred = list(base.pred_mask)
        for v in rng.choice(np.arange(1, n), size=int(rng.integers(1, n // 2 + 1)), replace=False):
            pred[int(v)] = 0
        out.append(S.Scenario(n, pred, cpu, base.gpu_us, base.xfer_us, base.load_us, base.vram_mib,
                              base.vram_budget_mib, base.slowdown_q10))
    return out
