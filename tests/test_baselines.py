"""Baseline policies (All-GPU, memory-aware greedy, HEFT): their defining rules
on CPU, and on the GPU their scores against the brute-force optimum."""
import numpy as np
import pytest

import pins
from paper_2607_22242_gb300 import baselines as B
from paper_2607_22242_gb300 import scenarios as S
from paper_2607_22242_gb300.scenarios import CPU, GPU_NOW


def _paper_fanout(ids):
    """S11-S13 of Table 3 with the Table 1 profiles."""
    tools = {t["tool"]: t for t in pins._load("paper_table1.json")["tools"]}
    sc = {s["id"]: s for s in pins._load("paper_table3.json")["scenarios"]}[ids]
    return pins._fanout([tools[name] for name in sc["tools"]], sc["budget"])


def test_all_gpu_is_every_tool_on_gpu_now():
    for i in range(4):
        scn = S.config(i)
        assert S.mapping_index(B.all_gpu(scn)) == sum(3 ** k for k in range(scn.n))


def test_greedy_on_the_paper_three_way_scenarios():
    # §4.4: by decreasing speedup into gpu_now until the budget is exhausted, then CPU.
    f7 = pins._load("paper_fig7.json")
    tools = [dict(cpu_ms=t["cpu"], gpu_ms=t["gpu"], load_ms=t["load"], vram_mb=t["mem"]) for t in f7["tools"]]
    s13 = pins._fanout(tools, f7["budget_mb"])         # Figure 7 profiles of S13, 1100 MB
    assert B.memory_aware_greedy(s13) == [GPU_NOW, GPU_NOW, CPU, CPU]
    assert B.memory_aware_greedy(_paper_fanout("S12")) == [GPU_NOW] * 4       # 1135 MB fits 1700
    assert B.memory_aware_greedy(_paper_fanout("S11")) == [CPU, GPU_NOW, GPU_NOW, GPU_NOW]  # ocr (8x) last


def test_greedy_rule_on_random_scenarios():
    rng = np.random.default_rng(5)
    for _ in range(200):
        scn = S.random_small(rng, int(rng.integers(1, 12)))
        modes = B.memory_aware_greedy(scn)
        order = sorted(range(scn.n), key=lambda i: (-scn.cpu_us[i] / (scn.gpu_us[i] + scn.xfer_us[i]), i))
        on = [i for i in order if modes[i] == GPU_NOW]
        assert on == order[:len(on)]                     # a prefix of the speedup order
        assert sum(scn.vram_mib[i] for i in on) <= scn.vram_budget_mib
        if len(on) < scn.n:                              # the next tool does not fit
            assert sum(scn.vram_mib[i] for i in on) + scn.vram_mib[order[len(on)]] > scn.vram_budget_mib


def test_heft_places_chain_tools_on_their_faster_device():
    rng = np.random.default_rng(6)
    for _ in range(100):
        n = int(rng.integers(1, 10))
        base = S.random_small(rng, n, max_time=500)
        chain = S.Scenario(n, [0] + [1 << (i - 1) for i in range(1, n)], base.cpu_us, base.gpu_us, base.xfer_us,
                           base.load_us, base.vram_mib, base.vram_budget_mib, base.slowdown_q10)
        want = [GPU_NOW if base.gpu_us[i] + base.xfer_us[i] < base.cpu_us[i] else CPU for i in range(n)]
        assert B.heft(chain) == want


def test_heft_shares_one_gpu_in_a_fanout():
    # four identical tools, GPU 10 us, CPU 25 us: HEFT (exclusive GPU) runs two on the GPU back to
    # back (finishing at 10 and 20) and puts the others on CPU cores (25 < 30)
    n = 4
    scn = S.Scenario(n, [0] * n, [25] * n, [10] * n, [0] * n, [0] * n, [1] * n, 100, S.slowdown_flat())
    assert B.heft(scn) == [GPU_NOW, GPU_NOW, CPU, CPU]


@pytest.mark.gpu
def test_gaps_scored_on_gpu_match_the_oracle():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import oracle
    from paper_2607_22242_gb300 import bf
    golden = pins._load("config_results.json")["configs"]
    for i in range(4):
        scn = S.config(i)
        with bf.create_scenario(scn) as h:
            g = B.gaps(h)
        best = g["optimum"]
        summary = golden[str(i)]["summary"]
        assert (best.index, best.makespan_us) == (summary["best_index"], summary["best_makespan"])
        for name in B.POLICIES:
            want = oracle.evaluate(scn, g[name].index)
            assert g[name].makespan_us == want and g[name].feasible == (want != 0xFFFFFFFF)
            if g[name].feasible:
                assert g[name].makespan_us >= best.makespan_us and g[name].gap >= 0.0
