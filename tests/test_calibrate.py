"""Contention-table calibration on the paper's S5 (Table 2) with the batched search."""
import pytest

import pins
from paper_2607_22242_gb300 import calibrate as C
from paper_2607_22242_gb300 import scenarios as S


def test_s5_inputs_follow_the_paper():
    scn = C.s5(C.table(0.35, 1.0))
    # Table 3: S5's total memory is the sum of the Table 1 footprints
    s5_row = {s["id"]: s for s in pins._load("paper_table3.json")["scenarios"]}["S5"]
    assert sum(scn.vram_mib) == s5_row["total"] == 4136
    # Table 2: isolated GPU latencies, vector_search_x15 measured on CPU
    assert scn.gpu_us == [370_000, 136_000, 277_000, 145_000]
    assert scn.cpu_us[2] == 706_000
    # §4.3: image_resize_x30's ratio is 3.7x
    assert abs(scn.cpu_us[3] / scn.gpu_us[3] - 3.7) < 1e-3
    # the oracle mapping offloads vector_search_x15 (Table 3: GPU, GPU, CPU, GPU)
    assert S.mapping_index(C.S5_ORACLE) == 1 + 3 + 27


def test_candidate_tables_are_valid():
    from paper_2607_22242_gb300 import _build, bf
    _build.build()
    for a, b in C.candidates(a_steps=11):
        f = C.table(a, b)
        assert f[1] == 1024 and all(f[k] <= f[k + 1] for k in range(1, 4))
        bf.validate_desc(C.s5(f))


@pytest.mark.gpu
def test_calibration_matches_oracle():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import oracle
    grid = C.candidates(a_steps=41)
    best, fits = C.calibrate(grid=grid)
    for fit in fits[::17] + [best]:
        scn = C.s5(fit.f)
        assert (fit.argmin, fit.optimum_us) == oracle.search(scn)
        assert fit.all_gpu_us == oracle.evaluate(scn, S.mapping_index(C.S5_ALL_GPU))
        assert fit.oracle_us == oracle.evaluate(scn, S.mapping_index(C.S5_ORACLE))
    assert best.paper_oracle_optimal
