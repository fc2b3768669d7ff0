"""The CPU oracle against its pins (no GPU)."""
import pytest

import pins


@pytest.mark.parametrize("check", pins.ALL_CHECKS, ids=lambda c: c.__name__)
def test_pin(check, oracle_lib):
    check(oracle_lib)


def test_table3_totals_match_table1():
    """Table 3's total memory is the sum of the Table 1 footprints of its four tools (to 1 MB)."""
    t1 = {t["tool"]: t for t in pins._load("paper_table1.json")["tools"]}
    for sc in pins._load("paper_table3.json")["scenarios"]:
        total = sum(t1[name]["vram_mb"] or 0 for name in sc["tools"])
        assert abs(total - sc["total"]) <= 1, sc
