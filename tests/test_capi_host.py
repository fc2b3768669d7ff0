"""Host-side checks of the C ABI: the library builds, loads, exports every
declared entry point, and rejects invalid scenarios -- no GPU needed."""
import ctypes
import os
import re

import pytest

from paper_2607_22242_gb300 import _build, bf
from paper_2607_22242_gb300 import scenarios as S

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "bf.h")


@pytest.fixture(scope="module")
def lib():
    _build.build()
    return bf.load()


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*BF_API\s+(?:int|void|const char\s*\*)\s*(bf_\w+)\s*\(", text, re.M)))


def test_header_declares_the_abi():
    assert declared_functions() == sorted(bf.EXPORTED)


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert bf.version().startswith("bf ")


def test_only_declared_symbols_are_exported(lib):
    """The library exports its C entry points and nothing of its internals."""
    import subprocess
    out = subprocess.run(["nm", "-D", "--defined-only", bf.LIB_PATH], capture_output=True, text=True)
    if out.returncode != 0:
        pytest.skip("nm unavailable")
    names = {line.split()[-1] for line in out.stdout.splitlines() if line.split()[1:2] == ["T"]}
    assert {n for n in names if n.startswith("bf_")} == set(declared_functions())
    assert not [n for n in names if n.startswith("_ZN3bfk")], "internal C++ symbols are exported"


def test_generated_configs_validate(lib):
    for i in range(4):
        bf.validate_desc(S.config(i))
    for s in S.config4(64):
        bf.validate_desc(s)


def _base():
    return S.config0()


def _with(**kw):
    d = _base().to_dict()
    d.update(kw)
    return S.Scenario(**d)


INVALID = {
    "n=0": lambda: _with(n=0),
    "n=33": lambda: S.Scenario(33, [0] * 33, [1] * 33, [1] * 33, [0] * 33, [0] * 33, [1] * 33, 10,
                               S.slowdown_flat(33)),
    "f missing above k=20": lambda: S.Scenario(21, [0] * 21, [1] * 21, [1] * 21, [0] * 21, [0] * 21, [1] * 21, 10,
                                               S.slowdown_flat()),
    "backward edge": lambda: _with(pred_mask=[0, 0, 1 << 5] + [0] * 5),
    "self loop": lambda: _with(pred_mask=[0, 1 << 1] + [0] * 6),
    "zero cpu": lambda: _with(cpu_us=[0] + _base().cpu_us[1:]),
    "zero gpu": lambda: _with(gpu_us=[0] + _base().gpu_us[1:]),
    "queued work too long": lambda: _with(load_us=[1 << 22] + _base().load_us[1:]),
    "vram too large": lambda: _with(vram_mib=[(1 << 27) + 1] + _base().vram_mib[1:]),
    "f[1] != 1024": lambda: _with(slowdown_q10=[0, 1000] + [1024] * 19),
    "f decreasing": lambda: _with(slowdown_q10=[0, 1024, 2000, 1500] + [2000] * 17),
    "f too large": lambda: _with(slowdown_q10=[0, 1024, 70000] + [70000] * 18),
    "makespan overflow": lambda: _with(cpu_us=[2_000_000_000] * 8),
}


@pytest.mark.parametrize("case", sorted(INVALID))
def test_invalid_desc_rejected(lib, case):
    with pytest.raises(bf.BfError) as ei:
        bf.validate_desc(INVALID[case]())
    assert ei.value.code == bf.BF_EINVAL
    assert ei.value.message.startswith("bf_validate_desc:"), ei.value.message


def test_null_desc(lib):
    assert lib.bf_validate_desc(None) == bf.BF_EINVAL
    assert "NULL" in bf.last_error()


def test_null_out_pointer(lib):
    d = bf.to_desc(_base())
    assert lib.bf_create_scenario(ctypes.byref(d), None) == bf.BF_EINVAL


def test_destroy_null_is_ok(lib):
    assert lib.bf_destroy_scenario(None) == bf.BF_OK


def test_null_handle_calls_rejected(lib):
    r = bf.CResult()
    assert lib.bf_search_best(None, ctypes.byref(r), None) == bf.BF_EINVAL
    assert lib.bf_search_range(None, 0, 1, ctypes.byref(r), None) == bf.BF_EINVAL
    assert lib.bf_eval_mappings(None, 0, 1, None, None, None) == bf.BF_EINVAL


def test_batch_reports_bad_position(lib):
    descs = (bf.Desc * 3)(bf.to_desc(_base()), bf.to_desc(_base()), bf.to_desc(_with(n=0)))
    out = (bf.CResult * 3)()
    assert lib.bf_search_batch(descs, 3, out, None) == bf.BF_EINVAL
    assert "descs[2]" in bf.last_error()


def test_empty_batch_is_ok(lib):
    assert lib.bf_search_batch(None, 0, None, None) == bf.BF_OK


def test_boundary_values_accepted(lib):
    # largest queued work and n = 20 with a makespan bound just inside 32 bits
    n = 20
    s = S.Scenario(n, [0] + [1 << (i - 1) for i in range(1, n)], [1] * n, [(1 << 22) - 1] + [1] * 19,
                   [0] * n, [0] * n, [1 << 27] * n, 1 << 31, [0, 1024] + [65536] * 19)
    bf.validate_desc(s)


def test_wide_desc_accepted(lib):
    """32 tools validate; the enumerating batch search refuses more than 20 before touching the GPU."""
    n = 32
    s = S.Scenario(n, [0] + [1 << (i - 1) for i in range(1, n)], [1000] * n, [100] * n, [0] * n, [0] * n,
                   [1] * n, 10, S.slowdown_linear(35, kmax=n))
    bf.validate_desc(s)
    bf.validate_desc(S.wide28())
    bf.validate_desc(S.wide32())
    bf.validate_desc(S.layered24())
    descs = (bf.Desc * 1)(bf.to_desc(s))
    out = (bf.CResult * 1)()
    assert lib.bf_search_batch(descs, 1, out, None) == bf.BF_EINVAL
    assert "n <= 20" in bf.last_error()
    assert lib.bf_search_batch_noalloc(descs, 1, out, None) == bf.BF_EINVAL


def test_binding_rejects_bad_output_buffers(lib):
    """Buffer checks are exceptions (not asserts that `python -O` would drop)."""
    import torch
    with pytest.raises(ValueError):
        bf.eval_indices(S.config0(), torch.zeros(4, dtype=torch.int64))   # a CPU tensor
    with pytest.raises(ValueError):
        bf._check_out(torch.zeros(4, dtype=torch.int32), torch.zeros(4, dtype=torch.uint8), 4)
