"""Host-side fault injection with a GPU present: failures are made on the host (an
allocation the library is told to fail), never on the GPU."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SCRIPT = r"""
import sys
sys.path.insert(0, {root!r})
import torch
from paper_2607_22242_gb300 import bf, scenarios as S
torch.cuda.set_device(0)
scn = S.config0()
try:
    bf.create_scenario(scn)
    print("created")
except bf.BfError as e:
    print("error", e.code, e.message)
# the library still works after the injected failure
with bf.create_scenario(scn) as h:
    print("after", bf.search_best(h).index)
"""


@pytest.fixture(scope="module", autouse=True)
def built():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


@pytest.mark.parametrize("nth", ["1", "2"])
def test_injected_allocation_failure(nth):
    env = dict(os.environ, BF_FAIL_ALLOC=nth)
    out = subprocess.run([sys.executable, "-c", SCRIPT.format(root=ROOT)], env=env, capture_output=True,
                         text=True, timeout=300)
    assert out.returncode == 0, out.stderr
    lines = out.stdout.split("\n")
    assert lines[0].startswith("error 3 ")            # BF_ENOMEM
    assert "bf_create_scenario" in lines[0]
    assert lines[1] == "after 3280"                    # the N=8 workload's optimum


def test_no_injection_by_default():
    env = {k: v for k, v in os.environ.items() if k != "BF_FAIL_ALLOC"}
    out = subprocess.run([sys.executable, "-c", SCRIPT.format(root=ROOT)], env=env, capture_output=True,
                         text=True, timeout=300)
    assert out.returncode == 0, out.stderr
    assert out.stdout.split("\n")[:2] == ["created", "after 3280"]
