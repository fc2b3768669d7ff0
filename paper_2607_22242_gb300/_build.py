"""Build ``libbf.so`` in-tree with nvcc for sm_103a (GB300).

Each window-width bucket of ``csrc/bf_kernels.cu`` is its own translation unit
(``-DBF_NW=<slots>``); the units compile in parallel and link with ``bf_tree.cu``
(the tree search and 32-slot index lists), ``bf_capi.cu`` and ``bf_capi_tree.cu`` into
``paper_2607_22242_gb300/_build/libbf.so`` (CUDA runtime linked statically, so
the library carries no path to a toolkit; no undefined symbol is allowed).
"""
from __future__ import annotations

import concurrent.futures as cf
import hashlib
import re
import os
import shutil
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(os.path.dirname(HERE), "include")
BUILD_DIR = os.path.join(HERE, "_build")
LIB_PATH = os.path.join(BUILD_DIR, "libbf.so")
BUCKETS = tuple(range(4, 21))  # window widths (bf_sim.cuh): one unit per width from 4 to 20
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden",
              f"-I{INCLUDE}"]


def nvcc() -> str:
    path = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(path):
        raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libbf.so")
    return path


def _sources():
    return ([os.path.join(CSRC, f) for f in sorted(os.listdir(CSRC))] + [os.path.join(INCLUDE, "bf.h")]
            + [os.path.abspath(__file__)])  # the build recipe itself


def _fingerprint(extra) -> str:
    """Hash of the kernel sources and flags, independent of where the repository lives."""
    h = hashlib.sha256()
    for path in _sources():
        with open(path, "rb") as fh:
            h.update(os.path.basename(path).encode() + fh.read())
    flags = [f for f in NVCC_FLAGS if not f.startswith("-I")]
    h.update(" ".join(ARCH + flags + list(extra)).encode())
    return h.hexdigest()


# Sources of the enumerating kernels' translation unit (bf_kernels.cu and what it includes), and
# the host planner that chooses their launches (splits, windows, grid sizes).
KERNEL_UNIT = ("bf_kernels.cu", "bf_enum.cuh", "bf_sim.cuh", "bf_launch.h", "bf_plan.h")


def _code_only(text: str) -> str:
    """C++ source without comments and with whitespace runs collapsed (no string literal in the
    kernel unit contains a comment marker)."""
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    return " ".join(text.split())


# Sources of the lane-tree batch kernel's translation unit, and the planner of its launches.
LANETREE_UNIT = ("bf_lanetree.cu", "bf_lanetree.cuh", "bf_lanetree_launch.h", "bf_enum.cuh", "bf_sim.cuh",
                 "bf_launch.h", "bf_plan.h")


def kernel_fingerprint(csrc: str = CSRC, unit=KERNEL_UNIT) -> str:
    """Hash of a kernel translation unit's code (comments and layout ignored) and flags -- by default
    the enumerating kernels', LANETREE_UNIT for the lane-tree batch kernel: a profile taken of those
    kernels stays valid while this is unchanged (changes elsewhere in the library, or to comments,
    do not touch them)."""
    h = hashlib.sha256()
    for name in unit:
        with open(os.path.join(csrc, name), encoding="utf-8") as fh:
            h.update(name.encode() + _code_only(fh.read()).encode())
    flags = [f for f in NVCC_FLAGS if not f.startswith("-I")]
    h.update(" ".join(ARCH + flags).encode())
    return h.hexdigest()


def build(force: bool = False, extra_flags=(), verbose: bool = False) -> str:
    """Compile and link libbf.so unless an up-to-date copy exists; return its path."""
    os.makedirs(BUILD_DIR, exist_ok=True)
    stamp = os.path.join(BUILD_DIR, "libbf.stamp")
    fp = _fingerprint(extra_flags)
    if not force and os.path.exists(LIB_PATH) and os.path.exists(stamp):
        with open(stamp) as fh:
            if fh.read().strip() == fp:
                return LIB_PATH
    cc = nvcc()
    jobs = []
    for nt in BUCKETS:
        obj = os.path.join(BUILD_DIR, f"bf_kernels_nw{nt}.o")
        jobs.append([cc, *ARCH, *NVCC_FLAGS, *extra_flags, f"-DBF_NW={nt}", "-c",
                     os.path.join(CSRC, "bf_kernels.cu"), "-o", obj])
    for unit in ("bf_tree", "bf_lanetree", "bf_capi", "bf_capi_tree"):
        jobs.append([cc, *ARCH, *NVCC_FLAGS, *extra_flags, "-c", os.path.join(CSRC, unit + ".cu"), "-o",
                     os.path.join(BUILD_DIR, unit + ".o")])

    def run(cmd):
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError(f"nvcc failed: {' '.join(cmd)}\n{res.stdout}\n{res.stderr}")
        if verbose:
            print(res.stdout + res.stderr)
        return cmd[-1]

    workers = min(len(jobs), max(1, os.cpu_count() or 1))
    with cf.ThreadPoolExecutor(workers) as pool:
        objs = list(pool.map(run, jobs))
    tmp = LIB_PATH + f".tmp{os.getpid()}"
    run([cc, *ARCH, "-shared", "-cudart", "static", "-Xlinker", "--no-undefined", "-o", tmp, *objs])
    os.replace(tmp, LIB_PATH)
    with open(stamp, "w") as fh:
        fh.write(fp)
    return LIB_PATH


if __name__ == "__main__":
    print(build(force=True, verbose=False))
