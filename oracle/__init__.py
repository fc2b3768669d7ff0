"""CPU oracle for the brute-force device-mapping search -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg may import this package.  It shares no code with the CUDA search.

Three restatements of the same integer latency model live here:

* ``bf_oracle.cpp`` (loaded through ctypes): the plain single-threaded event
  simulator plus enumerator; host threads only split index ranges.
* :mod:`oracle.pysim`: a structurally different Python restatement (per-tool
  remaining work, FIFO list) used to cross-check the C++ one on small N.
* :mod:`oracle.exact`: the same model in exact rational arithmetic with no
  rounding, used to bound the integer model's rounding error.

The model itself is stated at the top of ``bf_oracle.cpp``; the paper passages
it rests on are §2.1 (problem formulation), §2.3 (Factors A and B, the
brute-force oracle), Table 1 (profiles, gpu_queue = GPU + Load) and §4.1.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Sequence, Tuple

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
BUILD_DIR = os.path.join(HERE, "_build")
LIB_PATH = os.path.join(BUILD_DIR, "libbforacle.so")
SOURCE = os.path.join(HERE, "bf_oracle.cpp")

MAX_TOOLS = 32
FLAT_WORDS = 2 + 6 * MAX_TOOLS + (MAX_TOOLS + 1)
INFEASIBLE = 0xFFFFFFFF

_default = None


def build(force: bool = False, source: str = SOURCE, out: str = LIB_PATH) -> str:
    """Compile the oracle with g++ (-O2, portable flags only)."""
    os.makedirs(os.path.dirname(out), exist_ok=True)
    if (not force and os.path.exists(out)
            and os.path.getmtime(out) >= os.path.getmtime(source)):
        return out
    tmp = out + f".tmp{os.getpid()}"
    subprocess.check_call(["g++", "-O2", "-std=c++17", "-shared", "-fPIC", "-pthread",
                           source, "-o", tmp])
    os.replace(tmp, out)
    return out


def flat(scn) -> np.ndarray:
    """The oracle's own flat record: n, M, pred[32], c[32], g[32], x[32], l[32], m[32], f[33]."""
    w = np.zeros(FLAT_WORDS, dtype=np.uint32)
    n = scn.n
    w[0] = n
    w[1] = scn.vram_budget_mib
    cols = (scn.pred_mask, scn.cpu_us, scn.gpu_us, scn.xfer_us, scn.load_us, scn.vram_mib)
    for j, col in enumerate(cols):
        w[2 + j * MAX_TOOLS: 2 + j * MAX_TOOLS + n] = np.asarray(col[:n], dtype=np.uint64)
    f = np.asarray(scn.slowdown_q10[:MAX_TOOLS + 1], dtype=np.uint64)
    w[2 + 6 * MAX_TOOLS: 2 + 6 * MAX_TOOLS + len(f)] = f
    return w


def _ptr(a, ctype):
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def default_threads() -> int:
    if hasattr(os, "sched_getaffinity"):
        return max(1, len(os.sched_getaffinity(0)))
    return max(1, os.cpu_count() or 1)


class OracleLib:
    """ctypes view of one compiled copy of ``bf_oracle.cpp``."""

    def __init__(self, lib_path: str):
        lib = ctypes.CDLL(lib_path)
        u32p = ctypes.POINTER(ctypes.c_uint32)
        u64p = ctypes.POINTER(ctypes.c_uint64)
        u8p = ctypes.POINTER(ctypes.c_uint8)
        lib.bf_oracle_flat_words.restype = ctypes.c_int
        lib.bf_oracle_evaluate.argtypes = [u32p, ctypes.c_uint64]
        lib.bf_oracle_evaluate.restype = ctypes.c_uint64
        lib.bf_oracle_eval_range.argtypes = [u32p, ctypes.c_uint64, ctypes.c_uint64, u64p, u8p, ctypes.c_int]
        lib.bf_oracle_eval_range.restype = None
        lib.bf_oracle_search_range.argtypes = [u32p, ctypes.c_uint64, ctypes.c_uint64, u64p, u64p, ctypes.c_int]
        lib.bf_oracle_search_range.restype = ctypes.c_int
        lib.bf_oracle_search_batch.argtypes = [u32p, ctypes.c_uint64, u64p, u64p, ctypes.c_int]
        lib.bf_oracle_search_batch.restype = None
        lib.bf_oracle_summary_range.argtypes = [u32p, ctypes.c_uint64, ctypes.c_uint64, u64p, ctypes.c_int]
        lib.bf_oracle_summary_range.restype = None
        lib.bf_oracle_search_binary_range.argtypes = [u32p, ctypes.c_uint64, ctypes.c_uint64, u64p, u64p,
                                                      ctypes.c_int]
        lib.bf_oracle_search_binary_range.restype = ctypes.c_int
        assert lib.bf_oracle_flat_words() == FLAT_WORDS
        self.lib = lib

    def evaluate(self, scn, idx: int) -> int:
        """Makespan (us) of one mapping, or INFEASIBLE."""
        w = flat(scn)
        return int(self.lib.bf_oracle_evaluate(_ptr(w, ctypes.c_uint32), idx))

    def eval_range(self, scn, first: int, count: int, threads: int = 1) -> Tuple[np.ndarray, np.ndarray]:
        """(makespan uint64[count], feasible uint8[count]) of mappings [first, first+count)."""
        w = flat(scn)
        ms = np.empty(count, dtype=np.uint64)
        fe = np.empty(count, dtype=np.uint8)
        self.lib.bf_oracle_eval_range(_ptr(w, ctypes.c_uint32), first, count,
                                      _ptr(ms, ctypes.c_uint64), _ptr(fe, ctypes.c_uint8), threads)
        return ms, fe

    def search_range(self, scn, first: int, count: int, threads: int = 1) -> Tuple[int, int]:
        """(index, makespan) of the best feasible mapping in [first, first+count); (-1, INFEASIBLE) if none."""
        w = flat(scn)
        idx = np.zeros(1, dtype=np.uint64)
        ms = np.zeros(1, dtype=np.uint64)
        found = self.lib.bf_oracle_search_range(_ptr(w, ctypes.c_uint32), first, count,
                                                _ptr(idx, ctypes.c_uint64), _ptr(ms, ctypes.c_uint64), threads)
        if not found:
            return -1, INFEASIBLE
        return int(idx[0]), int(ms[0])

    def search(self, scn, threads: int = 1) -> Tuple[int, int]:
        return self.search_range(scn, 0, 3 ** scn.n, threads)

    def search_binary_range(self, scn, first: int, count: int, threads: int = 1) -> Tuple[int, int]:
        """Best feasible mapping among members [first, first+count) of the binary (cpu/gpu_now)
        decision space, member b having a_i = bit i of b; (index, makespan), (-1, INFEASIBLE) if none."""
        w = flat(scn)
        idx = np.zeros(1, dtype=np.uint64)
        ms = np.zeros(1, dtype=np.uint64)
        found = self.lib.bf_oracle_search_binary_range(_ptr(w, ctypes.c_uint32), first, count,
                                                       _ptr(idx, ctypes.c_uint64), _ptr(ms, ctypes.c_uint64),
                                                       threads)
        if not found:
            return -1, INFEASIBLE
        return int(idx[0]), int(ms[0])

    def search_binary(self, scn, threads: int = 1) -> Tuple[int, int]:
        """Optimum of the binary decision space (§4.1's S1-S10: each tool on the CPU or the GPU)."""
        return self.search_binary_range(scn, 0, 2 ** scn.n, threads)

    def summary_range(self, scn, first: int, count: int, threads: int = 1) -> dict:
        """Feasible count, makespan sum, order-sensitive hash and argmin of a range."""
        w = flat(scn)
        out = np.zeros(5, dtype=np.uint64)
        self.lib.bf_oracle_summary_range(_ptr(w, ctypes.c_uint32), first, count,
                                         _ptr(out, ctypes.c_uint64), threads)
        return dict(feasible=int(out[0]), makespan_sum=int(out[1]), hash=int(out[2]),
                    best_index=int(out[3]), best_makespan=int(out[4]))

    def search_batch(self, scns: Sequence, threads: int = 1) -> Tuple[np.ndarray, np.ndarray]:
        flats = np.concatenate([flat(s) for s in scns]) if len(scns) else np.zeros(FLAT_WORDS, np.uint32)
        idx = np.empty(len(scns), dtype=np.uint64)
        ms = np.empty(len(scns), dtype=np.uint64)
        self.lib.bf_oracle_search_batch(_ptr(flats, ctypes.c_uint32), len(scns),
                                        _ptr(idx, ctypes.c_uint64), _ptr(ms, ctypes.c_uint64), threads)
        return idx, ms


def default() -> OracleLib:
    global _default
    if _default is None:
        _default = OracleLib(build())
    return _default


def evaluate(scn, idx: int) -> int:
    return default().evaluate(scn, idx)


def eval_range(scn, first: int, count: int, threads: int = 1):
    return default().eval_range(scn, first, count, threads)


def search_range(scn, first: int, count: int, threads: int = 1):
    return default().search_range(scn, first, count, threads)


def search(scn, threads: int = 1):
    return default().search(scn, threads)


def search_batch(scns: Sequence, threads: int = 1):
    return default().search_batch(scns, threads)


def search_binary(scn, threads: int = 1):
    return default().search_binary(scn, threads)


def search_binary_range(scn, first: int, count: int, threads: int = 1):
    return default().search_binary_range(scn, first, count, threads)


def summary_range(scn, first: int, count: int, threads: int = 1):
    return default().summary_range(scn, first, count, threads)


def stream_hash(makespans: np.ndarray, first: int) -> int:
    """The summary's order-sensitive hash of a makespan stream starting at index ``first``."""
    ms = np.asarray(makespans, dtype=np.uint64)
    idx = np.arange(first, first + ms.size, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return int(np.sum(ms * (idx * np.uint64(2654435761) + np.uint64(1)), dtype=np.uint64))
