"""Python binding of ``libbf.so`` (C ABI in ``include/bf.h``).

Argument marshalling only: every step of the search runs in the library's
CUDA kernels.  PyTorch supplies device buffers (``eval_mappings`` outputs) and
streams (``torch.cuda.current_stream()`` by default).  The functions mirror
the C entry points without their ``bf_`` prefix: ``validate_desc``,
``create_scenario``, ``destroy_scenario``, ``eval_mappings``, ``search_best``,
``search_range``, ``search_batch``, ``search_batch_noalloc``, ``eval_indices``,
``whatif``, ``search_pruned``, ``set_wait_timeout_ms``, ``last_error``,
``version``.

There is no CPU fallback: if ``libbf.so`` has not been built, or no CUDA
device is present, these calls raise.
"""
from __future__ import annotations

import ctypes
import dataclasses
import itertools
import os
from typing import List, Optional, Sequence, Tuple, Union

from .scenarios import MAX_TOOLS, Scenario

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_build", "libbf.so")

BF_OK, BF_EINVAL, BF_ERANGE, BF_ENOMEM, BF_ECUDA, BF_ETIMEOUT = range(6)
STATUS_NAMES = {0: "BF_OK", 1: "BF_EINVAL", 2: "BF_ERANGE", 3: "BF_ENOMEM", 4: "BF_ECUDA", 5: "BF_ETIMEOUT"}
INFEASIBLE = 0xFFFFFFFF
EXPORTED = ("bf_validate_desc", "bf_create_scenario", "bf_destroy_scenario", "bf_eval_mappings",
            "bf_search_best", "bf_search_range", "bf_search_batch", "bf_search_batch_noalloc",
            "bf_eval_indices", "bf_whatif", "bf_search_pruned", "bf_search_tree", "bf_set_wait_timeout_ms",
            "bf_last_error", "bf_version")
SPACE_BINARY, SPACE_FULL = 2, 3
TREE_NO_PRUNE = 1
MAX_PROBES = 2 * MAX_TOOLS + MAX_TOOLS * MAX_TOOLS
NOALLOC_MAX_SCENARIOS = 1024


class BfError(RuntimeError):
    def __init__(self, code: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(code, code)}: {message}")
        self.code = code
        self.message = message


U32xT = ctypes.c_uint32 * MAX_TOOLS


class Desc(ctypes.Structure):
    """``bf_scenario_desc``."""
    _fields_ = [("n", ctypes.c_uint32), ("pred_mask", U32xT), ("cpu_us", U32xT), ("gpu_us", U32xT),
                ("xfer_us", U32xT), ("load_us", U32xT), ("vram_mib", U32xT),
                ("vram_budget_mib", ctypes.c_uint32), ("slowdown_q10", ctypes.c_uint32 * (MAX_TOOLS + 1))]


class CResult(ctypes.Structure):
    """``bf_result``."""
    _fields_ = [("index", ctypes.c_uint64), ("makespan_us", ctypes.c_uint32), ("feasible", ctypes.c_uint32),
                ("mode", ctypes.c_uint8 * MAX_TOOLS)]


class CProbe(ctypes.Structure):
    """``bf_probe``."""
    _fields_ = [("index", ctypes.c_uint64), ("makespan_us", ctypes.c_uint32), ("feasible", ctypes.c_uint32),
                ("kind", ctypes.c_uint8), ("tool", ctypes.c_uint8), ("mode", ctypes.c_uint8),
                ("other", ctypes.c_uint8)]


@dataclasses.dataclass
class Probe:
    """One what-if probe of Algorithm 1: kind 'single' (tool -> mode) or 'swap'
    (tool -> gpu_now, other -> gpu_queue)."""
    kind: str
    tool: int
    mode: int
    other: Optional[int]
    index: int
    makespan_us: int
    feasible: bool


class CTreeStats(ctypes.Structure):
    """``bf_tree_stats``."""
    _fields_ = [("nodes", ctypes.c_uint64), ("leaf_nodes", ctypes.c_uint64), ("leaves", ctypes.c_uint64),
                ("launches", ctypes.c_uint32), ("leaf_depth", ctypes.c_uint32), ("incumbent_us", ctypes.c_uint32),
                ("pad", ctypes.c_uint32)]


@dataclasses.dataclass
class Result:
    index: int
    makespan_us: int
    feasible: bool
    modes: List[int]


_lib = None


def load(path: str = LIB_PATH):
    """Load libbf.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(path)
    vp, u64, u32 = ctypes.c_void_p, ctypes.c_uint64, ctypes.c_uint32
    lib.bf_validate_desc.argtypes = [ctypes.POINTER(Desc)]
    lib.bf_create_scenario.argtypes = [ctypes.POINTER(Desc), ctypes.POINTER(vp)]
    lib.bf_destroy_scenario.argtypes = [vp]
    lib.bf_eval_mappings.argtypes = [vp, u64, u64, vp, vp, vp]
    lib.bf_search_best.argtypes = [vp, ctypes.POINTER(CResult), vp]
    lib.bf_search_range.argtypes = [vp, u64, u64, ctypes.POINTER(CResult), vp]
    lib.bf_search_batch.argtypes = [ctypes.POINTER(Desc), u32, ctypes.POINTER(CResult), vp]
    lib.bf_search_batch_noalloc.argtypes = [ctypes.POINTER(Desc), u32, ctypes.POINTER(CResult), vp]
    lib.bf_eval_indices.argtypes = [vp, vp, u64, vp, vp, vp]
    lib.bf_whatif.argtypes = [vp, u64, ctypes.POINTER(CProbe), u32, ctypes.POINTER(u32), vp]
    lib.bf_search_pruned.argtypes = [vp, u64, ctypes.POINTER(CResult), vp]
    lib.bf_search_tree.argtypes = [vp, u32, u32, u64, ctypes.POINTER(CResult), ctypes.POINTER(CTreeStats), vp]
    for name in ("bf_validate_desc", "bf_create_scenario", "bf_destroy_scenario", "bf_eval_mappings",
                 "bf_search_best", "bf_search_range", "bf_search_batch", "bf_search_batch_noalloc",
                 "bf_eval_indices", "bf_whatif", "bf_search_pruned", "bf_search_tree"):
        getattr(lib, name).restype = ctypes.c_int
    lib.bf_set_wait_timeout_ms.argtypes = [u32]
    lib.bf_set_wait_timeout_ms.restype = None
    lib.bf_last_error.restype = ctypes.c_char_p
    lib.bf_version.restype = ctypes.c_char_p
    _lib = lib
    return lib


def _check(code: int):
    if code != BF_OK:
        raise BfError(code, last_error())


def last_error() -> str:
    return load().bf_last_error().decode()


def version() -> str:
    return load().bf_version().decode()


def set_wait_timeout_ms(ms: int) -> None:
    load().bf_set_wait_timeout_ms(ms)


def to_desc(scn: Scenario) -> Desc:
    d = Desc()
    d.n = scn.n
    for name in ("pred_mask", "cpu_us", "gpu_us", "xfer_us", "load_us", "vram_mib"):
        arr = getattr(d, name)
        for i, v in enumerate(getattr(scn, name)[:MAX_TOOLS]):
            arr[i] = v
    d.vram_budget_mib = scn.vram_budget_mib
    for k, v in enumerate(scn.slowdown_q10[:MAX_TOOLS + 1]):
        d.slowdown_q10[k] = v
    return d


DESC_WORDS = ctypes.sizeof(Desc) // 4


def pack_descs(scns: Sequence[Scenario]):
    """Pack scenarios into a contiguous (count, DESC_WORDS) uint32 array laid out as bf_scenario_desc[]."""
    import numpy as np
    count = len(scns)
    arr = np.zeros((count, DESC_WORDS), dtype=np.uint32)
    if count == 0:
        return arr
    cols = ("pred_mask", "cpu_us", "gpu_us", "xfer_us", "load_us", "vram_mib")
    sizes = {sc.n for sc in scns}
    if len(sizes) == 1:  # one tool count: fill whole columns at once
        n = sizes.pop()
        arr[:, 0] = n
        flat = lambda rows, width: np.fromiter(itertools.chain.from_iterable(rows), dtype=np.uint32,
                                               count=count * width).reshape(count, width)
        for j, name in enumerate(cols):
            arr[:, 1 + MAX_TOOLS * j: 1 + MAX_TOOLS * j + n] = flat((getattr(sc, name)[:n] for sc in scns), n)
        arr[:, 1 + 6 * MAX_TOOLS] = np.fromiter((sc.vram_budget_mib for sc in scns), dtype=np.uint32, count=count)
        pad = [0] * (MAX_TOOLS + 1)
        arr[:, 2 + 6 * MAX_TOOLS:] = flat(((sc.slowdown_q10 + pad)[:MAX_TOOLS + 1] for sc in scns), MAX_TOOLS + 1)
        return arr
    for r, sc in enumerate(scns):
        arr[r, 0] = sc.n
        for j, name in enumerate(cols):
            arr[r, 1 + MAX_TOOLS * j: 1 + MAX_TOOLS * j + sc.n] = getattr(sc, name)[:sc.n]
        arr[r, 1 + 6 * MAX_TOOLS] = sc.vram_budget_mib
        f = sc.slowdown_q10[:MAX_TOOLS + 1]
        arr[r, 2 + 6 * MAX_TOOLS: 2 + 6 * MAX_TOOLS + len(f)] = f
    return arr


def _result(r: CResult, n: int) -> Result:
    return Result(int(r.index), int(r.makespan_us), bool(r.feasible), [int(r.mode[i]) for i in range(n)])


def _stream_handle(stream) -> int:
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream) if hasattr(stream, "cuda_stream") else int(stream)


def validate_desc(scn: Scenario) -> None:
    """Raise BfError(BF_EINVAL) if the scenario is outside the library's limits."""
    d = to_desc(scn)
    _check(load().bf_validate_desc(ctypes.byref(d)))


class ScenarioHandle:
    """An owned ``bf_scenario*``; released by :meth:`close` (or garbage collection)."""

    def __init__(self, scn: Scenario):
        self.scenario = scn
        self._ptr = ctypes.c_void_p()
        d = to_desc(scn)
        _check(load().bf_create_scenario(ctypes.byref(d), ctypes.byref(self._ptr)))

    @property
    def ptr(self):
        if not self._ptr:
            raise ValueError("scenario handle is closed")
        return self._ptr

    def close(self):
        if self._ptr:
            ptr, self._ptr = self._ptr, ctypes.c_void_p()
            _check(load().bf_destroy_scenario(ptr))

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()


def create_scenario(scn: Scenario) -> ScenarioHandle:
    return ScenarioHandle(scn)


def destroy_scenario(handle: ScenarioHandle) -> None:
    handle.close()


def _handle(h: Union[ScenarioHandle, Scenario]) -> Tuple[ScenarioHandle, bool]:
    if isinstance(h, ScenarioHandle):
        return h, False
    return ScenarioHandle(h), True


def _check_out(out_makespan, out_feasible, count: int) -> None:
    """Output buffers: contiguous CUDA tensors of >= count 4-byte / 1-byte elements."""
    for t, size, name in ((out_makespan, 4, "out_makespan"), (out_feasible, 1, "out_feasible")):
        if not (t.is_cuda and t.is_contiguous() and t.element_size() == size and t.numel() >= count):
            raise ValueError(f"{name} must be a contiguous CUDA tensor of >= {count} {size}-byte elements")


def eval_mappings(h: Union[ScenarioHandle, Scenario], first: int, count: int, out_makespan=None,
                  out_feasible=None, stream=None):
    """Makespans (torch.int32 CUDA tensor holding u32 bit patterns) and feasibility
    flags (torch.uint8) of mappings [first, first+count).  Asynchronous on ``stream``;
    the scenario's tables travel by value with the launch, so a temporary handle
    may be released as soon as the call returns."""
    import torch
    handle, owned = _handle(h)
    try:
        if out_makespan is None:
            out_makespan = torch.empty(count, dtype=torch.int32, device="cuda")
        if out_feasible is None:
            out_feasible = torch.empty(count, dtype=torch.uint8, device="cuda")
        _check_out(out_makespan, out_feasible, count)
        _check(load().bf_eval_mappings(handle.ptr, first, count, ctypes.c_void_p(out_makespan.data_ptr()),
                                       ctypes.c_void_p(out_feasible.data_ptr()),
                                       ctypes.c_void_p(_stream_handle(stream))))
        return out_makespan, out_feasible
    finally:
        if owned:
            handle.close()


def search_best(h: Union[ScenarioHandle, Scenario], stream=None) -> Result:
    """Optimal feasible mapping over all 3^n (ties to the lowest index)."""
    handle, owned = _handle(h)
    try:
        r = CResult()
        _check(load().bf_search_best(handle.ptr, ctypes.byref(r), ctypes.c_void_p(_stream_handle(stream))))
        return _result(r, handle.scenario.n)
    finally:
        if owned:
            handle.close()


def search_range(h: Union[ScenarioHandle, Scenario], first: int, count: int, stream=None) -> Result:
    """Best feasible mapping in [first, first+count) (feasible=False if none)."""
    handle, owned = _handle(h)
    try:
        r = CResult()
        _check(load().bf_search_range(handle.ptr, first, count, ctypes.byref(r),
                                      ctypes.c_void_p(_stream_handle(stream))))
        return _result(r, handle.scenario.n)
    finally:
        if owned:
            handle.close()


def _batch_call(fn, scns: Sequence[Scenario], stream, packed=None) -> List[Result]:
    count = len(scns)
    if packed is None and count:
        packed = pack_descs(scns)
    descs = packed.ctypes.data_as(ctypes.POINTER(Desc)) if count else None
    results = (CResult * max(count, 1))()
    _check(fn(descs, count, results, ctypes.c_void_p(_stream_handle(stream))))
    if not count:
        return []
    import numpy as np
    arr = np.ctypeslib.as_array(results)  # one structured view instead of per-field ctypes reads
    modes = arr["mode"][:, :max(sc.n for sc in scns)].tolist()
    return [Result(i, m, bool(f), md[:sc.n]) for i, m, f, md, sc in
            zip(arr["index"].tolist(), arr["makespan_us"].tolist(), arr["feasible"].tolist(), modes, scns)]


def search_batch(scns: Sequence[Scenario], stream=None, packed=None) -> List[Result]:
    """Full search of each scenario, the whole batch in one call.  ``packed`` (from
    :func:`pack_descs` of the same scenarios) skips the packing when a batch is searched repeatedly."""
    return _batch_call(load().bf_search_batch, scns, stream, packed)


def search_batch_noalloc(scns: Sequence[Scenario], stream=None) -> List[Result]:
    """As :func:`search_batch`, but the library allocates no memory for the call.

    For callers that cannot allocate device memory while they search (their GPU
    memory belongs to another allocator's pool, or a cudaMalloc/cudaFree pair
    would synchronise the device inside a latency-critical loop).  The scratch is
    a fixed array in the library's device image; at most NOALLOC_MAX_SCENARIOS
    scenarios per call.  Calls on one device are serialised; after a call that
    timed out, the next one first waits for that call's stream.
    """
    return _batch_call(load().bf_search_batch_noalloc, scns, stream)


def eval_indices(h: Union[ScenarioHandle, Scenario], indices, out_makespan=None, out_feasible=None, stream=None):
    """Makespans (torch.int32, u32 bit patterns) and flags (torch.uint8; 0xFF for an
    index outside [0, 3^n)) of the mappings in `indices` (a CUDA int64 tensor)."""
    import torch
    if not (indices.is_cuda and indices.dtype == torch.int64 and indices.is_contiguous()):
        raise ValueError("indices must be a contiguous CUDA int64 tensor")
    handle, owned = _handle(h)
    try:
        count = indices.numel()
        if out_makespan is None:
            out_makespan = torch.empty(count, dtype=torch.int32, device=indices.device)
        if out_feasible is None:
            out_feasible = torch.empty(count, dtype=torch.uint8, device=indices.device)
        _check_out(out_makespan, out_feasible, count)
        _check(load().bf_eval_indices(handle.ptr, ctypes.c_void_p(indices.data_ptr()), count,
                                      ctypes.c_void_p(out_makespan.data_ptr()),
                                      ctypes.c_void_p(out_feasible.data_ptr()),
                                      ctypes.c_void_p(_stream_handle(stream))))
        return out_makespan, out_feasible
    finally:
        if owned:
            handle.close()


def whatif(h: Union[ScenarioHandle, Scenario], base_index: int, stream=None) -> List[Probe]:
    """The single-tool and swap reprobes of Algorithm 1 around `base_index`, scored on the GPU."""
    handle, owned = _handle(h)
    try:
        out = (CProbe * MAX_PROBES)()
        count = ctypes.c_uint32(0)
        _check(load().bf_whatif(handle.ptr, base_index, out, MAX_PROBES, ctypes.byref(count),
                                ctypes.c_void_p(_stream_handle(stream))))
        return [Probe("swap" if p.kind else "single", p.tool, p.mode, None if p.kind == 0 else p.other,
                      p.index, p.makespan_us, bool(p.feasible)) for p in out[:count.value]]
    finally:
        if owned:
            handle.close()


def search_pruned(h: Union[ScenarioHandle, Scenario], hint_index: Optional[int] = None, stream=None) -> Result:
    """The optimum of :func:`search_best`, found by branch and bound (exact)."""
    handle, owned = _handle(h)
    try:
        r = CResult()
        hint = (1 << 64) - 1 if hint_index is None else hint_index
        _check(load().bf_search_pruned(handle.ptr, hint, ctypes.byref(r), ctypes.c_void_p(_stream_handle(stream))))
        return _result(r, handle.scenario.n)
    finally:
        if owned:
            handle.close()


def search_tree(h: Union[ScenarioHandle, Scenario], space: int = SPACE_FULL, prune: bool = True,
                hint_index: Optional[int] = None, stream=None) -> Tuple[Result, dict]:
    """Optimum of the full (space=3) or binary cpu/gpu_now (space=2) decision space of a scenario of up to
    32 tools, by depth-first branch and bound (prune=False: every mapping simulated); (result, stats)."""
    handle, owned = _handle(h)
    try:
        r = CResult()
        st = CTreeStats()
        hint = (1 << 64) - 1 if hint_index is None else hint_index
        _check(load().bf_search_tree(handle.ptr, space, 0 if prune else TREE_NO_PRUNE, hint, ctypes.byref(r),
                                     ctypes.byref(st), ctypes.c_void_p(_stream_handle(stream))))
        stats = dict(nodes=st.nodes, leaf_nodes=st.leaf_nodes, leaves=st.leaves, launches=st.launches,
                     leaf_depth=st.leaf_depth, incumbent_us=st.incumbent_us)
        return _result(r, handle.scenario.n), stats
    finally:
        if owned:
            handle.close()
