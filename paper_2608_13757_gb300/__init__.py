"""Python binding of the GB300 barrier-free semaphore engine.

A thin ctypes layer over ``include/sync.h``: it marshals arguments and owns
torch tensors for outputs; every step of the path runs in the library's CUDA
kernels.  The first call loads ``_lib/libsyncgb.so`` and fails loudly if it
is missing -- there is no CPU fallback.

    import paper_2608_13757_gb300 as sg
    h = sg.sync_load_programs(batch)                  # workloads.Batch or dict
    thr = sg.sync_eval_thresholds(h, sg.THR_PERLOOP)  # int32 [n_pairs_padded]
    counts, first_bad = sg.sync_check_minimal(h, sg.THR_PERLOOP, thr)
    res = sg.sync_simulate(h, sg.THR_PERLOOP, thr, sg.SimParams(), sg.SIM_BARRIER_FREE)
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libsyncgb.so")

OK, ERR_ARG, ERR_MALFORMED, ERR_NOT_ALLOCATABLE, ERR_OVERFLOW, ERR_CUDA, ERR_OOM = range(7)
THR_COUNT, THR_PERLOOP, THR_PERENGINE = 0, 1, 2
SIM_BARRIER_FREE, SIM_BARRIER, SIM_UNROLLED = 0, 1, 2
PROG_OK, PROG_OVERFLOW, PROG_DEADLOCK, PROG_ROUND_GUARD, PROG_TIMEOUT = 0, 4, 7, 8, 10

# every symbol include/sync.h declares
EXPORTS = ("sync_load_programs", "sync_query", "sync_pair_offsets", "sync_eval_thresholds",
           "sync_check_minimal", "sync_simulate", "sync_simulate_fused", "sync_simulate_noalloc",
           "sync_free_programs", "sync_last_error", "sync_kernel_launches", "sync_validate_programs")
NOALLOC_SCRATCH_BYTES = 64 << 20
CODE_BYTES_PER_INSTR = 16


class SyncError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"status {status}: {message}")
        self.status = status


class BatchDesc(ctypes.Structure):
    _fields_ = [("n_programs", ctypes.c_int32)] + [
        (n, ctypes.POINTER(ctypes.c_int32)) for n in (
            "prog_loop_ptr", "prog_instr_ptr", "prog_dep_ptr", "prog_n_engines",
            "loop_parent", "loop_pos", "instr_loop", "instr_pos", "instr_engine",
            "instr_latency", "dep_prod", "dep_cons", "dep_k")
    ] + [("trip_ptr", ctypes.POINTER(ctypes.c_int64)), ("trips", ctypes.POINTER(ctypes.c_int32)),
         ("eng_trip_ptr", ctypes.POINTER(ctypes.c_int64)), ("eng_trips", ctypes.POINTER(ctypes.c_int32)),
         ("nonalloc_policy", ctypes.c_int32)]

NONALLOC_REJECT, NONALLOC_BARRIER = 0, 1


class Sizes(ctypes.Structure):
    _fields_ = [("n_pairs", ctypes.c_int64), ("n_pairs_padded", ctypes.c_int64),
                ("n_instances", ctypes.c_int64), ("n_loop_iters", ctypes.c_int64),
                ("n_programs", ctypes.c_int32), ("n_loops", ctypes.c_int32),
                ("n_instrs", ctypes.c_int32), ("n_deps", ctypes.c_int32),
                ("device_bytes", ctypes.c_int64), ("h2d_bytes", ctypes.c_int64),
                ("struct_bytes", ctypes.c_int64), ("code_bytes_looped", ctypes.c_int64),
                ("code_bytes_unrolled", ctypes.c_int64), ("n_split_programs", ctypes.c_int32),
                ("n_pieces", ctypes.c_int32)]


class SimParams(ctypes.Structure):
    """Timing-model constants (cycles); defaults as in the library's docs."""
    _fields_ = [(n, ctypes.c_int32) for n in (
        "ii", "c_branch", "c_regop", "c_wait_ops_count", "c_wait_ops_perloop", "c_barrier",
        "c_wait_ops_perengine_level", "trip_register_elision", "licm", "cse")]

    def __init__(self, ii=1, c_branch=1, c_regop=1, c_wait_ops_count=3, c_wait_ops_perloop=5,
                 c_barrier=32, c_wait_ops_perengine_level=3, trip_register_elision=0, licm=0, cse=0):
        super().__init__(ii, c_branch, c_regop, c_wait_ops_count, c_wait_ops_perloop, c_barrier,
                         c_wait_ops_perengine_level, trip_register_elision, licm, cse)


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with "
                          "`python -m paper_2608_13757_gb300.build` (no CPU fallback exists)")
    lib = ctypes.CDLL(path)
    P = ctypes.POINTER
    vp = ctypes.c_void_p
    lib.sync_load_programs.argtypes = [P(BatchDesc), ctypes.c_int, vp, P(vp)]
    lib.sync_validate_programs.argtypes = [P(BatchDesc)]
    lib.sync_query.argtypes = [vp, P(Sizes)]
    lib.sync_pair_offsets.argtypes = [vp, P(ctypes.c_int64), P(ctypes.c_int32)]
    lib.sync_eval_thresholds.argtypes = [vp, ctypes.c_int, vp, vp]
    lib.sync_check_minimal.argtypes = [vp, ctypes.c_int, vp, vp, vp, vp]
    lib.sync_simulate.argtypes = [vp, ctypes.c_int, vp, P(SimParams), ctypes.c_int, vp, vp, vp,
                                  vp, vp, vp]
    lib.sync_simulate_noalloc.argtypes = lib.sync_simulate.argtypes
    lib.sync_simulate_fused.argtypes = [vp, ctypes.c_int, P(SimParams), ctypes.c_int, vp, vp, vp, vp, vp,
                                        vp, vp, vp]
    lib.sync_free_programs.argtypes = [vp]
    lib.sync_free_programs.restype = None
    lib.sync_last_error.argtypes = []
    lib.sync_last_error.restype = ctypes.c_char_p
    lib.sync_kernel_launches.argtypes = []
    lib.sync_kernel_launches.restype = ctypes.c_int64
    for f in EXPORTS:
        if f not in ("sync_free_programs", "sync_last_error", "sync_kernel_launches"):
            getattr(lib, f).restype = ctypes.c_int
    return lib


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded library (loaded on first use; raises if it was not built)."""
    global _lib
    if _lib is None:
        _lib = load_library()
    return _lib


def kernel_launches() -> int:
    """Kernels the library has launched in this process so far."""
    return int(lib().sync_kernel_launches())


def _check(status: int):
    if status != OK:
        raise SyncError(status, lib().sync_last_error().decode())


def _stream(stream):
    import torch
    if stream is None:
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, torch.cuda.Stream):
        return ctypes.c_void_p(stream.cuda_stream)
    return ctypes.c_void_p(int(stream))


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else None


def batch_desc(batch):
    """(BatchDesc, keep-alive list) for a workloads.Batch or a dict of arrays."""
    get = (lambda k: batch[k]) if isinstance(batch, dict) else (lambda k: getattr(batch, k))
    keep = []
    desc = BatchDesc()
    desc.n_programs = int(get("n_programs"))
    try:
        desc.nonalloc_policy = int(get("nonalloc_policy"))
    except (KeyError, AttributeError):
        desc.nonalloc_policy = NONALLOC_REJECT
    for name, _ in BatchDesc._fields_[1:-1]:
        is64 = name in ("trip_ptr", "eng_trip_ptr")
        try:
            v = get(name)
        except (KeyError, AttributeError):
            v = None
        if v is None:                       # shared trips: per-engine rows stay NULL
            continue
        a = np.ascontiguousarray(v, dtype=np.int64 if is64 else np.int32)
        keep.append(a)
        setattr(desc, name, a.ctypes.data_as(ctypes.POINTER(ctypes.c_int64 if is64 else ctypes.c_int32)))
    return desc, keep


class Programs:
    """A loaded batch (owns the device encoding; freed on close / GC)."""

    def __init__(self, handle: ctypes.c_void_p, device: int):
        self._h = handle
        self.device = device
        s = Sizes()
        _check(lib().sync_query(self._h, ctypes.byref(s)))
        self.sizes = s
        self._pairs = None

    def _pair_layout(self):
        """(segment offsets [n_deps + 1], pairs per dependency [n_deps]),
        read back on first use."""
        if self._pairs is None:
            n = self.sizes.n_deps
            off = np.zeros(n + 1, dtype=np.int64)
            cnt = np.zeros(max(n, 1), dtype=np.int32)
            _check(lib().sync_pair_offsets(self.handle, off.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)),
                                          cnt.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))))
            self._pairs = (off, cnt[:n])
        return self._pairs

    @property
    def pair_offsets(self) -> np.ndarray:
        return self._pair_layout()[0]

    @property
    def pair_counts(self) -> np.ndarray:
        return self._pair_layout()[1]

    def unpadded_index(self) -> np.ndarray:
        """Indices into a threshold array, in pair order without padding."""
        if self.sizes.n_deps == 0:
            return np.zeros(0, dtype=np.int64)
        starts = np.repeat(self.pair_offsets[:-1], self.pair_counts)
        base = np.repeat(np.cumsum(self.pair_counts) - self.pair_counts, self.pair_counts)
        return starts + (np.arange(int(self.pair_counts.sum()), dtype=np.int64) - base)

    @property
    def handle(self):
        if not self._h:
            raise ValueError("programs already freed")
        return self._h

    def close(self):
        if self._h:
            lib().sync_free_programs(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def sync_load_programs(batch, device: int = 0, stream=None) -> Programs:
    import torch
    desc, keep = batch_desc(batch)
    h = ctypes.c_void_p()
    with torch.cuda.device(device):
        _check(lib().sync_load_programs(ctypes.byref(desc), int(device), _stream(stream),
                                       ctypes.byref(h)))
    del keep
    return Programs(h, device)


def sync_eval_thresholds(h: Programs, mode: int = THR_PERLOOP, out=None, stream=None):
    import torch
    n = h.sizes.n_pairs_padded
    if out is None:
        out = torch.empty(max(n, 4), dtype=torch.int32, device=f"cuda:{h.device}")
    _check(lib().sync_eval_thresholds(h.handle, int(mode), _ptr(out), _stream(stream)))
    return out


def sync_check_minimal(h: Programs, mode, thr, counts=None, first_bad=None, stream=None):
    """Returns (counts uint64-as-int64 tensor [2], first_bad int64 tensor [1])."""
    import torch
    dev = f"cuda:{h.device}"
    if counts is None:
        counts = torch.empty(2, dtype=torch.int64, device=dev)
    if first_bad is None:
        first_bad = torch.empty(1, dtype=torch.int64, device=dev)
    _check(lib().sync_check_minimal(h.handle, int(mode), _ptr(thr), _ptr(counts), _ptr(first_bad),
                                   _stream(stream)))
    return counts, first_bad


@dataclass
class SimOutputs:
    makespan: "object"
    checksum: "object"      # int64 tensor holding the uint64 bit pattern
    status: "object"
    issue: "object" = None
    retire: "object" = None


def sync_simulate(h: Programs, mode, thr, params: SimParams | None = None,
                  variant: int = SIM_BARRIER_FREE, timeline: bool = False, out: SimOutputs | None = None,
                  stream=None) -> SimOutputs:
    import torch
    dev = f"cuda:{h.device}"
    P = h.sizes.n_programs
    if out is None:
        out = SimOutputs(torch.empty(max(P, 1), dtype=torch.int32, device=dev),
                         torch.empty(max(P, 1), dtype=torch.int64, device=dev),
                         torch.empty(max(P, 1), dtype=torch.int32, device=dev))
        if timeline:
            n = max(h.sizes.n_instances, 1)
            out.issue = torch.full((n,), -1, dtype=torch.int32, device=dev)
            out.retire = torch.full((n,), -1, dtype=torch.int32, device=dev)
    prm = params if params is not None else SimParams()
    _check(lib().sync_simulate(h.handle, int(mode), _ptr(thr), ctypes.byref(prm), int(variant),
                              _ptr(out.makespan), _ptr(out.checksum), _ptr(out.status),
                              _ptr(out.issue), _ptr(out.retire), _stream(stream)))
    return out


def sync_simulate_fused(h: Programs, mode, params: SimParams | None = None,
                        variant: int = SIM_BARRIER_FREE, timeline: bool = False, check: bool = False,
                        out: SimOutputs | None = None, counts=None, first_bad=None, stream=None):
    """Simulation with every wait value computed inside the simulators (no
    threshold array).  Returns the SimOutputs, and with check=True also
    (counts [2], first_bad [1]) as sync_check_minimal does, for the programs
    whose status is OK."""
    import torch
    dev = f"cuda:{h.device}"
    P = h.sizes.n_programs
    if out is None:
        out = SimOutputs(torch.empty(max(P, 1), dtype=torch.int32, device=dev),
                         torch.empty(max(P, 1), dtype=torch.int64, device=dev),
                         torch.empty(max(P, 1), dtype=torch.int32, device=dev))
        if timeline:
            n = max(h.sizes.n_instances, 1)
            out.issue = torch.full((n,), -1, dtype=torch.int32, device=dev)
            out.retire = torch.full((n,), -1, dtype=torch.int32, device=dev)
    if check:
        if counts is None:
            counts = torch.empty(2, dtype=torch.int64, device=dev)
        if first_bad is None:
            first_bad = torch.empty(1, dtype=torch.int64, device=dev)
    prm = params if params is not None else SimParams()
    _check(lib().sync_simulate_fused(h.handle, int(mode), ctypes.byref(prm), int(variant),
                                    _ptr(out.makespan), _ptr(out.checksum), _ptr(out.status),
                                    _ptr(out.issue), _ptr(out.retire),
                                    _ptr(counts) if check else None, _ptr(first_bad) if check else None,
                                    _stream(stream)))
    return (out, counts, first_bad) if check else out


def sync_simulate_noalloc(h: Programs, mode, thr, params: SimParams | None = None,
                          variant: int = SIM_BARRIER_FREE, out: SimOutputs | None = None,
                          timeline: bool = False, stream=None) -> SimOutputs:
    """sync_simulate for callers that cannot allocate device memory around a
    simulation: the call allocates nothing and uses the library's static
    scratch (NOALLOC_SCRATCH_BYTES per GPU).  Pass preallocated outputs in
    `out` to keep the whole call free of allocations; without `out` this
    wrapper allocates the output tensors itself (the library call does not).
    Calls share the scratch, so calls that overlap on the GPU race."""
    import torch
    dev = f"cuda:{h.device}"
    P = h.sizes.n_programs
    if out is None:
        out = SimOutputs(torch.empty(max(P, 1), dtype=torch.int32, device=dev),
                         torch.empty(max(P, 1), dtype=torch.int64, device=dev),
                         torch.empty(max(P, 1), dtype=torch.int32, device=dev))
        if timeline:
            n = max(h.sizes.n_instances, 1)
            out.issue = torch.full((n,), -1, dtype=torch.int32, device=dev)
            out.retire = torch.full((n,), -1, dtype=torch.int32, device=dev)
    prm = params if params is not None else SimParams()
    _check(lib().sync_simulate_noalloc(h.handle, int(mode), _ptr(thr), ctypes.byref(prm), int(variant),
                                       _ptr(out.makespan), _ptr(out.checksum), _ptr(out.status),
                                       _ptr(out.issue), _ptr(out.retire), _stream(stream)))
    return out


def sync_free_programs(h: Programs):
    h.close()
