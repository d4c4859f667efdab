"""CPU oracle for barrier-free semaphore thresholds -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  It wraps ``oracle.c`` (plain C, built
with gcc) through ctypes and shares no code with the GPU library.

Layouts (see ``oracle.h``): thresholds in *pair* layout -- dependency-major,
one entry per consumer instance in the order of the consumer loop's global
iteration index, no padding; issue/retire in *instance* layout --
instruction-major, one entry per global iteration of the instruction's loop.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIBDIR = os.path.join(_HERE, "_lib")
_LIB = os.path.join(_LIBDIR, "liboracle.so")
_SRC = [os.path.join(_HERE, "oracle.c")]
_HDR = [os.path.join(_HERE, "oracle.h")]

COUNT, PERLOOP, PERENGINE = 0, 1, 2
BARRIER_FREE, BARRIER, UNROLLED = 0, 1, 2
CASE_PS, CASE_NEST_FWD, CASE_NEST_BWD, CASE_NONE, CASE_BARRIER = 0, 1, 2, 3, 4
SIM_OK, SIM_OVERFLOW, SIM_DEADLOCK = 0, 4, 7


def build(force: bool = False) -> str:
    """Compile ``oracle/_lib/liboracle.so`` (gcc -O2, no SIMD intrinsics)."""
    os.makedirs(_LIBDIR, exist_ok=True)
    newest = max(os.path.getmtime(p) for p in _SRC + _HDR)
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= newest:
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", "-O2", "-std=gnu11", "-Wall", "-Wextra", "-fPIC", "-shared",
                           "-o", tmp] + _SRC)
    os.replace(tmp, _LIB)
    return _LIB


class _Batch(ctypes.Structure):
    _fields_ = [("n_programs", ctypes.c_int32)] + [
        (n, ctypes.POINTER(ctypes.c_int32)) for n in (
            "prog_loop_ptr", "prog_instr_ptr", "prog_dep_ptr", "prog_n_engines",
            "loop_parent", "loop_pos", "instr_loop", "instr_pos", "instr_engine",
            "instr_latency", "dep_prod", "dep_cons", "dep_k")
    ] + [("trip_ptr", ctypes.POINTER(ctypes.c_int64)), ("trips", ctypes.POINTER(ctypes.c_int32)),
         ("eng_trip_ptr", ctypes.POINTER(ctypes.c_int64)), ("eng_trips", ctypes.POINTER(ctypes.c_int32)),
         ("nonalloc_policy", ctypes.c_int32)]


class SimParams(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "ii", "c_branch", "c_regop", "c_wait_ops_count", "c_wait_ops_perloop", "c_barrier",
        "c_wait_ops_perengine_level", "trip_register_elision", "licm", "cse")]


def sim_params(**kw) -> SimParams:
    """Timing-model constants; defaults ii=1, c_branch=1, c_regop=1, 3 / 5 wait
    ops per dependency (count / per-loop, Table 1), c_barrier=32, and 3 more
    ops per enclosing loop level for a per-engine wait (Sec. 6.1); the ALU
    reductions of Sec. 6.2 (licm, cse) off."""
    d = dict(ii=1, c_branch=1, c_regop=1, c_wait_ops_count=3, c_wait_ops_perloop=5, c_barrier=32,
             c_wait_ops_perengine_level=3, trip_register_elision=0, licm=0, cse=0)
    d.update(kw)
    return SimParams(**d)


_lib = None


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.POINTER
        i32p, i64p, u64p = P(ctypes.c_int32), P(ctypes.c_int64), P(ctypes.c_uint64)
        bp = P(_Batch)
        lib.orc_sizes.argtypes = [bp, i64p, i64p]
        lib.orc_classify.argtypes = [bp, i32p, i32p, i32p, i32p, i32p]
        lib.orc_code_size.argtypes = [bp, i64p, i64p]
        lib.orc_thresholds_bruteforce.argtypes = [bp, ctypes.c_int, i32p]
        lib.orc_thresholds.argtypes = [bp, ctypes.c_int, i32p]
        lib.orc_register_replay.argtypes = [bp, ctypes.c_int, i32p]
        lib.orc_check.argtypes = [bp, ctypes.c_int, i32p, u64p, i64p]
        lib.orc_simulate.argtypes = [bp, ctypes.c_int, i32p, P(SimParams), ctypes.c_int, i32p,
                                     u64p, i32p, i32p, i32p]
        for f in ("orc_sizes", "orc_code_size", "orc_classify", "orc_thresholds_bruteforce", "orc_thresholds",
                  "orc_register_replay", "orc_check", "orc_simulate"):
            getattr(lib, f).restype = ctypes.c_int
        _lib = lib
    return _lib


def _ptr(a, ct):
    return a.ctypes.data_as(ctypes.POINTER(ct))


class _View:
    """Keeps contiguous copies of a batch's arrays alive for one call."""

    def __init__(self, batch):
        self.keep = {}
        cb = _Batch()
        cb.n_programs = int(batch.n_programs)
        cb.nonalloc_policy = int(getattr(batch, "nonalloc_policy", 0))
        for name, _ in _Batch._fields_[1:-1]:
            a = getattr(batch, name, None)
            if a is None:                 # shared trips: the per-engine rows stay NULL
                continue
            dt = np.int64 if name in ("trip_ptr", "eng_trip_ptr") else np.int32
            a = np.ascontiguousarray(a, dtype=dt)
            self.keep[name] = a
            setattr(cb, name, _ptr(a, ctypes.c_int64 if dt == np.int64 else ctypes.c_int32))
        self.cb = cb


class OracleError(RuntimeError):
    pass


def _check(rc, what):
    if rc != 0:
        raise OracleError(f"{what} failed with status {rc}")


def sizes(batch):
    """(number of pairs, number of instruction instances)."""
    lib, v = _load(), _View(batch)
    npairs, ninst = ctypes.c_int64(), ctypes.c_int64()
    _check(lib.orc_sizes(ctypes.byref(v.cb), ctypes.byref(npairs), ctypes.byref(ninst)), "sizes")
    return npairs.value, ninst.value


CODE_BYTES_PER_INSTR = 16


def code_size(batch):
    """(looped, unrolled) code-size proxy in instructions (see oracle.h)."""
    lib, v = _load(), _View(batch)
    lp, un = ctypes.c_int64(), ctypes.c_int64()
    _check(lib.orc_code_size(ctypes.byref(v.cb), ctypes.byref(lp), ctypes.byref(un)), "code_size")
    return lp.value, un.value


@dataclass
class Classes:
    S: np.ndarray
    P: np.ndarray
    kase: np.ndarray
    N: np.ndarray
    K: np.ndarray


def classify(batch) -> Classes:
    lib, v = _load(), _View(batch)
    n = batch.dep_prod.shape[0]
    out = [np.zeros(n, dtype=np.int32) for _ in range(5)]
    _check(lib.orc_classify(ctypes.byref(v.cb), *[_ptr(o, ctypes.c_int32) for o in out]),
           "classify")
    return Classes(*out)


def _thr(fn, batch, mode):
    lib, v = _load(), _View(batch)
    npairs, _ = sizes(batch)
    out = np.full(npairs, -7, dtype=np.int32)
    _check(getattr(lib, fn)(ctypes.byref(v.cb), int(mode), _ptr(out, ctypes.c_int32)), fn)
    return out


def thresholds(batch, mode=PERLOOP) -> np.ndarray:
    """Eq. (1) thresholds (counting form), pair layout."""
    return _thr("orc_thresholds", batch, mode)


def thresholds_bruteforce(batch, mode=PERLOOP) -> np.ndarray:
    """Eq. (1) thresholds (pairwise lexicographic comparison), pair layout."""
    return _thr("orc_thresholds_bruteforce", batch, mode)


def register_replay(batch, mode=PERLOOP) -> np.ndarray:
    """Wait values computed by the paper's registers, replayed per engine."""
    return _thr("orc_register_replay", batch, mode)


def check(batch, thr, mode=PERLOOP):
    """(unsafe, oversync, first bad pair index or -1) for a pair-layout array."""
    lib, v = _load(), _View(batch)
    thr = np.ascontiguousarray(thr, dtype=np.int32)
    counts = np.zeros(2, dtype=np.uint64)
    fb = ctypes.c_int64()
    _check(lib.orc_check(ctypes.byref(v.cb), int(mode), _ptr(thr, ctypes.c_int32),
                         _ptr(counts, ctypes.c_uint64), ctypes.byref(fb)), "check")
    return int(counts[0]), int(counts[1]), fb.value


@dataclass
class SimResult:
    makespan: np.ndarray
    checksum: np.ndarray
    status: np.ndarray
    issue: np.ndarray | None = None
    retire: np.ndarray | None = None


def simulate(batch, thr, mode=PERLOOP, variant=BARRIER_FREE, params: SimParams | None = None,
             timeline: bool = False) -> SimResult:
    lib, v = _load(), _View(batch)
    thr = np.ascontiguousarray(thr, dtype=np.int32)
    P = batch.n_programs
    ms = np.zeros(P, dtype=np.int32)
    ck = np.zeros(P, dtype=np.uint64)
    st = np.zeros(P, dtype=np.int32)
    iss = ret = None
    if timeline:
        _, ninst = sizes(batch)
        iss = np.full(ninst, -1, dtype=np.int32)
        ret = np.full(ninst, -1, dtype=np.int32)
    prm = params if params is not None else sim_params()
    _check(lib.orc_simulate(ctypes.byref(v.cb), int(mode), _ptr(thr, ctypes.c_int32),
                            ctypes.byref(prm), int(variant), _ptr(ms, ctypes.c_int32),
                            _ptr(ck, ctypes.c_uint64), _ptr(st, ctypes.c_int32),
                            _ptr(iss, ctypes.c_int32) if timeline else None,
                            _ptr(ret, ctypes.c_int32) if timeline else None), "simulate")
    return SimResult(ms, ck, st, iss, ret)
