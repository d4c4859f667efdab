"""Seeded synthetic batches of structured multi-engine programs.

This package is the shared input generator of the repository: it decides the
shape of a workload (loop trees, instruction placement on engines, dependency
lists, trip counts per parent iteration) and nothing else.  It holds none of
the synchronisation method's arithmetic, so both the CPU oracle and the GPU
library can consume the same batch without sharing any computation.

A batch is a structure of arrays (program-local ids, int32 unless noted):

* ``prog_loop_ptr``, ``prog_instr_ptr``, ``prog_dep_ptr`` -- CSR row pointers
  ``[n_programs+1]`` into the loop, instruction and dependency arrays;
* ``prog_n_engines`` -- engines per program (1..32);
* ``loop_parent`` (-1 for loop 0, the top-level loop), ``loop_pos`` (position
  of the loop among the items of its parent's body);
* ``instr_loop``, ``instr_pos``, ``instr_engine``, ``instr_latency``;
* ``dep_prod``, ``dep_cons``, ``dep_k`` -- producer, consumer, offset on the
  innermost common loop;
* ``trip_ptr`` (int64, ``[n_loops+1]``) and ``trips``: the trips of loop ``l``
  during each global iteration of its parent, ``trips[trip_ptr[l]:trip_ptr[l+1]]``;
  the top-level loop has the single trip 1;
* optional, for engines whose trip counts diverge: ``eng_trip_ptr`` (int64,
  one entry per (program, loop, engine) row plus one) and ``eng_trips``: row
  ``R_p + l*n_engines + e`` (``R_p`` = rows of the programs before ``p``)
  holds the trips of loop ``l`` on engine ``e`` during each global iteration
  of its parent on that engine.  When present they replace ``trips`` (which
  then holds engine 0's trips).

The named configurations follow the five workload families the engine is
measured on (a small single-loop program, a depth-2 nest, a tiled GEMM, causal
flash attention, random chain programs and their synchronisation-bound
variant).  Every program is a pure function of ``(config, seed, program id)``,
so a contiguous range of programs can be generated on its own and is identical
to the same range of the full batch.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass, fields

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIBDIR = os.path.join(_HERE, "_lib")
_LIB = os.path.join(_LIBDIR, "libsynth.so")
_SRC = [os.path.join(_HERE, "synth.c")]
_HDR = [os.path.join(_HERE, "synth.h")]

TREE, SMALL, DEPTH2, GEMM, ATTENTION, CHAIN, SYNCBOUND = range(7)

# name -> (config id, default number of programs)
CONFIGS = {
    "small": (SMALL, 1),
    "depth2": (DEPTH2, 4096),
    "gemm": (GEMM, 1),
    "attention": (ATTENTION, 256),
    "chain": (CHAIN, 65536),
    "syncbound": (SYNCBOUND, 65536),
}


def config_seed(cfg: int) -> int:
    """Seed of a named configuration: 0x5EED0000 + its id."""
    return 0x5EED0000 + int(cfg)


def build(force: bool = False) -> str:
    """Compile the generator into ``workloads/_lib/libsynth.so`` (gcc, -O2)."""
    os.makedirs(_LIBDIR, exist_ok=True)
    newest = max(os.path.getmtime(p) for p in _SRC + _HDR)
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= newest:
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-Wall", "-Wextra", "-fPIC", "-shared",
                           "-o", tmp] + _SRC)
    os.replace(tmp, _LIB)
    return _LIB


class _CBatch(ctypes.Structure):
    _fields_ = [
        ("n_programs", ctypes.c_int32),
        ("n_loops", ctypes.c_int64), ("n_instrs", ctypes.c_int64),
        ("n_deps", ctypes.c_int64), ("n_trips", ctypes.c_int64),
        ("prog_loop_ptr", ctypes.POINTER(ctypes.c_int32)),
        ("prog_instr_ptr", ctypes.POINTER(ctypes.c_int32)),
        ("prog_dep_ptr", ctypes.POINTER(ctypes.c_int32)),
        ("prog_n_engines", ctypes.POINTER(ctypes.c_int32)),
        ("loop_parent", ctypes.POINTER(ctypes.c_int32)),
        ("loop_pos", ctypes.POINTER(ctypes.c_int32)),
        ("instr_loop", ctypes.POINTER(ctypes.c_int32)),
        ("instr_pos", ctypes.POINTER(ctypes.c_int32)),
        ("instr_engine", ctypes.POINTER(ctypes.c_int32)),
        ("instr_latency", ctypes.POINTER(ctypes.c_int32)),
        ("dep_prod", ctypes.POINTER(ctypes.c_int32)),
        ("dep_cons", ctypes.POINTER(ctypes.c_int32)),
        ("dep_k", ctypes.POINTER(ctypes.c_int32)),
        ("trip_ptr", ctypes.POINTER(ctypes.c_int64)),
        ("trips", ctypes.POINTER(ctypes.c_int32)),
    ]


class TreeParams(ctypes.Structure):
    """Parameters of the general random-tree generator (tests)."""
    _fields_ = [(n, ctypes.c_int32) for n in (
        "engines_lo", "engines_hi", "max_depth", "loops_lo", "loops_hi", "body_lo", "body_hi",
        "trip_lo", "trip_hi", "cond_permille", "lat_lo", "lat_hi", "dep_permille",
        "max_deps_per_cons", "k_max", "any_k", "nest_far_permille")]


def tree_params(**kw) -> TreeParams:
    d = dict(engines_lo=1, engines_hi=4, max_depth=3, loops_lo=0, loops_hi=4, body_lo=0,
             body_hi=4, trip_lo=0, trip_hi=3, cond_permille=150, lat_lo=1, lat_hi=8,
             dep_permille=500, max_deps_per_cons=2, k_max=2, any_k=0, nest_far_permille=0)
    d.update(kw)
    return TreeParams(**d)


@dataclass
class Batch:
    n_programs: int
    prog_loop_ptr: np.ndarray
    prog_instr_ptr: np.ndarray
    prog_dep_ptr: np.ndarray
    prog_n_engines: np.ndarray
    loop_parent: np.ndarray
    loop_pos: np.ndarray
    instr_loop: np.ndarray
    instr_pos: np.ndarray
    instr_engine: np.ndarray
    instr_latency: np.ndarray
    dep_prod: np.ndarray
    dep_cons: np.ndarray
    dep_k: np.ndarray
    trip_ptr: np.ndarray
    trips: np.ndarray
    eng_trip_ptr: np.ndarray | None = None
    eng_trips: np.ndarray | None = None
    # what the loader does with non-allocatable dependencies: 0 rejects,
    # 1 falls back to barriers at the end of the carrying loop's iterations
    nonalloc_policy: int = 0

    @property
    def divergent(self) -> bool:
        return self.eng_trip_ptr is not None

    def engine_trips(self, p: int, l: int, e: int) -> np.ndarray:
        """Trips of program p's loop l on engine e (program-local l)."""
        if self.eng_trip_ptr is None:
            g = int(self.prog_loop_ptr[p]) + l
            return self.trips[self.trip_ptr[g]:self.trip_ptr[g + 1]]
        r = self.row_base(p) + l * int(self.prog_n_engines[p]) + e
        return self.eng_trips[self.eng_trip_ptr[r]:self.eng_trip_ptr[r + 1]]

    def row_base(self, p: int) -> int:
        nl = np.diff(self.prog_loop_ptr[:p + 1]).astype(np.int64)
        return int((nl * self.prog_n_engines[:p].astype(np.int64)).sum())

    @property
    def n_loops(self) -> int:
        return int(self.loop_parent.shape[0])

    @property
    def n_instrs(self) -> int:
        return int(self.instr_loop.shape[0])

    @property
    def n_deps(self) -> int:
        return int(self.dep_prod.shape[0])

    def arrays(self):
        return {f.name: getattr(self, f.name) for f in fields(self)
                if f.name not in ("n_programs", "nonalloc_policy") and getattr(self, f.name) is not None}

    def copy(self) -> "Batch":
        return Batch(self.n_programs, **{k: v.copy() for k, v in self.arrays().items()},
                     nonalloc_policy=self.nonalloc_policy)

    def nbytes(self) -> int:
        return int(sum(v.nbytes for v in self.arrays().values()))

    def program(self, p: int) -> "Batch":
        """Program ``p`` alone, as a one-program batch."""
        return concat([self], programs=[(0, p)])


_lib = None


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        lib.synth_generate.restype = ctypes.c_int
        lib.synth_generate.argtypes = [ctypes.c_int32, ctypes.c_uint64, ctypes.c_int64,
                                       ctypes.c_int64, ctypes.POINTER(_CBatch)]
        lib.synth_generate_tree.restype = ctypes.c_int
        lib.synth_generate_tree.argtypes = [ctypes.POINTER(TreeParams), ctypes.c_uint64,
                                            ctypes.c_int64, ctypes.c_int64,
                                            ctypes.POINTER(_CBatch)]
        lib.synth_free.restype = None
        lib.synth_free.argtypes = [ctypes.POINTER(_CBatch)]
        _lib = lib
    return _lib


def _take(lib, cb: _CBatch) -> Batch:
    def arr(ptr, n, dt):
        if n == 0:
            return np.zeros(0, dtype=dt)
        return np.ctypeslib.as_array(ptr, shape=(n,)).astype(dt, copy=True)

    P = cb.n_programs
    try:
        return Batch(
            n_programs=P,
            prog_loop_ptr=arr(cb.prog_loop_ptr, P + 1, np.int32),
            prog_instr_ptr=arr(cb.prog_instr_ptr, P + 1, np.int32),
            prog_dep_ptr=arr(cb.prog_dep_ptr, P + 1, np.int32),
            prog_n_engines=arr(cb.prog_n_engines, P, np.int32),
            loop_parent=arr(cb.loop_parent, cb.n_loops, np.int32),
            loop_pos=arr(cb.loop_pos, cb.n_loops, np.int32),
            instr_loop=arr(cb.instr_loop, cb.n_instrs, np.int32),
            instr_pos=arr(cb.instr_pos, cb.n_instrs, np.int32),
            instr_engine=arr(cb.instr_engine, cb.n_instrs, np.int32),
            instr_latency=arr(cb.instr_latency, cb.n_instrs, np.int32),
            dep_prod=arr(cb.dep_prod, cb.n_deps, np.int32),
            dep_cons=arr(cb.dep_cons, cb.n_deps, np.int32),
            dep_k=arr(cb.dep_k, cb.n_deps, np.int32),
            trip_ptr=arr(cb.trip_ptr, cb.n_loops + 1, np.int64),
            trips=arr(cb.trips, cb.n_trips, np.int32),
        )
    finally:
        lib.synth_free(ctypes.byref(cb))


def generate(config, n_programs: int | None = None, first_program: int = 0,
             seed: int | None = None) -> Batch:
    """Programs ``first_program .. first_program+n_programs-1`` of a named config."""
    cfg, default_n = CONFIGS[config] if isinstance(config, str) else (int(config), 1)
    n = default_n if n_programs is None else int(n_programs)
    s = config_seed(cfg) if seed is None else int(seed)
    lib = _load()
    cb = _CBatch()
    rc = lib.synth_generate(cfg, ctypes.c_uint64(s & 0xFFFFFFFFFFFFFFFF), first_program, n,
                            ctypes.byref(cb))
    if rc != 0:
        raise RuntimeError(f"synth_generate failed with status {rc}")
    return _take(lib, cb)


def random_trees(seed: int, n_programs: int, params: TreeParams | None = None,
                 first_program: int = 0) -> Batch:
    """General random loop trees (branching, conditionals, sparse positions)."""
    lib = _load()
    cb = _CBatch()
    p = params if params is not None else tree_params()
    rc = lib.synth_generate_tree(ctypes.byref(p), ctypes.c_uint64(seed & 0xFFFFFFFFFFFFFFFF),
                                 first_program, n_programs, ctypes.byref(cb))
    if rc != 0:
        raise RuntimeError(f"synth_generate_tree failed with status {rc}")
    return _take(lib, cb)


def concat(batches, programs=None) -> Batch:
    """Concatenate batches, or pick ``programs`` = [(batch index, program id), ...]."""
    if programs is None:
        programs = [(bi, p) for bi, b in enumerate(batches) for p in range(b.n_programs)]
    parts = {k: [] for k in ("loop_parent", "loop_pos", "instr_loop", "instr_pos",
                             "instr_engine", "instr_latency", "dep_prod", "dep_cons", "dep_k",
                             "trips")}
    lp, ip, dp, ne, tp = [0], [0], [0], [], []
    trip_base = 0
    divergent = any(batches[bi].divergent for bi, _ in programs)
    etp, etrips, ebase = [], [], 0
    for bi, p in programs:
        b = batches[bi]
        if divergent:               # one row per (loop, engine), shared trips repeated
            for l in range(int(b.prog_loop_ptr[p + 1] - b.prog_loop_ptr[p])):
                for e in range(int(b.prog_n_engines[p])):
                    t = b.engine_trips(p, l, e)
                    etp.append(ebase)
                    etrips.append(t)
                    ebase += len(t)
        l0, l1 = int(b.prog_loop_ptr[p]), int(b.prog_loop_ptr[p + 1])
        x0, x1 = int(b.prog_instr_ptr[p]), int(b.prog_instr_ptr[p + 1])
        d0, d1 = int(b.prog_dep_ptr[p]), int(b.prog_dep_ptr[p + 1])
        for k in ("loop_parent", "loop_pos"):
            parts[k].append(getattr(b, k)[l0:l1])
        for k in ("instr_loop", "instr_pos", "instr_engine", "instr_latency"):
            parts[k].append(getattr(b, k)[x0:x1])
        for k in ("dep_prod", "dep_cons", "dep_k"):
            parts[k].append(getattr(b, k)[d0:d1])
        t0, t1 = int(b.trip_ptr[l0]), int(b.trip_ptr[l1])
        parts["trips"].append(b.trips[t0:t1])
        tp.append(b.trip_ptr[l0:l1] - t0 + trip_base)
        trip_base += t1 - t0
        lp.append(lp[-1] + l1 - l0)
        ip.append(ip[-1] + x1 - x0)
        dp.append(dp[-1] + d1 - d0)
        ne.append(int(b.prog_n_engines[p]))
    tp.append(np.array([trip_base], dtype=np.int64))

    def cat(xs, dt):
        return np.concatenate(xs).astype(dt) if xs else np.zeros(0, dtype=dt)

    return Batch(
        n_programs=len(programs),
        prog_loop_ptr=np.array(lp, dtype=np.int32),
        prog_instr_ptr=np.array(ip, dtype=np.int32),
        prog_dep_ptr=np.array(dp, dtype=np.int32),
        prog_n_engines=np.array(ne, dtype=np.int32),
        trip_ptr=cat(tp, np.int64),
        eng_trip_ptr=np.array(etp + [ebase], dtype=np.int64) if divergent else None,
        eng_trips=cat(etrips, np.int32) if divergent else None,
        nonalloc_policy=max((batches[bi].nonalloc_policy for bi, _ in programs), default=0),
        **{k: cat(v, np.int32) for k, v in parts.items()},
    )


def diverge(batch: Batch, seed: int, permille: int = 200, trip_hi: int | None = None) -> Batch:
    """Per-engine trip counts from a shared-trip batch: every engine starts
    from the shared trips, each (loop, engine) trip is moved by one (up or
    down, not below 0) with probability permille/1000, and a parent iteration
    that exists on one engine only gets a trip drawn uniformly in
    [0, trip_hi] (default: the loop's largest shared trip).  Engine 0 keeps
    the shared trips of loops whose parents did not diverge, so some
    programs stay aligned.  A pure function of (batch, seed, program id)."""
    etp, etrips, ebase = [], [], 0
    trips0, tp0 = [], [0]
    for p in range(batch.n_programs):
        rng = np.random.default_rng([int(seed) & 0xFFFFFFFF, p])
        l0, l1 = int(batch.prog_loop_ptr[p]), int(batch.prog_loop_ptr[p + 1])
        ne = int(batch.prog_n_engines[p])
        par = batch.loop_parent[l0:l1]
        rows = [[None] * ne for _ in range(l1 - l0)]
        for e in range(ne):
            total = {}
            for l in range(l1 - l0):
                base = batch.trips[batch.trip_ptr[l0 + l]:batch.trip_ptr[l0 + l + 1]]
                if l == 0:
                    t = np.array([1], dtype=np.int64)
                else:
                    n = total[int(par[l])]
                    hi = trip_hi if trip_hi is not None else (int(base.max()) if base.size else 2)
                    t = np.empty(n, dtype=np.int64)
                    m = min(n, base.size)
                    t[:m] = base[:m]
                    if n > m:
                        t[m:] = rng.integers(0, hi + 1, size=n - m)
                    move = rng.random(n) < permille / 1000.0
                    step = np.where(rng.random(n) < 0.5, -1, 1)
                    t = np.where(move, np.maximum(t + step, 0), t)
                total[l] = int(t.sum())
                rows[l][e] = t.astype(np.int32)
        for l in range(l1 - l0):
            for e in range(ne):
                etp.append(ebase)
                etrips.append(rows[l][e])
                ebase += rows[l][e].size
            trips0.append(rows[l][0])
            tp0.append(tp0[-1] + rows[l][0].size)
    b = batch.copy()
    b.trips = np.concatenate(trips0).astype(np.int32) if trips0 else np.zeros(0, np.int32)
    b.trip_ptr = np.array(tp0, dtype=np.int64)
    b.eng_trip_ptr = np.array(etp + [ebase], dtype=np.int64)
    b.eng_trips = np.concatenate(etrips).astype(np.int32) if etrips else np.zeros(0, np.int32)
    return b


class ProgramBuilder:
    """Hand-written programs (paper figures, edge cases) as batches.

    ``loop(parent, pos, trips)`` takes the trips of the new loop during each
    global iteration of its parent, in order; ``instr(loop, pos, engine,
    latency)`` and ``dep(prod, cons, k)`` return / take program-local ids.
    """

    def __init__(self, n_engines: int):
        self.ne = n_engines
        self.eng = {}
        self.loops = [(-1, 0, [1])]
        self.instrs = []
        self.deps = []

    def loop(self, parent: int, pos: int, trips, eng_trips=None) -> int:
        """``eng_trips``: optional list of per-engine trip lists (divergent
        trip counts); without it every engine runs ``trips``."""
        self.loops.append((parent, pos, list(trips)))
        if eng_trips is not None:
            self.eng[len(self.loops) - 1] = [list(t) for t in eng_trips]
        return len(self.loops) - 1

    def instr(self, loop: int, pos: int, engine: int, latency: int = 1) -> int:
        self.instrs.append((loop, pos, engine, latency))
        return len(self.instrs) - 1

    def dep(self, prod: int, cons: int, k: int = 0) -> int:
        self.deps.append((prod, cons, k))
        return len(self.deps) - 1

    def batch(self) -> Batch:
        trips, tp = [], [0]
        for _, _, t in self.loops:
            trips.extend(t)
            tp.append(len(trips))
        i32 = lambda xs: np.array(xs, dtype=np.int32)
        col = lambda rows, i: i32([r[i] for r in rows])
        return Batch(
            n_programs=1,
            prog_loop_ptr=i32([0, len(self.loops)]),
            prog_instr_ptr=i32([0, len(self.instrs)]),
            prog_dep_ptr=i32([0, len(self.deps)]),
            prog_n_engines=i32([self.ne]),
            loop_parent=col(self.loops, 0), loop_pos=col(self.loops, 1),
            instr_loop=col(self.instrs, 0), instr_pos=col(self.instrs, 1),
            instr_engine=col(self.instrs, 2), instr_latency=col(self.instrs, 3),
            dep_prod=col(self.deps, 0) if self.deps else i32([]),
            dep_cons=col(self.deps, 1) if self.deps else i32([]),
            dep_k=col(self.deps, 2) if self.deps else i32([]),
            trip_ptr=np.array(tp, dtype=np.int64), trips=i32(trips),
            eng_trip_ptr=self._eng_ptr(), eng_trips=self._eng_trips(),
        )

    def _eng_rows(self):
        return [self.eng.get(l, [t] * self.ne)[e] for l, (_, _, t) in enumerate(self.loops)
                for e in range(self.ne)]

    def _eng_ptr(self):
        if not self.eng:
            return None
        return np.concatenate([[0], np.cumsum([len(r) for r in self._eng_rows()])]).astype(np.int64)

    def _eng_trips(self):
        if not self.eng:
            return None
        return np.array([x for r in self._eng_rows() for x in r], dtype=np.int32)
