"""The oracle over every program of a named configuration, on all host cores.

Test infrastructure: a configuration's programs are cut into contiguous
chunks, each chunk is generated on its own (a program depends only on the
configuration, the seed and its id, so a chunk equals the same range of the
full batch) and run through the oracle on a thread pool (ctypes releases the
GIL inside the oracle's C code).  The pair layout is dependency-major in
program order and the per-program outputs are in program order, so the
chunks' results concatenate into the full batch's.
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np

import oracle
import workloads


def chunks(n_programs: int, pieces: int | None = None):
    cores = len(os.sched_getaffinity(0))
    k = max(1, min(n_programs, pieces or 8 * cores))
    return [(n_programs * i // k, n_programs * (i + 1) // k) for i in range(k)
            if n_programs * (i + 1) // k > n_programs * i // k]


def run_config(name: str, mode: int, variants, params=None, n_programs: int | None = None):
    """(thresholds in pair layout, {variant: SimResult}) for programs
    0 .. n_programs-1 of configuration `name` (all of them by default)."""
    P = workloads.CONFIGS[name][1] if n_programs is None else n_programs
    prm = params if params is not None else oracle.sim_params()

    def work(rng):
        a, b = rng
        batch = workloads.generate(name, n_programs=b - a, first_program=a)
        thr = oracle.thresholds(batch, mode)
        sims = {v: oracle.simulate(batch, thr, mode, v, prm) for v in variants}
        return thr, sims

    with ThreadPoolExecutor(max_workers=len(os.sched_getaffinity(0))) as ex:
        parts = list(ex.map(work, chunks(P)))
    thr = np.concatenate([p[0] for p in parts]) if parts else np.zeros(0, np.int32)
    sims = {}
    for v in variants:
        sims[v] = oracle.SimResult(np.concatenate([p[1][v].makespan for p in parts]),
                                   np.concatenate([p[1][v].checksum for p in parts]),
                                   np.concatenate([p[1][v].status for p in parts]))
    return thr, sims


def unpadded_mask(pair_offsets: np.ndarray, pair_counts: np.ndarray) -> np.ndarray:
    """Boolean mask over a padded threshold array: True at the entries that
    are pairs (each dependency's segment starts at pair_offsets[d] and holds
    pair_counts[d] pairs, then padding up to the next segment)."""
    n = int(pair_offsets[-1]) if pair_offsets.size else 0
    if pair_counts.size == 0:
        return np.zeros(n, dtype=bool)
    pad = np.diff(pair_offsets) - pair_counts
    runs = np.empty(2 * pair_counts.size, dtype=np.int64)
    runs[0::2] = pair_counts
    runs[1::2] = pad
    flags = np.tile(np.array([True, False]), pair_counts.size)
    return np.repeat(flags, runs)
