"""Writes workload_fingerprints.dat: a SHA-256 prefix of every array of a few
generated input batches.  The generator's programs must not depend on the
machine that builds it (compiler, target, char signedness); the test
tests/test_workloads.py recomputes these and compares.

    python tests/golden/workload_fingerprints.py
"""
import hashlib
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))
import workloads  # noqa: E402

FIELDS = ("prog_loop_ptr", "prog_instr_ptr", "prog_dep_ptr", "prog_n_engines", "loop_parent", "loop_pos",
          "instr_loop", "instr_pos", "instr_engine", "instr_latency", "dep_prod", "dep_cons", "dep_k",
          "trip_ptr", "trips")

CASES = [("small", 0, 0), ("depth2", 16, 0), ("gemm", 0, 0), ("attention", 1, 0),
         ("chain", 64, 0), ("chain", 1, 38025), ("syncbound", 16, 0)]
TREES = [(5, 20, {}), (77, 20, {"any_k": 1, "k_max": 3})]


def fingerprint(b) -> str:
    m = hashlib.sha256()
    for f in FIELDS:
        a = np.ascontiguousarray(getattr(b, f))
        m.update(f.encode())
        m.update(a.tobytes())
    return m.hexdigest()[:16]


def entries():
    for name, n, first in CASES:
        b = workloads.generate(name, n_programs=n or None, first_program=first)
        yield f"{name} {n} {first}", fingerprint(b)
    for seed, n, kw in TREES:
        b = workloads.random_trees(seed, n, workloads.tree_params(**kw))
        yield f"trees {seed} {n} {','.join(f'{k}={v}' for k, v in kw.items()) or '-'}", fingerprint(b)


if __name__ == "__main__":
    with open(os.path.join(HERE, "workload_fingerprints.dat"), "w") as f:
        f.write("# input batches of the seeded generator (workloads/synth.c); written by\n")
        f.write("# tests/golden/workload_fingerprints.py\n")
        for key, fp in entries():
            f.write(f"{key}: {fp}\n")
