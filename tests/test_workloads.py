"""The seeded input generator gives the same programs on every machine: the
CPU oracle's tests, the GPU parity tests and the benchmark run on different
hosts (x86 here, Arm next to the GPU) and must see the same batches."""
import os

from tests.golden import workload_fingerprints as wf

HERE = os.path.dirname(os.path.abspath(__file__))


def stored():
    out = {}
    with open(os.path.join(HERE, "golden", "workload_fingerprints.dat")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            key, fp = line.rsplit(":", 1)
            out[key.strip()] = fp.strip()
    return out


def test_generated_batches_match_stored_fingerprints():
    want = stored()
    got = dict(wf.entries())
    assert got == want
