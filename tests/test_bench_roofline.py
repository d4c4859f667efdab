"""bench.py's roofline arithmetic on fixed inputs (no GPU): algorithmic
bytes and operations per launch, fractions against the given peaks, and the
profile-derived fields (DRAM traffic, warp-instruction issue) taken only
from a record of the current kernel sources."""
import types

import pytest

import bench


def _res():
    sz = types.SimpleNamespace(n_instances=1_000_000, n_pairs=400_000, n_pairs_padded=400_004,
                               struct_bytes=123_456)
    return {"per_kernel": {"thresholds": 0.5, "check": 0.6, "sim_barrier_free": 20.0, "sim_barrier": 18.0},
            "sizes": sz}


def test_roofline_arithmetic(monkeypatch):
    monkeypatch.setattr(bench, "profile_entry", lambda kernel, workload: None)
    dom, k = bench.roofline(_res(), 6000.0, "measured", 2000.0, "chain")
    alg = 4 * 400_004 + 123_456
    assert k["thresholds"]["alg_bytes"] == alg
    assert k["thresholds"]["achieved"] == pytest.approx(alg / 0.5e-3 / 1e9)
    assert k["check"]["frac"] == pytest.approx(alg / 0.6e-3 / 1e9 / 6000.0)
    ops = 12 * 1_000_000 + 2 * 400_000
    peak = 152 * 128 * 2000e6 / 1e12
    assert k["sim_barrier_free"]["alg_ops"] == ops
    assert k["sim_barrier_free"]["peak"] == pytest.approx(peak)
    assert k["sim_barrier"]["frac"] == pytest.approx(ops / 18e-3 / 1e12 / peak)
    # the dominant kernel is the slowest one, reported with its peak's source
    assert dom["kernel"] == "sim_barrier_free" and dom["bound"] == "alu"
    assert all(v["traffic"] is None for v in k.values()) and "issue" not in dom


def test_roofline_takes_profile_records(monkeypatch):
    recs = {"sim_barrier_free": {"dram_bytes_per_launch": 5_000_000, "warp_inst_per_instance": 15.0},
            "thresholds": {"dram_bytes_per_launch": 2_000_000}}
    monkeypatch.setattr(bench, "profile_entry", lambda kernel, workload: recs.get(kernel))
    dom, k = bench.roofline(_res(), 6000.0, "measured", 2000.0, "chain")
    assert k["thresholds"]["traffic"] == 2_000_000 and k["check"]["traffic"] is None
    issue = dom["issue"]
    assert issue["achieved"] == pytest.approx(15.0 * 1_000_000 / 20e-3 / 1e9)
    assert issue["peak"] == pytest.approx(152 * 4 * 2000e6 / 1e9)
    assert issue["frac"] == pytest.approx(issue["achieved"] / issue["peak"])


def test_profile_records_need_the_current_sources(monkeypatch):
    monkeypatch.setattr(bench, "kernel_hash", lambda *a, **k: "not-the-captured-hash")
    assert bench.traffic_for("thresholds", "chain") is None
    assert bench.profile_entry("sim_barrier_free", "chain") is None
