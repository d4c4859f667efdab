"""Piece-parallel simulation of large programs (a top-level body of one loop
L cut into runs of L's iterations on separate warps) against the oracle.

The loader splits a program when it is large against the batch; the floor
SYNCGB_SPLIT_MIN is lowered here so that small programs split too.  Random
trees wrapped in one loop of a few iterations (with their trips varied per
repetition) give pieces whose waits stay inside them and pieces whose waits
reach earlier pieces (dependencies once carried at the top level, now at L,
with an offset >= 1), which the validation sends to the whole-program sweep;
deadlocks and waits on later producers inside pieces do the same.  Every
result must equal the oracle's either way."""
import numpy as np
import pytest

import oracle
import workloads
from tests.test_gpu_parity import ALL_MODES, compare_all

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sg():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_13757_gb300 import build
    build.build()
    import paper_2608_13757_gb300 as m
    return m


def wrap_in_loop(batch, reps, seed):
    """Every program's top-level body moved into one loop L of `reps`
    iterations; the trips of the loops below are repeated per iteration of
    L, moved by -1, 0 or +1 (not below 0) per repetition."""
    rng = np.random.default_rng(seed)
    parts = []
    for p in range(batch.n_programs):
        one = batch.program(p)
        nl = one.n_loops
        par = np.concatenate([[-1, 0], np.where(one.loop_parent[1:] == 0, 1, one.loop_parent[1:] + 1)])
        pos = np.concatenate([[0, 0], one.loop_pos[1:]]).astype(np.int32)
        trips, tp = [np.array([1]), np.array([reps])], [0, 1, 2]
        totals = {0: 1, 1: reps}
        for l in range(1, nl):
            base = one.trips[one.trip_ptr[l]:one.trip_ptr[l + 1]]
            t = np.concatenate([np.maximum(base + rng.integers(-1, 2, size=base.size), 0) for _ in range(reps)]) \
                if totals[int(par[l + 1])] == reps * base.size else None
            if t is None:          # a parent whose iterations changed: draw its trips afresh
                n = totals[int(par[l + 1])]
                t = rng.integers(0, 4, size=n)
            trips.append(t)
            tp.append(tp[-1] + t.size)
            totals[l + 1] = int(t.sum())
        parts.append(workloads.Batch(
            n_programs=1, prog_loop_ptr=np.array([0, nl + 1], np.int32),
            prog_instr_ptr=one.prog_instr_ptr.copy(), prog_dep_ptr=one.prog_dep_ptr.copy(),
            prog_n_engines=one.prog_n_engines.copy(), loop_parent=par.astype(np.int32), loop_pos=pos,
            instr_loop=(one.instr_loop + 1).astype(np.int32), instr_pos=one.instr_pos.copy(),
            instr_engine=one.instr_engine.copy(), instr_latency=one.instr_latency.copy(),
            dep_prod=one.dep_prod.copy(), dep_cons=one.dep_cons.copy(), dep_k=one.dep_k.copy(),
            trip_ptr=np.array(tp, np.int64), trips=np.concatenate(trips).astype(np.int32)))
    return workloads.concat(parts)


@pytest.mark.parametrize("spec", ["0", "1"], ids=["probes", "speculation"])
@pytest.mark.parametrize("seed", range(3))
def test_pieces_random_trees(sg, seed, spec, monkeypatch):
    """Barrier-free pieces probed, or speculated (SYNCGB_SPLIT_SPEC=1)."""
    monkeypatch.setenv("SYNCGB_SPLIT_MIN", "1")
    monkeypatch.setenv("SYNCGB_SPLIT_SPEC", spec)
    base = workloads.random_trees(9500 + seed, 60, workloads.tree_params(
        engines_hi=5, loops_hi=5, body_hi=6, trip_hi=4, max_depth=3, max_deps_per_cons=2))
    batch = wrap_in_loop(base, 3 + seed, seed)
    h = sg.sync_load_programs(batch)
    assert h.sizes.n_split_programs > 0 and h.sizes.n_pieces > h.sizes.n_split_programs
    h.close()
    compare_all(sg, batch, timeline=True, modes=ALL_MODES,
                params=oracle.sim_params(ii=2, c_branch=3, c_regop=2, c_barrier=9))


@pytest.mark.parametrize("spec", ["0", "1"], ids=["probes", "speculation"])
@pytest.mark.parametrize("red", [dict(licm=1, cse=1), dict(trip_register_elision=1)])
def test_pieces_with_cost_switches(sg, red, spec, monkeypatch):
    monkeypatch.setenv("SYNCGB_SPLIT_MIN", "1")
    monkeypatch.setenv("SYNCGB_SPLIT_SPEC", spec)
    batch = wrap_in_loop(workloads.random_trees(9600, 60, workloads.tree_params(
        engines_hi=4, loops_hi=5, body_hi=6, trip_hi=4, max_depth=3)), 4, 7)
    compare_all(sg, batch, timeline=True, modes=ALL_MODES, params=oracle.sim_params(c_regop=2, **red))


@pytest.mark.parametrize("spec", ["0", "1"], ids=["probes", "speculation"])
def test_pieces_configs(sg, spec, monkeypatch):
    """The GEMM program and two attention programs split at the default
    floor (their 32 outer iterations are identical in shape, so speculation
    accepts most guesses); their results equal the oracle's."""
    monkeypatch.setenv("SYNCGB_SPLIT_SPEC", spec)
    for name, n in (("gemm", None), ("attention", 2)):
        batch = workloads.generate(name, n_programs=n)
        h = sg.sync_load_programs(batch)
        assert h.sizes.n_split_programs == batch.n_programs and h.sizes.n_pieces == 32 * batch.n_programs
        h.close()
        compare_all(sg, batch, timeline=name == "gemm", modes=ALL_MODES)


def test_pieces_refuse_waits_into_earlier_pieces(sg, monkeypatch):
    """Thresholds that name increments of earlier pieces (every per-loop
    value moved down by one iteration's increments where it stays positive)
    send the program to the whole-program sweep: still the oracle's results
    for those thresholds, deadlocks and all."""
    monkeypatch.setenv("SYNCGB_SPLIT_MIN", "1")
    batch = workloads.generate("gemm")
    h = sg.sync_load_programs(batch)
    idx = h.unpadded_index()
    import torch
    for mode in (oracle.COUNT, oracle.PERLOOP):
        want = oracle.thresholds(batch, mode)
        early = np.where(want > 300, want - 300, want).astype(np.int32)
        thr = sg.sync_eval_thresholds(h, mode)
        thr[torch.from_numpy(idx).to(thr.device)] = torch.from_numpy(early).to(thr.device)
        for v in (oracle.BARRIER_FREE, oracle.BARRIER):
            ref = oracle.simulate(batch, early, mode, v)
            r = sg.sync_simulate(h, mode, thr, variant=v)
            assert np.array_equal(r.status.cpu().numpy()[:1], ref.status)
            assert np.array_equal(r.makespan.cpu().numpy()[:1], ref.makespan)
            assert np.array_equal(r.checksum.cpu().numpy()[:1].view(np.uint64), ref.checksum)
    h.close()


@pytest.mark.parametrize("spec", ["0", "1"], ids=["probes", "speculation"])
def test_kernel_launch_count(sg, spec, monkeypatch):
    """The library's launch counter: one kernel per threshold and check
    call, two per simulation of unsplit programs (the sweep and the
    per-engine kernel), and the piece kernels on top where programs are
    split: barrier scheme validation, runs, composition and fixup;
    barrier-free validation, then probes (runs, composition) and/or
    speculation (start, four rounds of runs and acceptance), then fixup."""
    monkeypatch.setenv("SYNCGB_SPLIT_SPEC", spec)
    mode = oracle.PERLOOP
    for name, split in (("depth2", False), ("gemm", True)):
        batch = workloads.generate(name, n_programs=64 if name == "depth2" else None)
        h = sg.sync_load_programs(batch)
        assert (h.sizes.n_split_programs > 0) == split
        n0 = sg.kernel_launches()
        thr = sg.sync_eval_thresholds(h, mode)
        assert sg.kernel_launches() - n0 == 1
        sg.sync_check_minimal(h, mode, thr)
        assert sg.kernel_launches() - n0 == 2
        n0 = sg.kernel_launches()
        sg.sync_simulate(h, mode, thr, variant=oracle.BARRIER)
        assert sg.kernel_launches() - n0 == (2 + 4 if split else 2)
        n0 = sg.kernel_launches()
        sg.sync_simulate(h, mode, thr, variant=oracle.BARRIER_FREE)
        bf = sg.kernel_launches() - n0
        if not split:
            assert bf == 2
        elif spec == "1":
            assert bf == 2 + 1 + 1 + 4 * 2 + 1
        else:
            assert bf in (2 + 1 + 2 + 1, 2 + 1 + 2 + 9 + 1, 2 + 1 + 9 + 1)
        h.close()
