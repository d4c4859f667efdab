"""GPU parity of the barrier fallback for non-allocatable dependencies.

A batch loaded with SYNC_NONALLOC_BARRIER: nested producers with a forward
offset >= 1 or a backward offset >= 2 get no semaphore wait (wait value 0,
the checker's minimum) and their carrying loop ends every iteration with an
all-engine barrier.  Thresholds, check, barrier-free and barrier
simulations (array and fused, every mode, full timelines) must equal the
oracle's; the rejected combinations must fail loudly.
"""
import numpy as np
import pytest

import oracle
import workloads
from tests.test_fallback_pins import FAR, nested_program, with_policy
from tests.test_gpu_parity import _instances_per_program, gpu_thresholds, sim_params

pytestmark = pytest.mark.gpu

COUNT, PERLOOP, PERENGINE = oracle.COUNT, oracle.PERLOOP, oracle.PERENGINE


@pytest.fixture(scope="module")
def sg():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_13757_gb300 import build
    build.build()
    import paper_2608_13757_gb300 as m
    return m


def barrier_pairs(batch):
    """Per pair: does it belong to a barrier-fallback dependency."""
    cls = oracle.classify(batch).kase
    tot = np.zeros(batch.n_loops, dtype=np.int64)
    for l in range(batch.n_loops):
        tot[l] = batch.trips[batch.trip_ptr[l]:batch.trip_ptr[l + 1]].sum()
    out = []
    for p in range(batch.n_programs):
        l0, x0 = int(batch.prog_loop_ptr[p]), int(batch.prog_instr_ptr[p])
        for d in range(int(batch.prog_dep_ptr[p]), int(batch.prog_dep_ptr[p + 1])):
            n = int(tot[l0 + int(batch.instr_loop[x0 + int(batch.dep_cons[d])])])
            out.append(np.full(n, cls[d] == oracle.CASE_BARRIER))
    return np.concatenate(out) if out else np.zeros(0, dtype=bool)


def expected_thresholds(batch, mode):
    want = oracle.thresholds(batch, mode)
    want[barrier_pairs(batch)] = 0
    if mode != PERENGINE:                       # the register replay says the same
        assert np.array_equal(want, oracle.register_replay(batch, mode))
    return want


def compare_fallback(sg, batch, prm=None, modes=(COUNT, PERLOOP, PERENGINE)):
    prm = prm if prm is not None else oracle.sim_params()
    h = sg.sync_load_programs(batch)
    P = batch.n_programs
    ninst = oracle.sizes(batch)[1]
    ok_inst = None
    for mode in modes:
        thr, got = gpu_thresholds(sg, h, mode)
        want = expected_thresholds(batch, mode)
        assert np.array_equal(got, want), f"thresholds (mode {mode})"
        counts, fb = sg.sync_check_minimal(h, mode, thr)
        assert counts.cpu().tolist() == [0, 0] and fb.item() == -1, mode
        for v in (oracle.BARRIER_FREE, oracle.BARRIER):
            ref = oracle.simulate(batch, want, mode, v, prm, timeline=True)
            res = sg.sync_simulate(h, mode, thr, sim_params(prm), v, timeline=True)
            fused, fc, ff = sg.sync_simulate_fused(h, mode, sim_params(prm), v, timeline=True, check=True)
            assert fc.cpu().tolist() == [0, 0] and ff.item() == -1, (mode, v)
            ok_inst = np.repeat(ref.status == 0, _instances_per_program(batch))
            for name, r in (("array", res), ("fused", fused)):
                assert np.array_equal(r.status.cpu().numpy()[:P], ref.status), (name, mode, v)
                assert np.array_equal(r.makespan.cpu().numpy()[:P], ref.makespan), (name, mode, v)
                assert np.array_equal(r.checksum.cpu().numpy()[:P].view(np.uint64), ref.checksum), (name, mode, v)
                assert np.array_equal(r.issue.cpu().numpy()[:ninst][ok_inst], ref.issue[ok_inst]), (name, mode, v)
                assert np.array_equal(r.retire.cpu().numpy()[:ninst][ok_inst], ref.retire[ok_inst]), (name, mode, v)
    return h


@pytest.mark.parametrize("seed", range(3))
def test_fallback_random_trees(sg, seed):
    b = with_policy(workloads.random_trees(31000 + seed, 200, workloads.tree_params(**FAR)), 1)
    cls = oracle.classify(b).kase
    assert (cls == oracle.CASE_BARRIER).sum() > 50
    compare_fallback(sg, b, oracle.sim_params(ii=2, c_branch=3, c_regop=2, c_barrier=17))


def test_fallback_beside_sweep_programs(sg):
    """Fallback programs (per-engine kernel, barrier-free) in one batch with
    chain programs the sweep runs, and the hand-checked program."""
    b = workloads.concat([workloads.generate("chain", n_programs=64),
                          workloads.random_trees(31010, 60, workloads.tree_params(**FAR)),
                          nested_program(1), nested_program(2, backward=True)])
    compare_fallback(sg, with_policy(b, 1))


def test_fallback_hand_timeline(sg):
    b = with_policy(nested_program(1), 1)
    h = sg.sync_load_programs(b)
    thr, got = gpu_thresholds(sg, h, COUNT)
    assert got.tolist() == [0, 0, 0]
    r = sg.sync_simulate(h, COUNT, thr, sg.SimParams(), sg.SIM_BARRIER_FREE, timeline=True)
    assert r.issue.cpu().tolist()[:6] == [8, 57, 106, 8, 57, 106]
    assert r.retire.cpu().tolist()[:6] == [18, 67, 116, 9, 58, 107]
    assert r.makespan.cpu().tolist()[:1] == [148]


def test_fallback_check_minimum_zero_on_barrier_pairs(sg):
    b = with_policy(workloads.random_trees(31020, 80, workloads.tree_params(**FAR)), 1)
    h = sg.sync_load_programs(b)
    thr, got = gpu_thresholds(sg, h, PERLOOP)
    idx = h.unpadded_index()
    bar = barrier_pairs(b)
    assert bar.any()
    import torch
    junk = thr.clone()
    sel = torch.from_numpy(idx[bar]).to(junk.device)
    junk[sel] = 777                               # barriers enforce these: a wait over-synchronises
    counts, fb = sg.sync_check_minimal(h, PERLOOP, junk)
    assert counts.cpu().tolist() == [0, int(bar.sum())] and fb.item() == int(idx[bar][0])
    i = int(np.flatnonzero(~bar & (got > 0))[0])  # a waited pair below its minimum: unsafe
    junk[sel] = 0
    junk[int(idx[i])] = 0
    counts, fb = sg.sync_check_minimal(h, PERLOOP, junk)
    assert counts.cpu().tolist() == [1, 0] and fb.item() == int(idx[i])


def test_fallback_time_bound(sg):
    """The barrier-free bound counts the fallback barriers: c_barrier = 2^30
    with three iterations of S overflows (status 4) on both sides."""
    b = with_policy(nested_program(1), 1)
    prm = oracle.sim_params(c_barrier=1 << 30)
    want = expected_thresholds(b, COUNT)
    ref = oracle.simulate(b, want, COUNT, oracle.BARRIER_FREE, prm)
    h = sg.sync_load_programs(b)
    thr, _ = gpu_thresholds(sg, h, COUNT)
    r = sg.sync_simulate(h, COUNT, thr, sim_params(prm), sg.SIM_BARRIER_FREE)
    assert ref.status.tolist() == [oracle.SIM_OVERFLOW]
    assert r.status.cpu().tolist()[:1] == [sg.PROG_OVERFLOW]


def test_fallback_rejections(sg):
    with pytest.raises(sg.SyncError) as err:                 # default policy: rejected
        sg.sync_load_programs(nested_program(1))
    assert err.value.status == sg.ERR_NOT_ALLOCATABLE
    with pytest.raises(sg.SyncError) as err:                 # nested backward offset 0: no barrier helps
        sg.sync_load_programs(with_policy(nested_program(0, backward=True), 1))
    assert err.value.status == sg.ERR_NOT_ALLOCATABLE
    with pytest.raises(sg.SyncError) as err:                 # not a policy
        sg.sync_load_programs(with_policy(nested_program(1), 2))
    assert err.value.status == sg.ERR_ARG
    h = sg.sync_load_programs(with_policy(nested_program(1), 1))
    thr = sg.sync_eval_thresholds(h, PERENGINE)
    with pytest.raises(sg.SyncError) as err:                 # the unrolled program has no loops
        sg.sync_simulate(h, PERENGINE, thr, sg.SimParams(), sg.SIM_UNROLLED)
    assert err.value.status == sg.ERR_ARG
    pb = workloads.ProgramBuilder(2)                         # per-engine trips
    s = pb.loop(0, 0, [2])
    inner = pb.loop(s, 0, [1, 1], eng_trips=[[1, 1], [1, 2]])
    p = pb.instr(inner, 0, engine=1)
    c = pb.instr(s, 1, engine=0)
    pb.dep(p, c, 1)
    with pytest.raises(sg.SyncError) as err:
        sg.sync_load_programs(with_policy(pb.batch(), 1))
    assert err.value.status == sg.ERR_ARG


def test_fallback_loader_offsets(sg):
    """The fallback's zero-filled derived regions and unused consumer-grouped
    slots sit at offsets summed over the programs before them: each part of a
    batch, loaded alone, gives exactly its programs' share of the results."""
    from tests.test_gpu_parity import assert_parts_match
    b = with_policy(workloads.concat([
        workloads.random_trees(31030, 90, workloads.tree_params(**FAR)),
        workloads.generate("depth2", n_programs=12),
        workloads.random_trees(31031, 70, workloads.tree_params(**FAR))]), 1)
    assert_parts_match(sg, b, [0, 45, 90, 102, 172], (COUNT, PERLOOP, PERENGINE),
                       (sg.SIM_BARRIER_FREE, sg.SIM_BARRIER))

