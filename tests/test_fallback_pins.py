"""Pins of the oracle's barrier fallback for non-allocatable dependencies.

Sec. 5.2 keeps three dependency cases allocatable and sends any other nested
offset to the barrier-based scheme.  With the batch's nonalloc_policy set,
a producer nested below the carrying loop S with a forward offset k >= 1 or
a backward offset k >= 2 (its target lies in an earlier iteration of S) is
not waited on; instead every iteration of S ends with an all-engine barrier.
The pins: the classification, a timeline worked out by hand, the paper's
dependency-satisfaction condition Eq. (1) holding on every simulated
instance (the fallback must enforce what the wait would have), the barrier
scheme being unchanged by the fallback, the static bound's barrier term, and
the checker's minimum of 0 on barrier-enforced pairs, and the combinations
the fallback does not take.  No GPU.
"""
import numpy as np
import pytest

import oracle
import workloads

COUNT, PERLOOP, PERENGINE = oracle.COUNT, oracle.PERLOOP, oracle.PERENGINE

# random trees where many nested producers get far offsets, with trips long
# enough that such a consumer's target iteration exists
FAR = dict(nest_far_permille=500, dep_permille=700, trip_lo=2, trip_hi=5, k_max=1, cond_permille=0)


def with_policy(batch, policy):
    b = batch.copy()
    b.nonalloc_policy = policy
    return b


def nested_program(k, backward=False, lat_p=10, trip_s=3):
    """Two engines; S (trip trip_s) holds loop B (trip 1) with the producer on
    engine 1 and, after B (or before it: backward), the consumer on engine 0;
    one dependency producer -> consumer at offset k, carried at S."""
    pb = workloads.ProgramBuilder(2)
    s = pb.loop(0, 0, [trip_s])
    b = pb.loop(s, 1 if backward else 0, [1] * trip_s)
    p = pb.instr(b, 0, engine=1, latency=lat_p)
    c = pb.instr(s, 0 if backward else 1, engine=0, latency=1)
    pb.dep(p, c, k)
    return pb.batch()


def test_classification_of_nested_offsets():
    want = {  # (backward, k) -> case without / with the fallback
        (False, 0): (oracle.CASE_NEST_FWD, oracle.CASE_NEST_FWD),
        (False, 1): (oracle.CASE_NONE, oracle.CASE_BARRIER),
        (False, 3): (oracle.CASE_NONE, oracle.CASE_BARRIER),
        (True, 0): (oracle.CASE_NONE, oracle.CASE_NONE),      # unsatisfiable: the producer has not run
        (True, 1): (oracle.CASE_NEST_BWD, oracle.CASE_NEST_BWD),
        (True, 2): (oracle.CASE_NONE, oracle.CASE_BARRIER),
        (True, 4): (oracle.CASE_NONE, oracle.CASE_BARRIER),
    }
    for (bwd, k), (c0, c1) in want.items():
        b = nested_program(k, bwd)
        assert oracle.classify(with_policy(b, 0)).kase[0] == c0, (bwd, k)
        assert oracle.classify(with_policy(b, 1)).kase[0] == c1, (bwd, k)
    # a producer directly in S stays as it was: any offset is allocatable
    pb = workloads.ProgramBuilder(2)
    s = pb.loop(0, 0, [3])
    p = pb.instr(s, 0, engine=1)
    c = pb.instr(s, 1, engine=0)
    pb.dep(p, c, 3)
    assert oracle.classify(with_policy(pb.batch(), 1)).kase[0] == oracle.CASE_PS


def test_hand_timeline_forward_offset_one():
    """Default costs (ii 1, c_branch 1, c_regop 1, c_barrier 32), COUNT mode.
    Per S-iteration both engines pay S's start, B's statement and start; the
    producer (lat 10) and the consumer (no wait: the fallback) issue at the
    same cursor; the barrier then releases at max(t, last retire) + 32:
      S stmt 1, S start 4, B stmt 5, B start 8: issue 8, retires 18 / 9,
      release max(9, 18) + 32 = 50; next start 53, B 54, 57: issue 57,
      release 67 + 32 = 99; start 102, B 103, 106: issue 106, release 148."""
    b = with_policy(nested_program(1), 1)
    thr = oracle.register_replay(b, COUNT)
    assert thr.tolist() == [0, 0, 0]                          # no wait is emitted
    r = oracle.simulate(b, thr, COUNT, oracle.BARRIER_FREE, timeline=True)
    assert r.status.tolist() == [oracle.SIM_OK]
    assert r.issue.tolist() == [8, 57, 106, 8, 57, 106]       # producer, then consumer
    assert r.retire.tolist() == [18, 67, 116, 9, 58, 107]
    assert r.makespan.tolist() == [148]
    # Eq. (1): the consumer of S-iteration i needs the producer of i - 1
    assert r.issue[4] >= r.retire[0] and r.issue[5] >= r.retire[1]


def test_without_the_barrier_the_consumer_would_run_early():
    """The same program waited on by semaphore instead (no fallback; Eq. (1)
    thresholds): the consumer pays the 3 wait ops (COUNT) but no barrier, so
    it issues at 11, 22, 33 -- one producer latency apart -- where the
    fallback's barriers hold it to 8, 57, 106."""
    b0 = with_policy(nested_program(1), 0)
    r0 = oracle.simulate(b0, oracle.thresholds(b0, COUNT), COUNT, oracle.BARRIER_FREE, timeline=True)
    b1 = with_policy(nested_program(1), 1)
    r1 = oracle.simulate(b1, oracle.register_replay(b1, COUNT), COUNT, oracle.BARRIER_FREE, timeline=True)
    assert r0.status.tolist() == r1.status.tolist() == [oracle.SIM_OK]
    assert r0.makespan[0] < r1.makespan[0]
    assert r0.issue[3:].tolist() == [11, 22, 33]


def instance_offsets(batch):
    """Per global instruction, its first entry in the instance layout."""
    tot = np.zeros(batch.n_loops, dtype=np.int64)
    for l in range(batch.n_loops):
        tot[l] = batch.trips[batch.trip_ptr[l]:batch.trip_ptr[l + 1]].sum()
    off = np.zeros(batch.n_instrs + 1, dtype=np.int64)
    for p in range(batch.n_programs):
        l0 = int(batch.prog_loop_ptr[p])
        for x in range(int(batch.prog_instr_ptr[p]), int(batch.prog_instr_ptr[p + 1])):
            off[x + 1] = tot[l0 + int(batch.instr_loop[x])]
    return np.cumsum(off), tot


def assert_eq1_holds(batch, res):
    """Every consumer instance of every dependency issues no earlier than the
    retirement of the c-th producer instance, c = Eq. (1)'s count (programs
    that completed)."""
    ioff, tot = instance_offsets(batch)
    need = oracle.thresholds(batch, COUNT)             # Eq. (1), pair layout
    kase = oracle.classify(batch).kase
    pair = 0
    checked = [0, 0]                                   # semaphore-waited, barrier-enforced
    for p in range(batch.n_programs):
        l0, x0 = int(batch.prog_loop_ptr[p]), int(batch.prog_instr_ptr[p])
        for d in range(int(batch.prog_dep_ptr[p]), int(batch.prog_dep_ptr[p + 1])):
            cx, px = x0 + int(batch.dep_cons[d]), x0 + int(batch.dep_prod[d])
            n = int(tot[l0 + int(batch.instr_loop[cx])])
            if res.status[p] == oracle.SIM_OK:
                for g in range(n):
                    c = int(need[pair + g])
                    if c > 0:
                        assert res.issue[ioff[cx] + g] >= res.retire[ioff[px] + c - 1], (p, d, g)
                        checked[int(kase[d] == oracle.CASE_BARRIER)] += 1
            pair += n
    return checked


@pytest.mark.parametrize("mode", [COUNT, PERLOOP, PERENGINE])
@pytest.mark.parametrize("variant", [oracle.BARRIER_FREE, oracle.BARRIER])
def test_eq1_holds_under_the_fallback(mode, variant):
    b = with_policy(workloads.random_trees(20260, 300, workloads.tree_params(**FAR)), 1)
    cls = oracle.classify(b).kase
    assert (cls == oracle.CASE_BARRIER).sum() > 20 and (cls == oracle.CASE_NONE).sum() == 0
    thr = oracle.register_replay(b, mode) if mode != PERENGINE else oracle.thresholds(b, mode)
    if mode == PERENGINE:
        thr[np.concatenate([np.arange(s.start, s.stop) for s, k in zip(_slices(b), cls)
                            if k == oracle.CASE_BARRIER] + [np.zeros(0, dtype=np.int64)])] = 0
    r = oracle.simulate(b, thr, mode, variant, timeline=True)
    assert (r.status == oracle.SIM_OK).sum() > 250
    waited, by_barrier = assert_eq1_holds(b, r)
    assert waited > 1000 and by_barrier > 150


def _slices(batch):
    ioff, tot = instance_offsets(batch)
    out, off = [], 0
    for p in range(batch.n_programs):
        l0, x0 = int(batch.prog_loop_ptr[p]), int(batch.prog_instr_ptr[p])
        for d in range(int(batch.prog_dep_ptr[p]), int(batch.prog_dep_ptr[p + 1])):
            n = int(tot[l0 + int(batch.instr_loop[x0 + int(batch.dep_cons[d])])])
            out.append(slice(off, off + n))
            off += n
    return out


def test_barrier_scheme_is_unchanged_by_the_fallback():
    """Under the barrier scheme every iteration already ends with a barrier,
    so a barrier-fallback dependency waited on by semaphore (Eq. (1)
    thresholds, no fallback) gives the same schedule as the fallback."""
    base = workloads.random_trees(20261, 120, workloads.tree_params(**FAR))
    b0, b1 = with_policy(base, 0), with_policy(base, 1)
    for mode in (COUNT, PERLOOP):
        t0 = oracle.thresholds(b0, mode)
        r0 = oracle.simulate(b0, t0, mode, oracle.BARRIER, timeline=True)
        r1 = oracle.simulate(b1, oracle.register_replay(b1, mode), mode, oracle.BARRIER, timeline=True)
        assert np.array_equal(r0.status, r1.status)
        assert np.array_equal(r0.makespan, r1.makespan)
        assert np.array_equal(r0.checksum, r1.checksum)


def test_check_on_barrier_pairs_and_replay_matches_eq1_elsewhere():
    b = with_policy(workloads.random_trees(20262, 120, workloads.tree_params(**FAR)), 1)
    cls = oracle.classify(b).kase
    for mode in (COUNT, PERLOOP):
        rep = oracle.register_replay(b, mode)
        eq1 = oracle.thresholds(b, mode)
        bar = np.zeros(rep.shape[0], dtype=bool)
        for s, k in zip(_slices(b), cls):
            bar[s] = k == oracle.CASE_BARRIER
        assert bar.any() and (rep[bar] == 0).all()
        assert np.array_equal(rep[~bar], eq1[~bar])            # Thm. 1 on the allocatable pairs
        assert oracle.check(b, rep, mode)[:2] == (0, 0)
        junk = rep.copy()
        junk[bar] = 12345                  # a barrier enforces these: any wait is one too many
        assert oracle.check(b, junk, mode)[:2] == (0, int(bar.sum()))
        eq1_there = rep.copy()
        eq1_there[bar] = eq1[bar]          # Eq. (1)'s count waited on as well: redundant
        assert oracle.check(b, eq1_there, mode)[:2] == (0, int((eq1[bar] > 0).sum()))


def test_bound_counts_the_fallback_barriers():
    """c_barrier = 2^30 and three iterations of S: the barrier-free bound
    passes INT32_MAX only through the fallback's three barriers."""
    b0, b1 = with_policy(nested_program(1), 0), with_policy(nested_program(1), 1)
    prm = oracle.sim_params(c_barrier=1 << 30)
    r0 = oracle.simulate(b0, oracle.thresholds(b0, COUNT), COUNT, oracle.BARRIER_FREE, params=prm)
    r1 = oracle.simulate(b1, oracle.register_replay(b1, COUNT), COUNT, oracle.BARRIER_FREE, params=prm)
    assert r0.status.tolist() == [oracle.SIM_OK]
    assert r1.status.tolist() == [oracle.SIM_OVERFLOW] and r1.makespan.tolist() == [-1]
    two = with_policy(nested_program(1, trip_s=1), 1)          # one barrier: fits
    r2 = oracle.simulate(two, oracle.register_replay(two, COUNT), COUNT, oracle.BARRIER_FREE, params=prm)
    assert r2.status.tolist() == [oracle.SIM_OK]


def test_fallback_rejected_with_unrolled_and_per_engine_trips():
    b = with_policy(nested_program(1), 1)
    thr = oracle.thresholds(b, PERENGINE)
    with pytest.raises(oracle.OracleError):
        oracle.simulate(b, thr, PERENGINE, oracle.UNROLLED)
    pb = workloads.ProgramBuilder(2)
    s = pb.loop(0, 0, [2])
    inner = pb.loop(s, 0, [1, 1], eng_trips=[[1, 1], [1, 2]])
    p = pb.instr(inner, 0, engine=1)
    c = pb.instr(s, 1, engine=0)
    pb.dep(p, c, 1)
    d = with_policy(pb.batch(), 1)
    with pytest.raises(oracle.OracleError):
        oracle.simulate(d, np.zeros(2, dtype=np.int32), COUNT, oracle.BARRIER_FREE)
