"""Pins of the CPU oracle to facts fixed outside it.

Each test ties an oracle function to something other than the oracle itself:
values the paper prints for a worked example (tests/golden), closed forms on
single loops and nests, the paper's per-loop identity Eq. (4), exhaustive
brute force, the paper's register mechanism (Thm. 1 consequence), a second
statement of the timing model (tests/timing_model.py), and invariants of the
timing model.  None of these needs a GPU.
"""
import numpy as np
import pytest

import oracle
import workloads
from tests import golden_io
from tests import timing_model

COUNT, PERLOOP, PERENGINE = oracle.COUNT, oracle.PERLOOP, oracle.PERENGINE


def pair_slices(batch):
    """Per dependency, the slice of the pair layout it owns."""
    cls = oracle.classify(batch)
    out, off = [], 0
    for d in range(batch.n_deps):
        p = int(np.searchsorted(batch.prog_dep_ptr, d, side="right") - 1)
        x = int(batch.dep_cons[d]) + int(batch.prog_instr_ptr[p])
        l = int(batch.instr_loop[x]) + int(batch.prog_loop_ptr[p])
        n = loop_totals(batch)[l]
        out.append(slice(off, off + n))
        off += n
    return out


def loop_totals(batch):
    tot = np.zeros(batch.n_loops, dtype=np.int64)
    for p in range(batch.n_programs):
        l0, l1 = batch.prog_loop_ptr[p], batch.prog_loop_ptr[p + 1]
        for l in range(l0, l1):
            seg = batch.trips[batch.trip_ptr[l]:batch.trip_ptr[l + 1]]
            tot[l] = int(seg.sum())
    return tot


# ------------------------------------------------------------ golden values

@pytest.mark.parametrize("name", golden_io.all_names())
def test_golden_worked_examples(name):
    batch, expects = golden_io.load(name)
    sl = pair_slices(batch)
    for mode_name, d, want in expects:
        mode = COUNT if mode_name == "count" else PERLOOP
        for fn in (oracle.thresholds, oracle.thresholds_bruteforce, oracle.register_replay):
            got = fn(batch, mode)[sl[d]]
            assert got.tolist() == want, (name, fn.__name__, mode_name)


def test_motivating_example_timeline():
    """Sec. 2: with the barrier-free allocation, the third issue of I2 waits for
    the first completion of I3 and nothing else waits; the pre- and post-loop
    work of engine 0 runs back to back (Fig. 1b)."""
    batch, _ = golden_io.load("motivating_example.txt")
    thr = oracle.thresholds(batch, COUNT)
    zero = oracle.sim_params(ii=1, c_branch=0, c_regop=0, c_wait_ops_count=0,
                             c_wait_ops_perloop=0, c_barrier=0)
    r = oracle.simulate(batch, thr, COUNT, oracle.BARRIER_FREE, zero, timeline=True)
    assert r.status[0] == 0
    # instance layout: I0, I1 (1 each), I2 (3), I3 (3), I4, I5
    iss, ret = r.issue, r.retire
    i2 = slice(2, 5)
    i3 = slice(5, 8)
    assert iss[i2][2] >= ret[i3][0]
    assert iss[i2][2] == max(ret[i3][0], iss[i2][1] + 1)
    # engine 0 (I0, I5) never waits: I5 issues one cycle after I0
    assert iss[9] == iss[0] + 1


# ------------------------------------------------------------ closed forms

@pytest.mark.parametrize("trip,k", [(1, 0), (5, 0), (7, 1), (7, 2), (9, 5), (3, 4)])
def test_closed_form_single_loop(trip, k):
    """One loop under the top-level loop, producer and consumer directly in it:
    the g-th consumer instance (1-based) waits for max(0, g - k) completions."""
    b = workloads.ProgramBuilder(2)
    L = b.loop(0, 0, [trip])
    p = b.instr(L, 0, 0)
    c = b.instr(L, 1, 1)
    b.dep(p, c, k)
    batch = b.batch()
    want = [max(0, g - k) for g in range(1, trip + 1)]
    assert oracle.thresholds(batch, COUNT).tolist() == want
    assert oracle.thresholds_bruteforce(batch, COUNT).tolist() == want


@pytest.mark.parametrize("outer,m", [(1, 1), (4, 3), (6, 1), (5, 7)])
def test_closed_form_nested_forward(outer, m):
    """Producer in an inner loop of constant trip m, consumer after it in the
    outer loop (forward, offset 0): the wait in outer iteration g is m*g."""
    b = workloads.ProgramBuilder(2)
    A = b.loop(0, 0, [outer])
    B = b.loop(A, 0, [m] * outer)
    p = b.instr(B, 0, 0)
    c = b.instr(A, 1, 1)
    b.dep(p, c, 0)
    batch = b.batch()
    want = [m * g for g in range(1, outer + 1)]
    assert oracle.thresholds(batch, COUNT).tolist() == want
    assert oracle.register_replay(batch, COUNT).tolist() == want


def test_closed_form_top_level_offsets():
    """Carried at the top-level loop (runs once): offset 0 counts every
    earlier producer instance, any positive offset underflows."""
    b = workloads.ProgramBuilder(2)
    A = b.loop(0, 0, [5])
    p = b.instr(A, 0, 0)
    c0 = b.instr(0, 1, 1)
    c1 = b.instr(0, 2, 1)
    b.dep(p, c0, 0)
    b.dep(p, c1, 1)
    batch = b.batch()
    assert oracle.thresholds(batch, COUNT).tolist() == [5, 0]
    assert oracle.thresholds_bruteforce(batch, COUNT).tolist() == [5, 0]


@pytest.mark.parametrize("N", range(1, 9))
def test_per_loop_identity_eq4(N):
    """Eq. (4): after the K-th of N same-engine instructions of a loop body
    retires in iteration r, the shared semaphore holds N*r - (N - K).  Checked
    for every K and r: the per-loop threshold equals that value, and in the
    oracle's semaphore machine the consumer issues exactly when that producer
    instance retires (it neither waits for more nor for less)."""
    R = 4
    for K in range(1, N + 1):
        b = workloads.ProgramBuilder(2)
        A = b.loop(0, 0, [R])
        xs = [b.instr(A, i, 0, latency=3 + 5 * i) for i in range(N)]
        c = b.instr(A, N, 1)
        b.dep(xs[K - 1], c, 0)
        batch = b.batch()
        thr = oracle.thresholds(batch, PERLOOP)
        assert thr.tolist() == [N * r - (N - K) for r in range(1, R + 1)]
        zero = oracle.sim_params(c_branch=0, c_regop=0, c_wait_ops_count=0,
                                 c_wait_ops_perloop=0)
        res = oracle.simulate(batch, thr, PERLOOP, oracle.BARRIER_FREE, zero, timeline=True)
        # instance layout: N producers x R, then the consumer x R
        prod_ret = res.retire[(K - 1) * R:K * R]
        cons_iss = res.issue[N * R:(N + 1) * R]
        want, t = [], 0
        for r in range(R):
            want.append(max(t, int(prod_ret[r])))
            t = want[-1] + 1
        assert cons_iss.tolist() == want


def test_per_loop_decoding_is_exact():
    """T = 0 exactly when c = 0; otherwise T + N - K is a multiple of N and
    (T + N - K) / N = c (the per-loop value decodes back to the count)."""
    for seed in range(20):
        batch = workloads.random_trees(seed, 10)
        cls = oracle.classify(batch)
        tc = oracle.thresholds(batch, COUNT)
        tp = oracle.thresholds(batch, PERLOOP)
        for d, sl in enumerate(pair_slices(batch)):
            N, K = int(cls.N[d]), int(cls.K[d])
            c, T = tc[sl].astype(np.int64), tp[sl].astype(np.int64)
            assert ((T == 0) == (c == 0)).all()
            nz = c > 0
            assert ((T[nz] + N - K) % N == 0).all()
            assert ((T[nz] + N - K) // N == c[nz]).all()


# ---------------------------------------------- definitions agree (Thm. 1)

@pytest.mark.parametrize("mode", [COUNT, PERLOOP])
def test_bruteforce_counting_and_registers_agree(mode):
    """Eq. (1) by pairwise lexicographic comparison, Eq. (1) by counting, and
    the paper's registers (Eq. 2, 3, 5) replayed per engine give the same
    value on every pair of 1500 random allocatable programs."""
    for seed in range(150):
        batch = workloads.random_trees(seed, 10)
        a = oracle.thresholds_bruteforce(batch, mode)
        b = oracle.thresholds(batch, mode)
        r = oracle.register_replay(batch, mode)
        assert (a == b).all(), seed
        assert (a == r).all(), seed


def test_registers_differ_outside_allocatable_subset():
    """Offsets outside the allocatable cases are classified as such, and the
    register formula is then not the minimum (so the restriction matters)."""
    seen_diff = 0
    for seed in range(60):
        batch = workloads.random_trees(seed, 10, workloads.tree_params(any_k=1, k_max=3))
        cls = oracle.classify(batch)
        a = oracle.thresholds_bruteforce(batch, COUNT)
        r = oracle.register_replay(batch, COUNT)
        for d, sl in enumerate(pair_slices(batch)):
            if cls.kase[d] == oracle.CASE_NONE:
                assert (r[sl] == -1).all()
                continue
            assert (a[sl] == r[sl]).all()
        # a non-allocatable nested offset evaluated with the nested formula
        seen_diff += int((cls.kase == oracle.CASE_NONE).sum())
    assert seen_diff > 0


def test_classification_cases():
    """Sec. 5.2 cases on hand-built programs."""
    def one(prod_where, cons_where, k, same_engine=False):
        b = workloads.ProgramBuilder(2)
        A = b.loop(0, 0, [3])
        B = b.loop(A, 5, [2, 2, 2])
        loops = {"A": A, "B": B}
        p = b.instr(loops[prod_where[0]], prod_where[1], 0)
        c = b.instr(loops[cons_where[0]], cons_where[1], 0 if same_engine else 1)
        b.dep(p, c, k)
        return int(oracle.classify(b.batch()).kase[0])
    C = oracle
    # producer nested in B, consumer after B in A: forward, offset 0 only
    assert one(("B", 0), ("A", 9), 0) == C.CASE_NEST_FWD
    assert one(("B", 0), ("A", 9), 1) == C.CASE_NONE
    # consumer before B: backward, offset 1 only
    assert one(("B", 0), ("A", 1), 1) == C.CASE_NEST_BWD
    assert one(("B", 0), ("A", 1), 0) == C.CASE_NONE
    assert one(("B", 0), ("A", 1), 2) == C.CASE_NONE
    # producer in S: any offset; backward offset 0 only across engines
    assert one(("A", 9), ("A", 1), 0) == C.CASE_PS
    assert one(("A", 9), ("A", 1), 0, same_engine=True) == C.CASE_NONE
    assert one(("A", 9), ("A", 1), 1, same_engine=True) == C.CASE_PS
    assert one(("A", 1), ("B", 0), 0, same_engine=True) == C.CASE_PS
    assert one(("A", 9), ("B", 0), 0, same_engine=True) == C.CASE_NONE


# ------------------------------------------------- per-engine allocation

def engine_streams(batch, p):
    """Program p's dynamic instruction stream of every engine, in program
    order, as lists of (program-local instruction, global iteration of its
    loop): a direct walk of the loop tree with the actual trips."""
    l0, l1 = int(batch.prog_loop_ptr[p]), int(batch.prog_loop_ptr[p + 1])
    x0, x1 = int(batch.prog_instr_ptr[p]), int(batch.prog_instr_ptr[p + 1])
    nl = l1 - l0
    body = [[] for _ in range(nl)]
    for x in range(x1 - x0):
        body[int(batch.instr_loop[x0 + x])].append((int(batch.instr_pos[x0 + x]), "x", x))
    for l in range(1, nl):
        body[int(batch.loop_parent[l0 + l])].append((int(batch.loop_pos[l0 + l]), "l", l))
    for b in body:
        b.sort()
    trips = [batch.trips[batch.trip_ptr[l0 + l]:batch.trip_ptr[l0 + l + 1]] for l in range(nl)]
    nxt = [0] * nl
    nxt[0] = 1
    streams = {e: [] for e in range(int(batch.prog_n_engines[p]))}

    def run(l, g):
        for _, kind, i in body[l]:
            if kind == "x":
                streams[int(batch.instr_engine[x0 + i])].append((i, g))
            else:
                for _ in range(int(trips[i][g])):
                    gm = nxt[i]
                    nxt[i] += 1
                    run(i, gm)
    run(0, 0)
    return streams


def test_perengine_is_the_producer_ordinal_in_its_engine_stream():
    """Sec. 6.1: one semaphore per engine counts all its retirements, so the
    wait value is the 1-based position of the producer's c-th instance (c from
    Eq. 1) in its engine's dynamic stream; checked against a direct walk."""
    for seed in range(60):
        batch = workloads.random_trees(seed, 6)
        count = oracle.thresholds(batch, COUNT)
        per_engine = oracle.thresholds(batch, PERENGINE)
        assert np.array_equal(per_engine, oracle.thresholds_bruteforce(batch, PERENGINE))
        sl = pair_slices(batch)
        d = 0
        for p in range(batch.n_programs):
            streams = engine_streams(batch, p)
            pos = {e: {inst: k + 1 for k, inst in enumerate(st)} for e, st in streams.items()}
            x0 = int(batch.prog_instr_ptr[p])
            for _ in range(int(batch.prog_dep_ptr[p + 1] - batch.prog_dep_ptr[p])):
                px = int(batch.dep_prod[d])
                e = int(batch.instr_engine[x0 + px])
                want = [pos[e][(px, c - 1)] if c > 0 else 0 for c in count[sl[d]]]
                assert per_engine[sl[d]].tolist() == want, (seed, d)
                d += 1


def test_perengine_reduces_to_perloop_when_alone_on_the_engine():
    """When the producer's loop is the only place its engine has datapath
    instructions and that loop sits directly under the top level, the engine
    counter is the per-(loop, engine) counter: per-engine = per-loop (Eq. 5)."""
    for trips in ([5], [3, 0, 4], [1, 7]):
        b = workloads.ProgramBuilder(2)
        A = b.loop(0, 1, trips[:1])
        b.instr(0, 0, 1)                   # engine 1 only outside the loop
        p0 = b.instr(A, 0, 0)
        p1 = b.instr(A, 2, 0)
        c0 = b.instr(A, 1, 1)
        c1 = b.instr(A, 3, 1)
        b.dep(p0, c0, 0)
        b.dep(p1, c1, 1)
        b.dep(p1, c0, 2)
        batch = b.batch()
        assert np.array_equal(oracle.thresholds(batch, PERENGINE), oracle.thresholds(batch, PERLOOP))


def test_perengine_bounds():
    """The c-th producer instance is at least the c-th instruction of its
    engine, exactly so when the producer is its engine's only instruction;
    0 exactly when c = 0."""
    for seed in range(40):
        batch = workloads.random_trees(seed, 6)
        c = oracle.thresholds(batch, COUNT).astype(np.int64)
        t = oracle.thresholds(batch, PERENGINE).astype(np.int64)
        assert ((c == 0) == (t == 0)).all()
        assert (t >= c).all()
    b = workloads.ProgramBuilder(2)
    A = b.loop(0, 0, [6])
    B = b.loop(A, 1, [2, 0, 3, 1, 1, 2])
    p = b.instr(B, 0, 0)                   # engine 0's only instruction
    x = b.instr(A, 2, 1)
    b.dep(p, x, 0)
    batch = b.batch()
    assert np.array_equal(oracle.thresholds(batch, PERENGINE), oracle.thresholds(batch, COUNT))


def test_perengine_nondecreasing_where_nonzero():
    """For a fixed dependency the engine ordinal grows with c, so it is
    nondecreasing over the pairs where it is nonzero (the c-xi invariant)."""
    for seed in range(40):
        batch = workloads.random_trees(seed, 6)
        t = oracle.thresholds(batch, PERENGINE)
        for s in pair_slices(batch):
            nz = t[s][t[s] > 0]
            assert (np.diff(nz) >= 0).all()


# ---------------------------------------------------------------- checker

@pytest.mark.parametrize("mode", [COUNT, PERLOOP, PERENGINE])
def test_checker_counts_planted_errors(mode):
    batch = workloads.generate("depth2", n_programs=8)
    thr = oracle.thresholds(batch, mode)
    assert oracle.check(batch, thr, mode) == (0, 0, -1)
    rng = np.random.default_rng(7)
    idx = np.sort(rng.choice(thr.size, size=40, replace=False))
    bad = thr.copy()
    up, down = idx[::2], idx[1::2]
    bad[up] += 1
    bad[down] -= 1
    unsafe, over, first = oracle.check(batch, bad, mode)
    assert (unsafe, over, first) == (down.size, up.size, int(idx[0]))


# ------------------------------------------------------------ timing model

ZERO = dict(c_branch=0, c_regop=0, c_wait_ops_count=0, c_wait_ops_perloop=0)


@pytest.mark.parametrize("T,lat,cbar", [(1, 1, 32), (5, 3, 32), (16, 7, 5), (9, 1, 0)])
def test_timing_closed_form_one_engine(T, lat, cbar):
    """One engine, one loop of T iterations, one instruction, no control cost:
    barrier-free makespan = T - 1 + lat (pipelined issue every cycle);
    barrier scheme = T*(lat + c_barrier) + c_barrier (entry barrier plus a
    drained barrier after every iteration)."""
    b = workloads.ProgramBuilder(1)
    L = b.loop(0, 0, [T])
    b.instr(L, 0, 0, latency=lat)
    batch = b.batch()
    thr = np.zeros(0, dtype=np.int32)
    prm = oracle.sim_params(c_barrier=cbar, **ZERO)
    bf = oracle.simulate(batch, thr, COUNT, oracle.BARRIER_FREE, prm)
    bb = oracle.simulate(batch, thr, COUNT, oracle.BARRIER, prm)
    assert bf.makespan[0] == T - 1 + lat
    assert bb.makespan[0] == T * (lat + cbar) + cbar


def test_timing_straight_line_fig3():
    """Fig. 3: I2 waits for I1 (s0 >= 2).  Engine 0 issues I0 at 0, I1 at 1;
    I1 retires at max(1 + lat1, retire of I0); I2 issues then."""
    batch, _ = golden_io.load("fig3_straight_line.txt")
    batch.instr_latency[:] = [4, 2, 3, 1]
    thr = oracle.thresholds(batch, PERLOOP)
    prm = oracle.sim_params(**ZERO)
    r = oracle.simulate(batch, thr, PERLOOP, oracle.BARRIER_FREE, prm, timeline=True)
    assert r.issue.tolist() == [0, 1, 4, 5]      # I1 retires at max(3, 4) = 4
    assert r.retire.tolist() == [4, 4, 7, 7]
    assert r.makespan[0] == 7


def _random_batches(n=40, **kw):
    for seed in range(n):
        yield seed, workloads.random_trees(seed, 1, workloads.tree_params(**kw))


def loop_depths(batch):
    """Depth of every loop of a one-program batch (top level 0)."""
    dep = [0] * batch.n_loops
    for l in range(1, batch.n_loops):
        dep[l] = dep[int(batch.loop_parent[l])] + 1
    return dep


def wait_ops(batch, mode, prm):
    """Wait-value ops of each dependency (Table 1): 3 / 5 per wait, and for a
    per-engine wait one more term per loop strictly between the top level and
    the producer's loop (Sec. 6.1's path sum)."""
    if mode == COUNT:
        return prm.c_wait_ops_count
    if mode == PERLOOP:
        return prm.c_wait_ops_perloop
    dep = loop_depths(batch)
    lvl = [max(0, dep[int(batch.instr_loop[int(batch.dep_prod[d])])] - 1) for d in range(batch.n_deps)]
    return lambda d: prm.c_wait_ops_perloop + prm.c_wait_ops_perengine_level * lvl[d]


@pytest.mark.parametrize("mode,variant", [(COUNT, oracle.BARRIER_FREE), (COUNT, oracle.BARRIER),
                                          (PERLOOP, oracle.BARRIER_FREE), (PERLOOP, oracle.BARRIER),
                                          (PERENGINE, oracle.BARRIER_FREE), (PERENGINE, oracle.BARRIER),
                                          (PERENGINE, oracle.UNROLLED)])
def test_timing_matches_recursive_statement(mode, variant):
    """The event-stepped semaphore machine (waits on semaphore values, per
    mode: per producer, per (loop, engine), or per engine counting every
    retirement) and the recursive max-plus statement (waits on the c-th
    producer retirement) give identical makespans, checksums and timelines."""
    prm = oracle.sim_params(ii=2, c_branch=3, c_regop=1, c_barrier=7, c_wait_ops_perengine_level=2)
    n = 0
    for seed, batch in _random_batches(60):
        thr = oracle.thresholds(batch, mode)
        thr_c = oracle.thresholds(batch, COUNT)
        r = oracle.simulate(batch, thr, mode, variant, prm, timeline=True)
        assert r.status[0] == 0
        ms, chk, tl = timing_model.simulate(batch, thr_c, prm, variant == oracle.BARRIER,
                                            wait_ops(batch, mode, prm), unrolled=variant == oracle.UNROLLED)
        assert r.makespan[0] == ms, seed
        assert int(r.checksum[0]) == chk, seed
        off = 0
        tot = loop_totals(batch)
        for x in range(batch.n_instrs):
            for g in range(int(tot[batch.instr_loop[x]])):
                assert (r.issue[off + g], r.retire[off + g]) == tl[(x, g)]
            off += int(tot[batch.instr_loop[x]])
        n += 1
    assert n == 60


def test_unrolled_and_per_engine_cost_order():
    """Same waits, costs only removed or added (max-plus monotonicity): the
    unrolled program (no control, no wait ops) is never later than the
    barrier-free per-loop schedule, which is never later than the per-engine
    one (at least as many wait ops); with every cost zero all three agree."""
    prm = oracle.sim_params()
    zero = oracle.sim_params(c_branch=0, c_regop=0, c_wait_ops_count=0, c_wait_ops_perloop=0,
                             c_wait_ops_perengine_level=0)
    deeper = 0
    for seed, batch in _random_batches(60):
        t_pl = oracle.thresholds(batch, PERLOOP)
        t_pe = oracle.thresholds(batch, PERENGINE)
        un = oracle.simulate(batch, t_pe, PERENGINE, oracle.UNROLLED, prm).makespan[0]
        pl = oracle.simulate(batch, t_pl, PERLOOP, oracle.BARRIER_FREE, prm).makespan[0]
        pe = oracle.simulate(batch, t_pe, PERENGINE, oracle.BARRIER_FREE, prm).makespan[0]
        assert 0 <= un <= pl <= pe, seed
        z = [oracle.simulate(batch, t_pl, PERLOOP, oracle.BARRIER_FREE, zero).makespan[0],
             oracle.simulate(batch, t_pe, PERENGINE, oracle.BARRIER_FREE, zero).makespan[0],
             oracle.simulate(batch, t_pe, PERENGINE, oracle.UNROLLED, zero).makespan[0]]
        assert z[0] == z[1] == z[2] == un, seed
        dep = loop_depths(batch)
        deeper += any(dep[int(batch.instr_loop[int(batch.dep_prod[d])])] >= 2 for d in range(batch.n_deps))
    assert deeper > 10     # the per-level term is exercised


@pytest.mark.parametrize("mode", [COUNT, PERLOOP])
def test_timing_safety_and_exactness(mode):
    """Safety: no consumer instance issues before the producer instance its
    threshold names has retired.  Exactness: with zero wait-op cost it issues at
    max(cursor, those retirements), so it never waits longer than required."""
    prm = oracle.sim_params(**ZERO)
    for seed, batch in _random_batches(40, body_hi=5, loops_hi=5):
        thr_c = oracle.thresholds(batch, COUNT)
        thr = oracle.thresholds(batch, mode)
        r = oracle.simulate(batch, thr, mode, oracle.BARRIER_FREE, prm, timeline=True)
        tot = loop_totals(batch)
        inst_off = np.concatenate([[0], np.cumsum([tot[l] for l in batch.instr_loop])])
        for d, sl in enumerate(pair_slices(batch)):
            p, c = int(batch.dep_prod[d]), int(batch.dep_cons[d])
            for g, cnt in enumerate(thr_c[sl]):
                if cnt > 0:
                    assert r.issue[inst_off[c] + g] >= r.retire[inst_off[p] + cnt - 1], seed


def test_timing_barrier_free_never_slower_at_zero_cost():
    """With zero control and wait-op costs the barrier scheme only adds
    constraints to a monotone max-plus system: barrier-free <= barrier; on
    straight-line programs (no loops) the two coincide."""
    prm = oracle.sim_params(**ZERO)
    for seed, batch in _random_batches(80):
        thr = oracle.thresholds(batch, PERLOOP)
        bf = oracle.simulate(batch, thr, PERLOOP, oracle.BARRIER_FREE, prm)
        bb = oracle.simulate(batch, thr, PERLOOP, oracle.BARRIER, prm)
        assert bf.makespan[0] <= bb.makespan[0], seed
    for seed, batch in _random_batches(30, loops_lo=0, loops_hi=0, body_lo=1, body_hi=9):
        thr = oracle.thresholds(batch, PERLOOP)
        bf = oracle.simulate(batch, thr, PERLOOP, oracle.BARRIER_FREE, prm)
        bb = oracle.simulate(batch, thr, PERLOOP, oracle.BARRIER, prm)
        assert bf.makespan[0] == bb.makespan[0], seed


def test_timing_deadlocks():
    """A same-iteration cycle across two engines never issues (status 7 under
    both schemes, Sec. 7.5); a backward offset-0 dependency across a nested
    loop runs barrier-free but cannot pass the barrier in front of that loop."""
    b = workloads.ProgramBuilder(2)
    A = b.loop(0, 0, [3])
    x = b.instr(A, 0, 0)
    y = b.instr(A, 1, 1)
    b.dep(y, x, 0)
    b.dep(x, y, 0)
    batch = b.batch()
    thr = oracle.thresholds(batch, PERLOOP)
    for v in (oracle.BARRIER_FREE, oracle.BARRIER):
        r = oracle.simulate(batch, thr, PERLOOP, v)
        assert (r.status[0], r.makespan[0], int(r.checksum[0])) == (7, -1, 0)
    b = workloads.ProgramBuilder(2)
    A = b.loop(0, 0, [3])
    c = b.instr(A, 0, 1)
    b.loop(A, 1, [2, 2, 2])
    p = b.instr(A, 2, 0)
    b.dep(p, c, 0)
    batch = b.batch()
    assert int(oracle.classify(batch).kase[0]) == oracle.CASE_PS
    thr = oracle.thresholds(batch, PERLOOP)
    assert oracle.simulate(batch, thr, PERLOOP, oracle.BARRIER_FREE).status[0] == 0
    assert oracle.simulate(batch, thr, PERLOOP, oracle.BARRIER).status[0] == 7


def test_timing_overflow_status():
    """The static time bound above INT32_MAX gives status 4."""
    b = workloads.ProgramBuilder(1)
    L = b.loop(0, 0, [3])
    b.instr(L, 0, 0, latency=2 ** 30)
    batch = b.batch()
    thr = np.zeros(0, dtype=np.int32)
    r = oracle.simulate(batch, thr, COUNT, oracle.BARRIER_FREE)
    assert (r.status[0], r.makespan[0]) == (4, -1)
    b = workloads.ProgramBuilder(1)
    L = b.loop(0, 0, [1])
    b.instr(L, 0, 0, latency=2 ** 30)
    r = oracle.simulate(b.batch(), thr, COUNT, oracle.BARRIER_FREE)
    # statement (c_regop) + iteration start (c_branch + 2*c_regop) before issue
    assert r.status[0] == 0 and r.makespan[0] == 2 ** 30 + 4


def test_generated_configs_are_allocatable_and_deadlock_free():
    for name, n in (("small", None), ("depth2", 6), ("gemm", None), ("attention", 1),
                    ("chain", 64), ("syncbound", 64)):
        batch = workloads.generate(name, n_programs=n)
        assert (oracle.classify(batch).kase != oracle.CASE_NONE).all(), name
        thr = oracle.thresholds(batch, PERLOOP)
        for v in (oracle.BARRIER_FREE, oracle.BARRIER):
            assert (oracle.simulate(batch, thr, PERLOOP, v).status == 0).all(), name


def test_program_ranges_are_independent():
    full = workloads.generate("chain", n_programs=40)
    part = workloads.generate("chain", n_programs=10, first_program=17)
    sub = workloads.concat([full], programs=[(0, p) for p in range(17, 27)])
    for k, v in sub.arrays().items():
        assert np.array_equal(v, getattr(part, k)), k


# ------------------------------------------- per-engine trip counts (Sec. 7.5)

def _divergent_batches(n=30, permille=300, **kw):
    for seed in range(n):
        b = workloads.random_trees(500 + seed, 1, workloads.tree_params(**kw))
        yield seed, workloads.diverge(b, 900 + seed, permille)


def test_divergent_rows_equal_to_shared_trips_change_nothing():
    """Per-engine rows that repeat the shared trips give the shared batch's
    thresholds, checks and timelines exactly."""
    b = workloads.random_trees(31, 40, workloads.tree_params(engines_hi=4, loops_hi=5, trip_hi=4))
    same = workloads.diverge(b, 3, permille=0)
    assert same.divergent
    assert oracle.sizes(same) == oracle.sizes(b)
    for mode in (COUNT, PERLOOP):
        t0, t1 = oracle.thresholds(b, mode), oracle.thresholds(same, mode)
        assert np.array_equal(t0, t1)
        assert np.array_equal(oracle.thresholds_bruteforce(same, mode), t1)
        r0 = oracle.simulate(b, t0, mode, oracle.BARRIER_FREE, timeline=True)
        r1 = oracle.simulate(same, t1, mode, oracle.BARRIER_FREE, timeline=True)
        for f in ("status", "makespan", "checksum", "issue", "retire"):
            assert np.array_equal(getattr(r0, f), getattr(r1, f)), (mode, f)


@pytest.mark.parametrize("mode", [COUNT, PERLOOP])
def test_divergent_definition_counting_and_registers_agree(mode):
    """Eq. (1) by enumeration on the consumer engine's walk, the counting
    form and the consumer engine's register replay agree on divergent
    programs; the checker accepts the result."""
    n_div = 0
    for seed, b in _divergent_batches(40, engines_hi=4, loops_hi=5, body_hi=5, trip_hi=4, max_depth=3):
        t = oracle.thresholds(b, mode)
        assert np.array_equal(oracle.thresholds_bruteforce(b, mode), t), seed
        assert np.array_equal(oracle.register_replay(b, mode), t), seed
        assert oracle.check(b, t, mode) == (0, 0, -1)
        n_div += oracle.sizes(b) != oracle.sizes(workloads.random_trees(500 + seed, 1, workloads.tree_params(
            engines_hi=4, loops_hi=5, body_hi=5, trip_hi=4, max_depth=3)))
    assert n_div >= 10          # the rows really diverge


def test_divergence_example_sec75():
    """Sec. 7.5's case: offset 0 from a producer on one engine to a consumer
    on another, both in a loop that runs zero times on the producer's engine
    and once on the consumer's.  The consumer's threshold is 1 (its own
    engine entered the loop once), the producer's count never reaches it, and
    the program deadlocks."""
    b = workloads.ProgramBuilder(2)
    A = b.loop(0, 0, [1], eng_trips=[[0], [1]])
    p = b.instr(A, 0, 0)
    c = b.instr(A, 1, 1)
    b.dep(p, c, 0)
    batch = b.batch()
    assert oracle.sizes(batch) == (1, 1)     # one consumer instance; the producer never runs
    for mode in (COUNT, PERLOOP):
        t = oracle.thresholds(batch, mode)
        assert t.tolist() == [1]
        r = oracle.simulate(batch, t, mode, oracle.BARRIER_FREE)
        assert (r.status[0], r.makespan[0], int(r.checksum[0])) == (7, -1, 0)


@pytest.mark.parametrize("mp,mc,k", [(3, 3, 0), (2, 5, 1), (5, 2, 0), (4, 6, 2), (0, 3, 3), (2, 4, 1)])
def test_divergent_single_loop_closed_form(mp, mc, k):
    """One loop under the top level, producer on engine 0 (mp iterations) and
    consumer on engine 1 (mc iterations), offset k: the consumer's g-th
    instance (1-based) waits for max(0, g - k) producer instances, and the
    program deadlocks exactly when the last of these exceeds mp; otherwise
    every consumer issues after that producer instance retires."""
    b = workloads.ProgramBuilder(2)
    A = b.loop(0, 0, [mp], eng_trips=[[mp], [mc]])
    p = b.instr(A, 0, 0, latency=5)
    c = b.instr(A, 1, 1, latency=2)
    b.dep(p, c, k)
    batch = b.batch()
    want = [max(0, g - k) for g in range(1, mc + 1)]
    assert oracle.thresholds(batch, COUNT).tolist() == want
    assert oracle.thresholds(batch, PERLOOP).tolist() == want          # N = K = 1
    r = oracle.simulate(batch, np.array(want, np.int32), COUNT, oracle.BARRIER_FREE, timeline=True)
    if max(want, default=0) > mp:
        assert r.status[0] == 7
    else:
        assert r.status[0] == 0
        for g, c_ in enumerate(want):
            if c_ > 0:
                assert r.issue[mp + g] >= r.retire[c_ - 1]


def test_divergent_unreachable_wait_deadlocks():
    """A count threshold above the producer's instances on its own engine can
    never be met: every such program ends in deadlock (status 7)."""
    seen = 0
    for seed, b in _divergent_batches(60, engines_hi=4, loops_hi=5, body_hi=5, trip_hi=4, max_depth=3):
        t = oracle.thresholds(b, COUNT)
        r = oracle.simulate(b, t, COUNT, oracle.BARRIER_FREE)
        unreachable = False
        off = 0
        for d in range(b.n_deps):
            px, cx = int(b.dep_prod[d]), int(b.dep_cons[d])
            n_prod = _instances(b, px)
            n_cons = _instances(b, cx)
            if n_cons and int(t[off:off + n_cons].max()) > n_prod:
                unreachable = True
            off += n_cons
        if unreachable:
            seen += 1
            assert r.status[0] == 7, seed
    assert seen >= 3


def _instances(b, x):
    """Instances of instruction x of a one-program batch on its own engine."""
    e = int(b.instr_engine[x])
    tot = [0] * b.n_loops
    tot[0] = 1
    for l in range(1, b.n_loops):
        tot[l] = int(b.engine_trips(0, l, e).sum())
    return tot[int(b.instr_loop[x])]


@pytest.mark.parametrize("mode", [COUNT, PERLOOP])
def test_divergent_timing_matches_recursive_statement(mode):
    """Per-engine trips in the semaphore machine and in the recursive
    statement (each engine's events follow its own trips; a wait for a
    producer instance its engine never runs never ends): same makespans,
    checksums, timelines and deadlocks."""
    prm = oracle.sim_params(ii=2, c_branch=3, c_regop=1, c_barrier=7)
    n_ok = n_dead = 0
    for seed, b in _divergent_batches(80, permille=400, engines_hi=3, loops_hi=4, body_hi=4, trip_hi=3,
                                      max_depth=3):
        thr = oracle.thresholds(b, mode)
        thr_c = oracle.thresholds(b, COUNT)
        r = oracle.simulate(b, thr, mode, oracle.BARRIER_FREE, prm, timeline=True)
        try:
            ms, chk, tl = timing_model.simulate(b, thr_c, prm, False, wait_ops(b, mode, prm))
        except timing_model.Deadlock:
            assert r.status[0] == 7, seed
            n_dead += 1
            continue
        assert r.status[0] == 0, seed
        assert r.makespan[0] == ms and int(r.checksum[0]) == chk, seed
        off = 0
        for x in range(b.n_instrs):
            n = _instances(b, x)
            for g in range(n):
                assert (r.issue[off + g], r.retire[off + g]) == tl[(x, g)], seed
            off += n
        n_ok += 1
    assert n_ok >= 10 and n_dead >= 3


def test_divergent_rejects_barrier_and_per_engine():
    """The barrier scheme (no common barrier sequence) and per-engine values
    are not defined with per-engine trips."""
    _, b = next(_divergent_batches(1))
    with pytest.raises(oracle.OracleError):
        oracle.thresholds(b, PERENGINE)
    t = oracle.thresholds(b, PERLOOP)
    with pytest.raises(oracle.OracleError):
        oracle.simulate(b, t, PERLOOP, oracle.BARRIER)


# ------------------------------------------------ trip-register elision (Sec. 5.1)

def _no_rhat_loops(batch):
    """Loops (program-local, not the top level) at which no dependency with
    a nonzero offset is carried: their trip register can be omitted."""
    cls = oracle.classify(batch)
    needs = {int(cls.S[d]) for d in range(batch.n_deps) if int(batch.dep_k[d]) > 0}
    return {l for l in range(1, batch.n_loops) if l not in needs}


@pytest.mark.parametrize("T,lat", [(1, 1), (5, 3), (12, 1)])
def test_elision_closed_form_one_engine(T, lat):
    """One engine, one loop of T iterations with one instruction and no
    dependency: without r-hat the loop statement and every iteration start
    lose one register op, so the makespan drops by exactly c_regop * (1 + T)."""
    b = workloads.ProgramBuilder(1)
    L = b.loop(0, 0, [T])
    b.instr(L, 0, 0, latency=lat)
    batch = b.batch()
    t = oracle.thresholds(batch, PERLOOP)
    for c_regop in (1, 4):
        prm0 = oracle.sim_params(c_regop=c_regop, c_branch=2)
        prm1 = oracle.sim_params(c_regop=c_regop, c_branch=2, trip_register_elision=1)
        m0 = oracle.simulate(batch, t, PERLOOP, oracle.BARRIER_FREE, prm0).makespan[0]
        m1 = oracle.simulate(batch, t, PERLOOP, oracle.BARRIER_FREE, prm1).makespan[0]
        assert m0 - m1 == c_regop * (1 + T)
        # the barrier scheme has no registers to elide
        b0 = oracle.simulate(batch, t, PERLOOP, oracle.BARRIER, prm0).makespan[0]
        b1 = oracle.simulate(batch, t, PERLOOP, oracle.BARRIER, prm1).makespan[0]
        assert b0 == b1


def test_elision_keeps_rhat_for_carried_offsets():
    """A loop carrying a dependency with offset 1 keeps its trip register:
    the flag changes nothing for a program whose only loop carries one."""
    b = workloads.ProgramBuilder(2)
    L = b.loop(0, 0, [6])
    x = b.instr(L, 0, 0, latency=2)
    y = b.instr(L, 1, 1, latency=3)
    b.dep(x, y, 1)
    batch = b.batch()
    assert _no_rhat_loops(batch) == set()
    t = oracle.thresholds(batch, PERLOOP)
    m0 = oracle.simulate(batch, t, PERLOOP, oracle.BARRIER_FREE).makespan[0]
    m1 = oracle.simulate(batch, t, PERLOOP, oracle.BARRIER_FREE,
                         oracle.sim_params(trip_register_elision=1)).makespan[0]
    assert m0 == m1


@pytest.mark.parametrize("mode", [COUNT, PERLOOP, PERENGINE])
def test_elision_matches_recursive_statement(mode):
    """With trip-register elision the semaphore machine and the recursive
    statement (each elided loop's statement free, its iteration starts one
    register op cheaper) agree on makespans, checksums and timelines."""
    prm = oracle.sim_params(ii=2, c_branch=3, c_regop=2, c_wait_ops_perengine_level=2,
                            trip_register_elision=1)
    n = 0
    for seed, batch in _random_batches(50):
        thr = oracle.thresholds(batch, mode)
        thr_c = oracle.thresholds(batch, COUNT)
        r = oracle.simulate(batch, thr, mode, oracle.BARRIER_FREE, prm, timeline=True)
        assert r.status[0] == 0
        ms, chk, tl = timing_model.simulate(batch, thr_c, prm, False, wait_ops(batch, mode, prm),
                                            no_rhat=_no_rhat_loops(batch))
        assert r.makespan[0] == ms and int(r.checksum[0]) == chk, seed
        off = 0
        tot = loop_totals(batch)
        for x in range(batch.n_instrs):
            for g in range(int(tot[batch.instr_loop[x]])):
                assert (r.issue[off + g], r.retire[off + g]) == tl[(x, g)]
            off += int(tot[batch.instr_loop[x]])
        n += 1
    assert n == 50


# ------------------------------------------------------ code-size proxy (RQ2)

def test_code_size_small_by_hand():
    """The small config: 6 instructions on 2 engines in one loop of 16
    iterations, 3 dependencies.  Looped: 6 instructions + 3 x (5 wait-value
    ops + 1 wait) + 2 engines x 4 control ops = 32; unrolled: 96 instances +
    48 pairs = 144."""
    b = workloads.generate("small")
    assert oracle.sizes(b) == (48, 96)
    assert oracle.code_size(b) == (32, 144)


def test_code_size_counts_fallback_barriers_not_waits():
    """A nested producer at forward offset 1 taken by the barrier fallback:
    no wait instructions for it, one barrier per engine for its loop; the
    unrolled count leaves its pairs out."""
    b = workloads.ProgramBuilder(2)
    A = b.loop(0, 0, [3])
    B = b.loop(A, 0, [2, 2, 2])
    p = b.instr(B, 0, 0)
    c = b.instr(A, 1, 1)
    q = b.instr(A, 2, 0)
    b.dep(p, c, 1)                       # nested forward, offset 1: barrier fallback
    b.dep(c, q, 0)                       # producer in S, offset 0: a wait
    batch = b.batch()
    batch.nonalloc_policy = 1
    # 3 instructions + 1 waited dependency x 6 + 2 engines x (2 loops x 4 + 1 barrier loop)
    assert oracle.code_size(batch) == (3 + 6 + 2 * (8 + 1), 6 + 3 + 3 + 3)


def test_code_size_looped_is_independent_of_trips():
    """The looped program does not grow with the trip counts; the unrolled
    one grows with the instances and pairs."""
    small = workloads.generate("small")
    big = small.copy()
    big.trips = big.trips * np.array([1] + [10] * (big.trips.size - 1), dtype=np.int32)
    lo, un = oracle.code_size(small)
    lo2, un2 = oracle.code_size(big)
    npairs, ninst = oracle.sizes(big)
    assert lo2 == lo and un2 == ninst + npairs == 10 * un
