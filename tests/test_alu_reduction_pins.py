"""Pins of the oracle's ALU reductions (Sec. 6.2) in its timing model.

LICM keeps each per-engine path term of a loop above the producer's loop in
a cached partial sum, updated when that loop starts an iteration; a wait then
pays the per-loop term and one read.  CSE reuses, within one visit of a
straight-line segment on one engine, the wait value of an earlier wait on the
same producer at the same offset, the mask of one with the same carrying loop
and offset, and (per-engine) the outer partial sum of one with the same
producer loop and producer engine.  The pins are closed forms on programs
whose engines never stall, the segment and engine boundaries of the sharing,
the static bound's extra terms, and equality with the recursive statement of
the timing model (tests/timing_model.py) fed by a separate Python statement
of the cost rules."""
import numpy as np
import pytest

import oracle
import workloads
from tests import timing_model

COUNT, PERLOOP, PERENGINE = oracle.COUNT, oracle.PERLOOP, oracle.PERENGINE
BF = oracle.BARRIER_FREE


def _run(batch, mode, **kw):
    prm = oracle.sim_params(**kw)
    thr = oracle.thresholds(batch, mode)
    r = oracle.simulate(batch, thr, mode, BF, prm)
    assert r.status[0] == 0
    return int(r.makespan[0])


def _chain(depth, trips, m_consumers=1, distinct_producers=False):
    """One engine; loops L1 > L2 > ... > L_depth (each L_j runs trips[j-1]
    iterations per parent iteration); in the innermost body the producer(s)
    and then m consumers, each waiting at offset 0 in the same iteration.
    Latency 1 = ii, so no instruction ever waits (the producer retires when
    the cursor passes it)."""
    b = workloads.ProgramBuilder(1)
    par, tot = 0, 1
    for d in range(depth):
        par = b.loop(par, 0, [trips[d]] * tot)
        tot *= trips[d]
    prods = [b.instr(par, i, 0, latency=1) for i in range(m_consumers if distinct_producers else 1)]
    for i in range(m_consumers):
        x = b.instr(par, 10 + i, 0, latency=1)
        b.dep(prods[i] if distinct_producers else prods[0], x, 0)
    return b.batch(), tot


@pytest.mark.parametrize("depth,trips", [(1, [7]), (2, [3, 5]), (3, [2, 3, 4]), (4, [2, 2, 3, 2])])
@pytest.mark.parametrize("c_level,c_regop", [(3, 1), (5, 2), (1, 4)])
def test_licm_closed_form(depth, trips, c_level, c_regop):
    """Depth-D chain, one per-engine wait per innermost iteration: without
    LICM each wait pays c_level per loop strictly between the top level and
    the producer's loop (D - 1 of them); with LICM it pays one c_regop read,
    and each of those loops pays c_level per iteration (one producer
    engine).  The makespans differ by exactly
      n * (c_level * (D - 1) - c_regop * [D > 1]) - c_level * sum_{j<D} iters(L_j)."""
    b, n = _chain(depth, trips)
    kw = dict(ii=1, c_branch=2, c_regop=c_regop, c_wait_ops_perloop=5, c_wait_ops_perengine_level=c_level)
    off = _run(b, PERENGINE, **kw)
    on = _run(b, PERENGINE, licm=1, **kw)
    iters = np.cumprod(trips)[:-1].sum() if depth > 1 else 0
    assert off - on == n * (c_level * (depth - 1) - (c_regop if depth > 1 else 0)) - c_level * iters
    # count and per-loop waits have no path sum: LICM changes nothing there
    for mode in (COUNT, PERLOOP):
        assert _run(b, mode, **kw) == _run(b, mode, licm=1, **kw)


@pytest.mark.parametrize("m", [1, 2, 5])
@pytest.mark.parametrize("mode,c", [(COUNT, 3), (PERLOOP, 5), (PERENGINE, 5)])
def test_cse_identical_waits(m, mode, c):
    """m consumers of one producer at the same offset in one segment: with
    CSE only the first computes the wait value, T * (m - 1) * c cycles less."""
    b, T = _chain(1, [9], m_consumers=m)
    kw = dict(c_wait_ops_count=3, c_wait_ops_perloop=5)
    assert _run(b, mode, **kw) - _run(b, mode, cse=1, **kw) == T * (m - 1) * c


@pytest.mark.parametrize("c_regop", [0, 1, 2, 7])
def test_cse_shared_mask(c_regop):
    """m consumers of distinct producers in the same loop at the same offset
    share the mask isGT(r-hat_S, k): each but the first pays min(c_regop,
    wait ops) less."""
    m = 4
    b, T = _chain(1, [6], m_consumers=m, distinct_producers=True)
    for mode, c in ((COUNT, 3), (PERLOOP, 5)):
        kw = dict(c_regop=c_regop, c_wait_ops_count=3, c_wait_ops_perloop=5)
        diff = _run(b, mode, **kw) - _run(b, mode, cse=1, **kw)
        assert diff == T * (m - 1) * min(c_regop, c), (mode, c_regop)


def _nested_consumers(m, split=False, engines=1):
    """Loop A (trip 5) > loop B (trip 3 per A-iteration) holding m producers;
    after B in A's body, m consumers waiting on them at offset 0 (nested,
    forward).  split: a child loop sits between the first consumer and the
    rest; engines: consumers on engines 0, 1, ... in turn."""
    b = workloads.ProgramBuilder(engines)
    A = b.loop(0, 0, [5])
    B = b.loop(A, 0, [3] * 5)
    prods = [b.instr(B, i, 0, latency=1) for i in range(m)]
    for i in range(m):
        pos = 10 + i + (20 if split and i > 0 else 0)
        x = b.instr(A, pos, i % engines, latency=1)
        b.dep(prods[i], x, 0)
    if split:
        b.loop(A, 15, [1] * 5)
    return b.batch()


def test_cse_shared_partial_sum_per_engine():
    """Per-engine waits on distinct producers of one loop (one producer
    engine) share the mask and the outer partial sum (one level here): each
    but the first pays min(c_regop, c_perloop) + c_level less; with LICM the
    shared outer part is the read of the cached sum."""
    m, T = 3, 5
    b = _nested_consumers(m)
    kw = dict(c_regop=1, c_wait_ops_perloop=5, c_wait_ops_perengine_level=4)
    assert _run(b, PERENGINE, **kw) - _run(b, PERENGINE, cse=1, **kw) == T * (m - 1) * (1 + 4)
    assert _run(b, PERENGINE, licm=1, **kw) - _run(b, PERENGINE, licm=1, cse=1, **kw) == T * (m - 1) * (1 + 1)


def test_cse_stops_at_child_loops_and_engines():
    """A child loop ends the straight-line segment (a consumer after it
    shares nothing with one before it), and waits on different engines share
    nothing."""
    kw = dict(c_regop=1, c_wait_ops_perloop=5, c_wait_ops_perengine_level=4)
    m, T = 3, 5
    split = _nested_consumers(m, split=True)
    # consumers 1 and 2 share with each other, not with consumer 0
    assert _run(split, PERENGINE, **kw) - _run(split, PERENGINE, cse=1, **kw) == T * 1 * (1 + 4)
    eng = _nested_consumers(m, engines=3)
    assert _run(eng, PERENGINE, **kw) == _run(eng, PERENGINE, cse=1, **kw)


def test_cse_never_later_and_zero_cost_neutral():
    """CSE only removes wait ops: never a later makespan (max-plus
    monotonicity); with every wait-op cost 0 it changes nothing."""
    zero = dict(c_regop=0, c_wait_ops_count=0, c_wait_ops_perloop=0, c_wait_ops_perengine_level=0)
    for seed, batch in _random(40):
        for mode in (COUNT, PERLOOP, PERENGINE):
            assert _run(batch, mode, cse=1) <= _run(batch, mode), (seed, mode)
            assert _run(batch, mode, cse=1, **zero) == _run(batch, mode, **zero)
            assert _run(batch, mode, cse=1, licm=1, **zero) == _run(batch, mode, **zero)


def test_licm_bound_counts_the_hoisted_updates():
    """A loop of 1100 iterations above a producer loop, whose consumer sits
    in a conditional that never runs: without LICM the bound holds no wait
    cost at all (no pair), with LICM the 1100 cached-sum updates of 2^21
    cycles exceed INT32_MAX (status 4); at 2^20 cycles they do not."""
    b = workloads.ProgramBuilder(1)
    A = b.loop(0, 0, [1100])
    B = b.loop(A, 0, [1] * 1100)
    p = b.instr(B, 0, 0)
    C = b.loop(A, 1, [0] * 1100)             # a conditional that never runs
    x = b.instr(C, 0, 0)
    b.dep(p, x, 0)
    batch = b.batch()
    thr = oracle.thresholds(batch, PERENGINE)
    kw = dict(c_wait_ops_perengine_level=2 ** 21)
    assert oracle.simulate(batch, thr, PERENGINE, BF, oracle.sim_params(**kw)).status[0] == 0
    assert oracle.simulate(batch, thr, PERENGINE, BF, oracle.sim_params(licm=1, **kw)).status[0] == 4
    kw = dict(c_wait_ops_perengine_level=2 ** 20)
    assert oracle.simulate(batch, thr, PERENGINE, BF, oracle.sim_params(licm=1, **kw)).status[0] == 0


# ------------------------------------------------ the recursive statement

def _random(n):
    for seed in range(n):
        b = workloads.random_trees(7700 + seed, 1, workloads.tree_params(
            engines_hi=3, loops_hi=5, body_hi=5, trip_hi=3, max_depth=4, max_deps_per_cons=3))
        if oracle.sizes(b)[1] <= 3000:
            yield seed, b


def _cost_rules(batch, mode, prm):
    """The Sec. 6.2 cost rules stated from the batch alone: (per-instruction
    wait ops, per-(loop, engine) iteration-start extra)."""
    nl, nx = batch.n_loops, batch.n_instrs
    par = [int(v) for v in batch.loop_parent]
    depth = [0] * nl
    for l in range(1, nl):
        depth[l] = depth[par[l]] + 1

    def anc(l):
        out = [l]
        while par[out[-1]] >= 0:
            out.append(par[out[-1]])
        return out

    def lca(a, b):
        sa = set(anc(a))
        return next(l for l in anc(b) if l in sa)

    xl = [int(v) for v in batch.instr_loop]
    xe = [int(v) for v in batch.instr_engine]
    deps_of = {}
    for d in range(batch.n_deps):
        deps_of.setdefault(int(batch.dep_cons[d]), []).append(d)
    cw = prm.c_wait_ops_count if mode == COUNT else prm.c_wait_ops_perloop
    # body items in position order; child loops end segments
    items = {l: [] for l in range(nl)}
    for x in range(nx):
        items[xl[x]].append((int(batch.instr_pos[x]), "x", x))
    for l in range(1, nl):
        items[par[l]].append((int(batch.loop_pos[l]), "l", l))
    cost = [0] * nx
    for l in range(nl):
        seen = []
        for _, kind, x in sorted(items[l]):
            if kind == "l":
                seen = []
                continue
            for d in deps_of.get(x, []):
                p, k = int(batch.dep_prod[d]), int(batch.dep_k[d])
                Pl, S = xl[p], lca(xl[p], xl[x])
                lev = max(0, depth[Pl] - 1) if mode == PERENGINE else 0
                outer = 0 if mode != PERENGINE else (
                    (prm.c_regop if lev > 0 else 0) if prm.licm else prm.c_wait_ops_perengine_level * lev)
                c = cw + outer
                if prm.cse:
                    mine = [w for w in seen if w[0] == xe[x]]
                    if any(w[1] == p and w[2] == k for w in mine):
                        c = 0
                    else:
                        mask = any(w[3] == S and w[2] == k for w in mine)
                        part = any(w[4] == Pl and w[5] == xe[p] for w in mine)
                        c = cw - (min(prm.c_regop, cw) if mask else 0) + (0 if part else outer)
                    seen.append((xe[x], p, k, S, Pl, xe[p]))
                cost[x] += c
    extra = {}
    if prm.licm and mode == PERENGINE:
        for d in range(batch.n_deps):
            p, x = int(batch.dep_prod[d]), int(batch.dep_cons[d])
            l = par[xl[p]]
            while l > 0:
                extra.setdefault((l, xe[x]), set()).add(xe[p])
                l = par[l]
    return (lambda x: cost[x]), (lambda l, e: prm.c_wait_ops_perengine_level * len(extra.get((l, e), ())))


@pytest.mark.parametrize("mode", [COUNT, PERLOOP, PERENGINE])
@pytest.mark.parametrize("licm,cse", [(1, 0), (0, 1), (1, 1)])
def test_reductions_match_recursive_statement(mode, licm, cse):
    """The semaphore machine with LICM / CSE equals the recursive statement
    fed by the cost rules above: makespans, checksums and timelines."""
    prm = oracle.sim_params(ii=2, c_branch=3, c_regop=2, c_wait_ops_count=4, c_wait_ops_perloop=6,
                            c_wait_ops_perengine_level=3, licm=licm, cse=cse)
    n = 0
    for seed, batch in _random(40):
        thr = oracle.thresholds(batch, mode)
        thr_c = oracle.thresholds(batch, COUNT)
        r = oracle.simulate(batch, thr, mode, BF, prm, timeline=True)
        assert r.status[0] == 0
        iw, ie = _cost_rules(batch, mode, prm)
        ms, chk, tl = timing_model.simulate(batch, thr_c, prm, False, 0, inst_wait=iw, iter_extra=ie)
        assert r.makespan[0] == ms and int(r.checksum[0]) == chk, seed
        tot = [1] + [0] * (batch.n_loops - 1)
        for l in range(1, batch.n_loops):
            tot[l] = int(batch.engine_trips(0, l, 0).sum())
        off = 0
        for x in range(batch.n_instrs):
            for g in range(tot[int(batch.instr_loop[x])]):
                assert (r.issue[off + g], r.retire[off + g]) == tl[(x, g)], seed
            off += tot[int(batch.instr_loop[x])]
        n += 1
    assert n >= 25


def test_bound_counts_wait_ops_before_the_reductions():
    """The static bound takes the wait ops before CSE: 100 iterations of 8
    consumers of one producer at 2^22 ops per wait exceed INT32_MAX before
    CSE (status 4 with and without it), although with CSE only one wait per
    iteration pays (100 * 2^22 < INT32_MAX)."""
    b, T = _chain(1, [100], m_consumers=8)
    thr = oracle.thresholds(b, COUNT)
    for cse in (0, 1):
        r = oracle.simulate(b, thr, COUNT, BF, oracle.sim_params(c_wait_ops_count=2 ** 22, cse=cse))
        assert r.status[0] == 4 and r.makespan[0] == -1
    r = oracle.simulate(b, thr, COUNT, BF, oracle.sim_params(c_wait_ops_count=2 ** 18, cse=1))
    assert r.status[0] == 0 and r.makespan[0] > 100 * 2 ** 18
