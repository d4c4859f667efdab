"""GPU path vs the CPU oracle, through the C ABI.  All results are integers and
must match bit for bit: thresholds in both encodings, checker counts and first
offending index, simulated makespans, checksums, statuses and timelines."""
import numpy as np
import pytest

import oracle
import workloads
from tests import golden_io

pytestmark = pytest.mark.gpu

COUNT, PERLOOP, PERENGINE = oracle.COUNT, oracle.PERLOOP, oracle.PERENGINE
MODES = (COUNT, PERLOOP)
ALL_MODES = (COUNT, PERLOOP, PERENGINE)
VARIANTS = (oracle.BARRIER_FREE, oracle.BARRIER)


def variants_for(mode):
    """The unrolled variant runs on per-engine semaphores only."""
    return VARIANTS + ((oracle.UNROLLED,) if mode == PERENGINE else ())


@pytest.fixture(scope="module")
def sg():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_13757_gb300 import build
    build.build()
    import paper_2608_13757_gb300 as m
    return m


def gpu_thresholds(sg, h, mode):
    thr = sg.sync_eval_thresholds(h, mode)
    host = thr.cpu().numpy()
    n = h.sizes.n_pairs_padded
    pad = np.ones(n, dtype=bool)
    idx = h.unpadded_index()
    pad[idx] = False
    assert (host[:n][pad] == 0).all(), "padding entries must be 0"
    return thr, host[idx]


def sim_params(oracle_prm):
    import paper_2608_13757_gb300 as m
    return m.SimParams(*[getattr(oracle_prm, f) for f, _ in oracle_prm._fields_])


def compare_all(sg, batch, params=None, timeline=False, modes=MODES):
    prm = params if params is not None else oracle.sim_params()
    h = sg.sync_load_programs(batch)
    npairs, ninst = oracle.sizes(batch)
    assert h.sizes.n_pairs == npairs and h.sizes.n_instances == ninst
    for mode in modes:
        thr, got = gpu_thresholds(sg, h, mode)
        want = oracle.thresholds(batch, mode)
        assert np.array_equal(got, want), f"thresholds differ (mode {mode})"
        counts, fb = sg.sync_check_minimal(h, mode, thr)
        assert counts.cpu().tolist() == [0, 0] and fb.item() == -1
        vs = (oracle.BARRIER_FREE,) if batch.divergent else variants_for(mode)
        if getattr(batch, "nonalloc_policy", 0):     # barrier fallbacks: no unrolled variant
            vs = tuple(v for v in vs if v != oracle.UNROLLED)
        for v in vs:
            ref = oracle.simulate(batch, want, mode, v, prm, timeline=timeline)
            res = sg.sync_simulate(h, mode, thr, sim_params(prm), v, timeline=timeline)
            fused, fcounts, ffirst = sg.sync_simulate_fused(h, mode, sim_params(prm), v, timeline=timeline,
                                                            check=True)
            assert fcounts.cpu().tolist() == [0, 0] and ffirst.item() == -1, (mode, v)
            for name, r in (("array", res), ("fused", fused)):
                P = batch.n_programs
                st = r.status.cpu().numpy()[:P]
                assert np.array_equal(st, ref.status), (name, mode, v)
                assert np.array_equal(r.makespan.cpu().numpy()[:P], ref.makespan), (name, mode, v)
                ck = r.checksum.cpu().numpy()[:P].view(np.uint64)
                assert np.array_equal(ck, ref.checksum), (name, mode, v)
                if timeline:
                    ok = np.repeat(ref.status == 0, _instances_per_program(batch))
                    assert np.array_equal(r.issue.cpu().numpy()[:ninst][ok], ref.issue[ok]), (name, mode, v)
                    assert np.array_equal(r.retire.cpu().numpy()[:ninst][ok], ref.retire[ok]), (name, mode, v)
    return h


def _instances_per_program(batch):
    out = []
    for p in range(batch.n_programs):
        out.append(oracle.sizes(batch.program(p))[1])
    return np.array(out, dtype=np.int64)


# ------------------------------------------- per-engine trip counts (NEXT-2)

@pytest.mark.parametrize("seed", range(4))
def test_divergent_random_trees(sg, seed):
    """Engines on their own trips (Sec. 7.5): thresholds on the consumer
    engine's loop state, the checker, and the barrier-free simulation (array
    and fused) with its deadlocks, equal to the oracle's."""
    base = workloads.random_trees(6000 + seed, 150, workloads.tree_params(
        engines_hi=5, loops_hi=5, body_hi=6, trip_hi=4, max_depth=4))
    batch = workloads.diverge(base, 7000 + seed, permille=250)
    compare_all(sg, batch, timeline=True, modes=MODES,
                params=oracle.sim_params(ii=2, c_branch=3, c_regop=2))
    st = oracle.simulate(batch, oracle.thresholds(batch, COUNT), COUNT).status
    assert (st == 7).any() and (st == 0).any()          # both outcomes are exercised


@pytest.mark.parametrize("name,n", [("depth2", 48), ("chain", 300), ("attention", 2)])
def test_divergent_configs(sg, name, n):
    batch = workloads.diverge(workloads.generate(name, n_programs=n), 11, permille=30)
    compare_all(sg, batch, timeline=name == "depth2", modes=MODES)


def test_divergent_mixed_with_shared_and_aligned(sg):
    """A batch mixing aligned per-engine rows (identical to shared trips) and
    divergent ones: the aligned programs give the shared batch's results."""
    shared = workloads.random_trees(6100, 60)
    aligned = workloads.diverge(shared, 1, permille=0)
    mixed = workloads.concat([aligned, workloads.diverge(shared, 2, permille=400)])
    compare_all(sg, mixed, timeline=True, modes=MODES)
    h = sg.sync_load_programs(aligned)
    h2 = sg.sync_load_programs(shared)
    for mode in MODES:
        t1, t2 = sg.sync_eval_thresholds(h, mode), sg.sync_eval_thresholds(h2, mode)
        import torch
        assert torch.equal(t1, t2)
        r1 = sg.sync_simulate(h, mode, t1)
        r2 = sg.sync_simulate(h2, mode, t2)
        for f in ("status", "makespan", "checksum"):
            assert torch.equal(getattr(r1, f), getattr(r2, f)), (mode, f)


def test_divergent_rejects_barrier_and_per_engine(sg):
    batch = workloads.diverge(workloads.random_trees(6200, 10), 3, permille=300)
    h = sg.sync_load_programs(batch)
    with pytest.raises(sg.SyncError) as err:
        sg.sync_eval_thresholds(h, sg.THR_PERENGINE)
    assert err.value.status == sg.ERR_ARG
    thr = sg.sync_eval_thresholds(h, sg.THR_PERLOOP)
    for v in (sg.SIM_BARRIER, sg.SIM_UNROLLED):
        with pytest.raises(sg.SyncError) as err:
            sg.sync_simulate(h, sg.THR_PERLOOP, thr, variant=v)
        assert err.value.status == sg.ERR_ARG
    with pytest.raises(sg.SyncError):
        sg.sync_simulate_fused(h, sg.THR_PERLOOP, variant=sg.SIM_BARRIER)


# ------------------------------------------------------------------ configs

@pytest.mark.parametrize("name,n", [("small", None), ("depth2", 48), ("gemm", None),
                                    ("attention", 2), ("chain", 400), ("syncbound", 400)])
def test_configs_bit_exact(sg, name, n):
    batch = workloads.generate(name, n_programs=n)
    compare_all(sg, batch, timeline=name in ("small", "depth2"))


@pytest.mark.parametrize("seed", range(4))
def test_long_loops_bit_exact(sg, seed):
    """Inner loops of up to 40 iterations with offsets up to 2: the barrier
    sweep writes runs of replayed iterations in one pass, cut where a wait
    first targets other in-chunk increments or reaches past the chunk's;
    thresholds, schedules and full timelines equal the oracle's in both
    schemes."""
    batch = workloads.random_trees(9700 + seed, 60, workloads.tree_params(
        engines_hi=5, loops_hi=4, body_hi=8, trip_lo=2, trip_hi=40, max_depth=3, k_max=2, dep_permille=700))
    compare_all(sg, batch, timeline=True, modes=(COUNT, PERLOOP, PERENGINE),
                params=oracle.sim_params(ii=2, c_branch=3, c_regop=2, c_barrier=7))


@pytest.mark.parametrize("seed", range(6))
def test_random_trees_bit_exact(sg, seed):
    batch = workloads.random_trees(1000 + seed, 150, workloads.tree_params(
        engines_hi=6, loops_hi=6, body_hi=6, trip_hi=4, max_depth=4))
    compare_all(sg, batch, timeline=True,
                params=oracle.sim_params(ii=2, c_branch=3, c_regop=2, c_barrier=9))


def test_golden_fixtures_on_gpu(sg):
    for name in golden_io.all_names():
        batch, expects = golden_io.load(name)
        h = sg.sync_load_programs(batch)
        for mode_name, d, want in expects:
            mode = COUNT if mode_name == "count" else PERLOOP
            _, got = gpu_thresholds(sg, h, mode)
            off = np.concatenate([[0], np.cumsum(h.pair_counts)])
            assert got[off[d]:off[d + 1]].tolist() == want, name


# ------------------------------------------------------------------ checker

@pytest.mark.parametrize("mode", MODES)
def test_checker_planted_errors(sg, mode):
    import torch
    batch = workloads.generate("depth2", n_programs=24)
    h = sg.sync_load_programs(batch)
    thr, good = gpu_thresholds(sg, h, mode)
    idx = h.unpadded_index()
    rng = np.random.default_rng(11)
    pick = np.sort(rng.choice(idx.size, size=101, replace=False))
    bad = good.copy()
    bad[pick[::2]] += 1
    bad[pick[1::2]] -= 1
    dev = thr.clone()
    dev[torch.from_numpy(idx[pick]).to(dev.device)] = torch.from_numpy(bad[pick]).to(dev.device)
    counts, fb = sg.sync_check_minimal(h, mode, dev)
    unsafe, over, first = oracle.check(batch, bad, mode)
    assert counts.cpu().tolist() == [unsafe, over]
    assert fb.item() == int(idx[first])
    # calls overwrite, they do not accumulate
    counts, fb = sg.sync_check_minimal(h, mode, thr)
    assert counts.cpu().tolist() == [0, 0] and fb.item() == -1


# ------------------------------------------------- per-engine allocation

@pytest.mark.parametrize("name,n", [("small", None), ("depth2", 48), ("gemm", None),
                                    ("attention", 2), ("chain", 400), ("syncbound", 400)])
def test_perengine_thresholds_bit_exact(sg, name, n):
    """Sec. 6.1 thresholds (engine-stream position of the c-th producer
    instance) equal the oracle's, and the checker finds them minimal."""
    batch = workloads.generate(name, n_programs=n)
    h = sg.sync_load_programs(batch)
    thr, got = gpu_thresholds(sg, h, oracle.PERENGINE)
    assert np.array_equal(got, oracle.thresholds(batch, oracle.PERENGINE))
    counts, fb = sg.sync_check_minimal(h, sg.THR_PERENGINE, thr)
    assert counts.cpu().tolist() == [0, 0] and fb.item() == -1
    # the derived positions are kept: a second call gives the same values
    thr2, got2 = gpu_thresholds(sg, h, oracle.PERENGINE)
    assert np.array_equal(got2, got)


@pytest.mark.parametrize("seed", range(4))
def test_perengine_random_trees(sg, seed):
    batch = workloads.random_trees(2000 + seed, 200, workloads.tree_params(
        engines_hi=6, loops_hi=6, body_hi=6, trip_hi=4, max_depth=4))
    h = sg.sync_load_programs(batch)
    _, got = gpu_thresholds(sg, h, oracle.PERENGINE)
    assert np.array_equal(got, oracle.thresholds(batch, oracle.PERENGINE))


def test_perengine_checker_planted_errors(sg):
    test_checker_planted_errors(sg, oracle.PERENGINE)


@pytest.mark.parametrize("name,n", [("small", None), ("depth2", 48), ("gemm", None),
                                    ("attention", 2), ("chain", 400), ("syncbound", 400)])
def test_perengine_simulation_bit_exact(sg, name, n):
    """Per-engine semaphores (Sec. 6.1) under the barrier-free, barrier and
    unrolled schemes: makespans, checksums, statuses (and timelines on the
    small cases) equal the oracle's."""
    batch = workloads.generate(name, n_programs=n)
    compare_all(sg, batch, timeline=name in ("small", "depth2"), modes=(PERENGINE,))


@pytest.mark.parametrize("seed", range(4))
def test_perengine_simulation_random_trees(sg, seed):
    batch = workloads.random_trees(3000 + seed, 150, workloads.tree_params(
        engines_hi=6, loops_hi=6, body_hi=6, trip_hi=4, max_depth=4))
    compare_all(sg, batch, timeline=True, modes=(PERENGINE,),
                params=oracle.sim_params(ii=2, c_branch=3, c_regop=2, c_barrier=9,
                                         c_wait_ops_perengine_level=5))


def test_unrolled_requires_perengine(sg):
    batch = workloads.generate("small")
    h = sg.sync_load_programs(batch)
    for mode in MODES:
        thr = sg.sync_eval_thresholds(h, mode)
        with pytest.raises(sg.SyncError) as err:
            sg.sync_simulate(h, mode, thr, variant=sg.SIM_UNROLLED)
        assert err.value.status == sg.ERR_ARG


@pytest.mark.parametrize("mode", ALL_MODES)
def test_wide_index_kernels(sg, mode, monkeypatch):
    """The 64-bit-index threshold and check kernels (taken for batches past
    2^31 pair indices) give the same values and verdicts; the switch forces
    them on a small batch."""
    batch = workloads.random_trees(4000 + mode, 120, workloads.tree_params(
        engines_hi=5, loops_hi=5, body_hi=6, trip_hi=6, max_depth=4))
    h = sg.sync_load_programs(batch)
    _, narrow = gpu_thresholds(sg, h, mode)
    monkeypatch.setenv("SYNCGB_WIDE_INDEX", "1")
    thr, wide = gpu_thresholds(sg, h, mode)
    assert np.array_equal(wide, narrow)
    assert np.array_equal(wide, oracle.thresholds(batch, mode))
    counts, fb = sg.sync_check_minimal(h, mode, thr)
    assert counts.cpu().tolist() == [0, 0] and fb.item() == -1
    test_checker_planted_errors(sg, mode)


@pytest.mark.parametrize("cfg", ["random", "gemm"])
def test_wide_derive_path(sg, cfg, monkeypatch):
    """The derive kernel's 64-bit write path (taken where a warp's rows span
    past 2^31 derived entries) builds the same arrays: loaded with the
    switch set, the thresholds equal the oracle's and the 32-bit path's."""
    batch = (workloads.random_trees(4100, 150, workloads.tree_params(engines_hi=5, loops_hi=5, body_hi=6,
                                                                       trip_hi=9, max_depth=4))
             if cfg == "random" else workloads.generate("gemm"))
    _, narrow = gpu_thresholds(sg, sg.sync_load_programs(batch), PERLOOP)
    monkeypatch.setenv("SYNCGB_WIDE_INDEX", "1")
    h = sg.sync_load_programs(batch)
    monkeypatch.delenv("SYNCGB_WIDE_INDEX")
    _, wide = gpu_thresholds(sg, h, PERLOOP)
    assert np.array_equal(wide, narrow)
    assert np.array_equal(wide, oracle.thresholds(batch, PERLOOP))


def test_checker_detects_swapped_encoding(sg):
    """Count-mode values read as per-loop values are below the minimum wherever
    N > 1 and c > 0."""
    batch = workloads.generate("gemm")
    h = sg.sync_load_programs(batch)
    thr_c, good_c = gpu_thresholds(sg, h, COUNT)
    counts, _ = sg.sync_check_minimal(h, PERLOOP, thr_c)
    unsafe, over, _ = oracle.check(batch, good_c, PERLOOP)
    assert counts.cpu().tolist() == [unsafe, over] and unsafe > 0


# --------------------------------------------------------------- edge cases

def test_empty_batch(sg):
    b = workloads.generate("chain", n_programs=0)
    h = sg.sync_load_programs(b)
    assert h.sizes.n_pairs_padded == 0
    thr = sg.sync_eval_thresholds(h, PERLOOP)
    counts, fb = sg.sync_check_minimal(h, PERLOOP, thr)
    assert counts.cpu().tolist() == [0, 0] and fb.item() == -1
    sg.sync_simulate(h, PERLOOP, thr)


def test_edge_programs(sg):
    """Zero-trip consumer loops (empty segments), conditionals, programs with no
    dependencies, 32 engines, nesting 15 deep, a deadlock under both schemes,
    a deadlock under the barrier scheme only, and a time-bound overflow."""
    progs = []
    b = workloads.ProgramBuilder(3)          # empty segment in the middle
    A = b.loop(0, 0, [4])
    B = b.loop(A, 1, [0, 0, 0, 0])
    x = b.instr(A, 0, 0)
    y = b.instr(B, 0, 1)
    z = b.instr(A, 2, 2)
    b.dep(x, y, 0); b.dep(y, z, 0); b.dep(x, z, 1)
    progs.append(b.batch())
    b = workloads.ProgramBuilder(1)          # no dependencies
    b.instr(0, 0, 0, latency=5)
    progs.append(b.batch())
    b = workloads.ProgramBuilder(32)         # 32 engines, a ring of waits
    A = b.loop(0, 0, [5])
    xs = [b.instr(A, i, i, latency=1 + i % 7) for i in range(32)]
    for i in range(1, 32):
        b.dep(xs[i - 1], xs[i], 0)
    b.dep(xs[31], xs[0], 1)
    progs.append(b.batch())
    b = workloads.ProgramBuilder(2)          # nesting 15 deep, trips 1..2
    par, tot, inner = 0, 1, []
    for lvl in range(15):
        t = 2 if lvl >= 13 else 1
        par = b.loop(par, 1, [t] * tot)
        tot *= t
        inner.append(par)
    p = b.instr(inner[2], 0, 0)
    c = b.instr(inner[14], 0, 1)
    b.dep(p, c, 0)
    progs.append(b.batch())
    b = workloads.ProgramBuilder(2)          # same-iteration cycle: deadlock
    A = b.loop(0, 0, [3])
    u = b.instr(A, 0, 0); v = b.instr(A, 1, 1)
    b.dep(v, u, 0); b.dep(u, v, 0)
    progs.append(b.batch())
    b = workloads.ProgramBuilder(2)          # backward offset 0 across a loop
    A = b.loop(0, 0, [3])
    c = b.instr(A, 0, 1)
    b.loop(A, 1, [2, 2, 2])
    p = b.instr(A, 2, 0)
    b.dep(p, c, 0)
    progs.append(b.batch())
    b = workloads.ProgramBuilder(1)          # time bound above INT32_MAX
    L = b.loop(0, 0, [3])
    b.instr(L, 0, 0, latency=2 ** 30)
    progs.append(b.batch())
    batch = workloads.concat(progs)
    compare_all(sg, batch, timeline=True, modes=ALL_MODES)
    ref = oracle.simulate(batch, oracle.thresholds(batch, PERLOOP), PERLOOP, oracle.BARRIER)
    assert 7 in ref.status.tolist() and 4 in ref.status.tolist()


def test_zero_costs_and_large_costs(sg):
    batch = workloads.random_trees(77, 120)
    compare_all(sg, batch, modes=ALL_MODES,
                params=oracle.sim_params(ii=0, c_branch=0, c_regop=0, c_wait_ops_count=0,
                                         c_wait_ops_perloop=0, c_barrier=0,
                                         c_wait_ops_perengine_level=0))
    compare_all(sg, batch, modes=ALL_MODES,
                params=oracle.sim_params(ii=7, c_branch=100, c_regop=50, c_wait_ops_count=9,
                                         c_wait_ops_perloop=13, c_barrier=1000,
                                         c_wait_ops_perengine_level=21))


def test_repeated_calls_are_identical(sg):
    batch = workloads.generate("chain", n_programs=300)
    h = sg.sync_load_programs(batch)
    thr = sg.sync_eval_thresholds(h, PERLOOP)
    a = sg.sync_simulate(h, PERLOOP, thr)
    b = sg.sync_simulate(h, PERLOOP, thr, variant=sg.SIM_BARRIER)
    c = sg.sync_simulate(h, PERLOOP, thr)
    assert np.array_equal(a.makespan.cpu().numpy(), c.makespan.cpu().numpy())
    assert np.array_equal(a.checksum.cpu().numpy(), c.checksum.cpu().numpy())
    assert not np.array_equal(a.makespan.cpu().numpy(), b.makespan.cpu().numpy())


# ------------------------------------------------- trip-register elision

@pytest.mark.parametrize("seed", range(3))
def test_trip_register_elision(sg, seed):
    """Loops that carry only offset-0 dependencies keep no trip register
    (Sec. 5.1) when the switch is on: every mode and scheme, array and
    fused, equal to the oracle; and a batch where no loop qualifies gives the
    same schedules with the switch on and off."""
    batch = workloads.concat([workloads.random_trees(9000 + seed, 120, workloads.tree_params(
        engines_hi=5, loops_hi=6, body_hi=6, trip_hi=4, max_depth=4)), workloads.generate("depth2", n_programs=8),
        workloads.generate("small")])
    compare_all(sg, batch, timeline=True, modes=ALL_MODES,
                params=oracle.sim_params(ii=2, c_branch=3, c_regop=4, trip_register_elision=1))


def test_trip_register_elision_divergent(sg):
    batch = workloads.diverge(workloads.random_trees(9100, 80), 3, permille=200)
    compare_all(sg, batch, timeline=True, modes=MODES,
                params=oracle.sim_params(c_regop=3, trip_register_elision=1))


# ------------------------------------------------------------------ loader

def loaded_results(sg, batch, modes, variants=(oracle.BARRIER_FREE,)):
    """Per mode: unpadded thresholds, check counts, and per variant the
    per-program makespans, checksums and statuses with the timelines."""
    h = sg.sync_load_programs(batch)
    idx = h.unpadded_index()
    out = []
    for mode in modes:
        thr = sg.sync_eval_thresholds(h, mode)
        counts, _ = sg.sync_check_minimal(h, mode, thr)
        res = [thr.cpu().numpy()[idx], counts.cpu().numpy()]
        for v in variants:
            r = sg.sync_simulate(h, mode, thr, variant=v, timeline=True)
            P = batch.n_programs
            res += [r.makespan.cpu().numpy()[:P], r.checksum.cpu().numpy()[:P], r.status.cpu().numpy()[:P],
                    r.issue.cpu().numpy(), r.retire.cpu().numpy()]
        out.append(res)
    h.close()
    return out


def assert_parts_match(sg, batch, cuts, modes, variants=(oracle.BARRIER_FREE,)):
    """The loader places every program's tables at offsets summed over the
    programs before it: each part of a batch, loaded alone, gives exactly
    its programs' share of the whole batch's results (thresholds and
    timelines concatenate, check counts add up)."""
    whole = loaded_results(sg, batch, modes, variants)
    parts = [loaded_results(sg, workloads.concat([batch], [(0, p) for p in range(a, b)]), modes, variants)
             for a, b in zip(cuts, cuts[1:])]
    for m in range(len(modes)):
        for f in range(len(whole[m])):
            if f == 1:
                assert np.array_equal(whole[m][f], sum(pt[m][f] for pt in parts))
            else:
                assert np.array_equal(whole[m][f], np.concatenate([pt[m][f] for pt in parts])), (modes[m], f)


def test_loader_offsets_shift_identically(sg):
    """Programs of random trees, depth2 and per-engine trips: loaded in one
    batch or in parts, every program gets the same thresholds, checks and
    schedules."""
    batch = workloads.concat([workloads.random_trees(8000, 97, workloads.tree_params(
        engines_hi=5, loops_hi=5, body_hi=6, trip_hi=4, max_depth=4)), workloads.generate("depth2", n_programs=20)])
    assert_parts_match(sg, batch, [0, 1, 40, 97, 117], (COUNT, PERLOOP, PERENGINE), (oracle.BARRIER_FREE, oracle.BARRIER))
    div = workloads.diverge(workloads.random_trees(8001, 40), 5, permille=200)
    assert_parts_match(sg, div, [0, 13, 40], (COUNT, PERLOOP))


def test_concurrent_loads_share_the_host_pools(sg):
    """Loads on several host threads at once (each takes its own scratch and
    pinned arena from the loader's pools, or a new one): every handle gives
    the results of the same batch loaded alone."""
    import threading
    batches = [workloads.random_trees(8100 + i, 60, workloads.tree_params(
        engines_hi=5, loops_hi=5, body_hi=6, trip_hi=4, max_depth=4)) for i in range(3)]
    batches.append(workloads.generate("chain", n_programs=3000))
    want = [loaded_results(sg, b, (PERLOOP,)) for b in batches]
    got = [None] * len(batches)
    errors = []

    def run(i):
        try:
            for _ in range(2):
                got[i] = loaded_results(sg, batches[i], (PERLOOP,))
        except Exception as e:          # reported below, on the test's thread
            errors.append(e)

    threads = [threading.Thread(target=run, args=(i,)) for i in range(len(batches))]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not errors, errors
    for w, g in zip(want, got):
        for a, b in zip(w[0], g[0]):
            assert np.array_equal(a, b)


def test_handle_is_ready_on_any_stream(sg):
    """sync_load_programs returns with its device work queued on its stream;
    a call on another stream right away waits for it (the handle's event)."""
    import torch
    batch = workloads.generate("chain", n_programs=1000)
    want_thr = oracle.thresholds(batch, PERLOOP)
    ref = oracle.simulate(batch, want_thr, PERLOOP, oracle.BARRIER_FREE)
    load_stream = torch.cuda.Stream()
    other = torch.cuda.Stream()
    for _ in range(3):
        torch.cuda.synchronize()
        torch.cuda._sleep(20_000_000)            # keep the device busy so the load's work queues up
        h = sg.sync_load_programs(batch, stream=load_stream)
        with torch.cuda.stream(other):
            thr = sg.sync_eval_thresholds(h, PERLOOP, stream=other)
            r = sg.sync_simulate(h, PERLOOP, thr, stream=other)
        other.synchronize()
        idx = h.unpadded_index()
        assert np.array_equal(thr.cpu().numpy()[idx], want_thr)
        assert np.array_equal(r.makespan.cpu().numpy()[:batch.n_programs], ref.makespan)
        assert np.array_equal(r.checksum.cpu().numpy()[:batch.n_programs].view(np.uint64), ref.checksum)
        h.close()


def test_device_loader_reports_what_host_validation_does(sg):
    """sync_load_programs validates on the device with the same per-program
    routine that sync_validate_programs runs on the host: on malformed and
    non-allocatable batches both give the same status and message."""
    import ctypes
    from tests import test_abi_cpu as T
    cases = [T._mut(f) for f in (
        lambda b: b.loop_parent.__setitem__(1, 2), lambda b: b.instr_engine.__setitem__(0, 2),
        lambda b: b.trips.__setitem__(2, -1), lambda b: b.instr_pos.__setitem__(2, 5),
        lambda b: b.dep_prod.__setitem__(0, 3), lambda b: b.prog_n_engines.__setitem__(0, 33))]
    for seed in range(20):
        cases.append(workloads.random_trees(seed, 12, workloads.tree_params(any_k=1, k_max=2)))
    n_bad = 0
    for batch in cases:
        desc, keep = sg.batch_desc(batch)
        st_host = sg.lib().sync_validate_programs(ctypes.byref(desc))
        msg_host = sg.lib().sync_last_error().decode()
        h = ctypes.c_void_p()
        st_dev = sg.lib().sync_load_programs(ctypes.byref(desc), 0, None, ctypes.byref(h))
        msg_dev = sg.lib().sync_last_error().decode()
        if st_dev == sg.OK:
            sg.lib().sync_free_programs(h)
        assert st_host == st_dev and (st_host == sg.OK or msg_host == msg_dev), (st_host, msg_host, st_dev, msg_dev)
        n_bad += st_dev != sg.OK
    assert n_bad >= 20


# ------------------------------------------------- full sizes, every program

@pytest.mark.parametrize("name", ["chain", "depth2", "attention", "syncbound"])
def test_full_size_every_program(sg, name):
    """The full configuration in one launch per kernel, every program
    recomputed by the oracle (spread over the host cores): every threshold
    in all three encodings, and every program's status, makespan and
    checksum under each scheme -- from the threshold array and fused."""
    import torch
    from tests import oracle_pool
    batch = workloads.generate(name)
    P = batch.n_programs
    h = sg.sync_load_programs(batch)
    mask = oracle_pool.unpadded_mask(h.pair_offsets, h.pair_counts)
    for mode in ALL_MODES:
        variants = variants_for(mode)
        want_thr, want = oracle_pool.run_config(name, mode, variants)
        thr = sg.sync_eval_thresholds(h, mode)
        host = thr.cpu().numpy()[:mask.size]
        assert (host[~mask] == 0).all(), (name, mode, "padding")
        got = host[mask]
        assert got.size == want_thr.size
        bad = np.flatnonzero(got != want_thr)
        assert bad.size == 0, (name, mode, bad[:8], got[bad[:8]], want_thr[bad[:8]])
        del host, got
        counts, fb = sg.sync_check_minimal(h, mode, thr)
        assert counts.cpu().tolist() == [0, 0] and fb.item() == -1
        for v in variants:
            res = sg.sync_simulate(h, mode, thr, variant=v)
            f, fc, ff = sg.sync_simulate_fused(h, mode, variant=v, check=True)
            assert fc.cpu().tolist() == [0, 0] and ff.item() == -1, (name, mode, v)
            ref = want[v]
            for label, r in (("array", res), ("fused", f)):
                st = r.status.cpu().numpy()[:P]
                assert np.array_equal(st, ref.status), (name, mode, v, label, "status")
                ms = r.makespan.cpu().numpy()[:P]
                bad = np.flatnonzero(ms != ref.makespan)
                assert bad.size == 0, (name, mode, v, label, bad[:8])
                ck = r.checksum.cpu().numpy()[:P].view(np.uint64)
                assert np.array_equal(ck, ref.checksum), (name, mode, v, label, "checksum")
        del thr
        torch.cuda.empty_cache()
    h.close()


def test_full_size_gemm_timeline(sg):
    """The single 1.25M-instance GEMM program, complete timeline."""
    batch = workloads.generate("gemm")
    compare_all(sg, batch, timeline=True, modes=(PERLOOP,))


# ------------------------------------------------------ code-size proxy (RQ2)

def test_code_size_proxy_matches_oracle(sg):
    """sync_sizes' code-size proxy of the looped and unrolled programs equals
    the oracle's instruction counts times the stated instruction size, on
    every config shape, random trees, per-engine trips and the barrier
    fallback."""
    from tests.test_fallback_pins import FAR
    fb = workloads.random_trees(44, 40, workloads.tree_params(**FAR))
    fb.nonalloc_policy = 1
    batches = [workloads.generate(n, n_programs=k) for n, k in
               (("small", None), ("depth2", 16), ("gemm", None), ("attention", 1), ("chain", 300),
                ("syncbound", 300))]
    batches += [workloads.random_trees(45, 100),
                workloads.diverge(workloads.random_trees(46, 50), 1, permille=200), fb]
    for b in batches:
        h = sg.sync_load_programs(b)
        lo, un = oracle.code_size(b)
        assert h.sizes.code_bytes_looped == sg.CODE_BYTES_PER_INSTR * lo
        assert h.sizes.code_bytes_unrolled == sg.CODE_BYTES_PER_INSTR * un
        h.close()


# ---------------------------------------- Sec. 6.2's ALU reductions (NEXT-3)

REDUCTIONS = [dict(licm=1), dict(cse=1), dict(licm=1, cse=1)]


@pytest.mark.parametrize("red", REDUCTIONS, ids=["licm", "cse", "licm+cse"])
@pytest.mark.parametrize("seed", range(3))
def test_alu_reductions_random_trees(sg, red, seed):
    """LICM / CSE in every mode and scheme, array and fused, timelines
    included, equal to the oracle on random trees with several waits per
    consumer and deep producer loops."""
    batch = workloads.random_trees(9300 + seed, 150, workloads.tree_params(
        engines_hi=5, loops_hi=6, body_hi=6, trip_hi=4, max_depth=4, max_deps_per_cons=3))
    compare_all(sg, batch, timeline=True, modes=ALL_MODES,
                params=oracle.sim_params(ii=2, c_branch=3, c_regop=2, c_wait_ops_count=4, c_wait_ops_perloop=6,
                                         c_wait_ops_perengine_level=3, **red))


@pytest.mark.parametrize("name,n", [("depth2", 24), ("gemm", None), ("attention", 1), ("chain", 300),
                                    ("syncbound", 300)])
def test_alu_reductions_configs(sg, name, n):
    batch = workloads.generate(name, n_programs=n)
    for red in REDUCTIONS:
        compare_all(sg, batch, timeline=name == "depth2", modes=ALL_MODES, params=oracle.sim_params(**red))


def test_alu_reductions_in_the_per_engine_kernel(sg):
    """Programs the sweep hands to the per-engine kernel -- barrier
    fallbacks (barrier-free), waits on later producers, per-engine trips --
    with the reductions on."""
    from tests.test_fallback_pins import FAR
    from tests.test_gpu_fallback import compare_fallback
    fb = workloads.random_trees(9400, 60, workloads.tree_params(**FAR))
    fb.nonalloc_policy = 1
    b = workloads.ProgramBuilder(2)          # a consumer ahead of its producer on another engine
    A = b.loop(0, 0, [3])
    B = b.loop(A, 1, [2, 2, 2])
    c = b.instr(A, 0, 1)
    p = b.instr(B, 0, 0)
    q = b.instr(A, 2, 0)
    b.dep(q, c, 0)
    b.dep(p, c, 1)
    b.dep(p, q, 0)
    fwd = workloads.concat([b.batch(), workloads.generate("depth2", n_programs=6)])
    mixed = workloads.concat([fb, workloads.generate("depth2", n_programs=6)])
    for red in REDUCTIONS:
        prm = oracle.sim_params(c_regop=2, c_wait_ops_perengine_level=4, **red)
        compare_fallback(sg, mixed, prm=prm)           # fallback barriers: wait values 0 on their pairs
        compare_all(sg, fwd, timeline=True, modes=ALL_MODES, params=prm)
    div = workloads.diverge(workloads.random_trees(9401, 60, workloads.tree_params(max_deps_per_cons=3)), 4,
                            permille=200)
    compare_all(sg, div, timeline=True, modes=MODES, params=oracle.sim_params(cse=1))


def test_alu_reductions_overflow_bound(sg):
    """The static bound with LICM's cached-sum updates (the oracle's pinned
    overflow case) and with wait ops counted before CSE."""
    b = workloads.ProgramBuilder(1)
    A = b.loop(0, 0, [1100])
    B = b.loop(A, 0, [1] * 1100)
    p = b.instr(B, 0, 0)
    C = b.loop(A, 1, [0] * 1100)
    x = b.instr(C, 0, 0)
    b.dep(p, x, 0)
    c = workloads.ProgramBuilder(1)
    L = c.loop(0, 0, [100])
    pc = c.instr(L, 0, 0)
    for i in range(8):
        c.dep(pc, c.instr(L, 10 + i, 0), 0)
    batch = workloads.concat([b.batch(), c.batch()])
    for kw in (dict(c_wait_ops_perengine_level=2 ** 21, licm=1), dict(c_wait_ops_perengine_level=2 ** 20, licm=1),
               dict(c_wait_ops_count=2 ** 22, c_wait_ops_perloop=2 ** 22, cse=1)):
        compare_all(sg, batch, modes=ALL_MODES, params=oracle.sim_params(**kw))
    thr = oracle.thresholds(batch, PERENGINE)
    st = oracle.simulate(batch, thr, PERENGINE, oracle.BARRIER_FREE,
                         oracle.sim_params(c_wait_ops_perengine_level=2 ** 21, licm=1)).status
    assert st[0] == 4
