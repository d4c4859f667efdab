"""sync_simulate_noalloc, the simulation entry point for callers that cannot
allocate device memory around a call: through the C ABI it must give exactly
what sync_simulate gives, on two calls in a row (the calls share one static
scratch array that keeps the previous call's contents), and refuse batches
whose scratch needs exceed its fixed size.  Collected last on purpose."""
import ctypes

import numpy as np
import pytest

import workloads

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


def _batch():
    parts = [workloads.generate("depth2", n_programs=12), workloads.generate("small"),
             workloads.random_trees(41, 60, workloads.tree_params(engines_hi=5, loops_hi=5))]
    # a consumer waiting for a later producer on another engine (handed to the
    # per-engine kernel) and a cycle (deadlock)
    b = workloads.ProgramBuilder(2)
    A = b.loop(0, 0, [3])
    c = b.instr(A, 0, 1)
    b.loop(A, 1, [2, 2, 2])
    p = b.instr(A, 2, 0)
    b.dep(p, c, 0)
    parts.append(b.batch())
    b = workloads.ProgramBuilder(2)
    A = b.loop(0, 0, [3])
    u = b.instr(A, 0, 0)
    v = b.instr(A, 1, 1)
    b.dep(v, u, 0)
    b.dep(u, v, 0)
    parts.append(b.batch())
    return workloads.concat(parts)


def _instances_per_program(batch):
    out = []
    for p in range(batch.n_programs):
        l0, l1 = int(batch.prog_loop_ptr[p]), int(batch.prog_loop_ptr[p + 1])
        tot = [int(batch.trips[batch.trip_ptr[l]:batch.trip_ptr[l + 1]].sum()) for l in range(l0, l1)]
        x0, x1 = int(batch.prog_instr_ptr[p]), int(batch.prog_instr_ptr[p + 1])
        out.append(sum(tot[int(batch.instr_loop[x])] for x in range(x0, x1)))
    return np.array(out, dtype=np.int64)


def _outputs(sg, h):
    import torch
    P, n = h.sizes.n_programs, max(h.sizes.n_instances, 1)
    return sg.SimOutputs(torch.empty(P, dtype=torch.int32, device="cuda"),
                         torch.empty(P, dtype=torch.int64, device="cuda"),
                         torch.empty(P, dtype=torch.int32, device="cuda"),
                         torch.full((n,), -1, dtype=torch.int32, device="cuda"),
                         torch.full((n,), -1, dtype=torch.int32, device="cuda"))


def test_noalloc_matches_simulate_on_consecutive_calls(sg):
    """Two calls in a row per mode and scheme equal sync_simulate's results
    and, independently of that path, the oracle's (statuses, makespans,
    checksums and the timelines of the programs that complete)."""
    import torch
    import oracle
    batch = _batch()
    h = sg.sync_load_programs(batch)
    P = h.sizes.n_programs
    inst = _instances_per_program(batch)
    idx = h.unpadded_index()
    for mode in (sg.THR_COUNT, sg.THR_PERLOOP, sg.THR_PERENGINE):
        thr = sg.sync_eval_thresholds(h, mode)
        want_thr = oracle.thresholds(batch, mode)
        assert np.array_equal(thr.cpu().numpy()[idx], want_thr)
        unrolled = (sg.SIM_UNROLLED,) if mode == sg.THR_PERENGINE else ()
        for variant in (sg.SIM_BARRIER_FREE, sg.SIM_BARRIER) + unrolled:
            ref = sg.sync_simulate(h, mode, thr, variant=variant, timeline=True)
            orc = oracle.simulate(batch, want_thr, mode, variant, timeline=True)
            torch.cuda.synchronize()
            ok = ref.status.cpu().numpy() == sg.PROG_OK
            assert ok.sum() >= P - 2 and (~ok).any()
            defined = torch.from_numpy(np.repeat(ok, inst)).cuda()   # timelines of OK programs
            for _ in range(2):
                out = _outputs(sg, h)
                sg.sync_simulate_noalloc(h, mode, thr, variant=variant, out=out)
                torch.cuda.synchronize()
                for f in ("status", "makespan", "checksum"):
                    assert torch.equal(getattr(out, f), getattr(ref, f)), (mode, variant, f)
                for f in ("issue", "retire"):
                    assert torch.equal(getattr(out, f)[defined], getattr(ref, f)[defined]), (mode, variant, f)
                assert np.array_equal(out.status.cpu().numpy(), orc.status), (mode, variant)
                assert np.array_equal(out.makespan.cpu().numpy(), orc.makespan), (mode, variant)
                assert np.array_equal(out.checksum.cpu().numpy().view(np.uint64), orc.checksum), (mode, variant)
                mask = np.repeat(orc.status == 0, inst)
                for f in ("issue", "retire"):
                    got = getattr(out, f).cpu().numpy()[:mask.size]
                    assert np.array_equal(got[mask], getattr(orc, f)[mask]), (mode, variant, f)
    h.close()


def test_noalloc_refuses_batches_beyond_its_scratch(sg):
    h = sg.sync_load_programs(workloads.generate("chain", n_programs=4096))
    thr = sg.sync_eval_thresholds(h, sg.THR_PERLOOP)
    with pytest.raises(sg.SyncError) as err:
        sg.sync_simulate_noalloc(h, sg.THR_PERLOOP, thr)
    assert err.value.status == sg.ERR_ARG
    assert "scratch" in str(err.value)
    h.close()


def test_noalloc_with_the_barrier_fallback(sg):
    """Programs with fallback barriers (handed to the per-engine kernel,
    barrier-free) beside ordinary ones: the same results as sync_simulate,
    and the unrolled variant refused here too."""
    import torch
    from tests.test_fallback_pins import FAR, nested_program
    batch = workloads.concat([workloads.generate("depth2", n_programs=8),
                              workloads.random_trees(43, 40, workloads.tree_params(**FAR)),
                              nested_program(1), nested_program(3, backward=True)])
    batch.nonalloc_policy = 1
    h = sg.sync_load_programs(batch)
    inst = _instances_per_program(batch)
    for mode in (sg.THR_COUNT, sg.THR_PERLOOP, sg.THR_PERENGINE):
        thr = sg.sync_eval_thresholds(h, mode)
        for variant in (sg.SIM_BARRIER_FREE, sg.SIM_BARRIER):
            ref = sg.sync_simulate(h, mode, thr, variant=variant, timeline=True)
            torch.cuda.synchronize()
            ok = ref.status.cpu().numpy() == sg.PROG_OK
            defined = torch.from_numpy(np.repeat(ok, inst)).cuda()
            out = _outputs(sg, h)
            sg.sync_simulate_noalloc(h, mode, thr, variant=variant, out=out)
            torch.cuda.synchronize()
            for f in ("status", "makespan", "checksum"):
                assert torch.equal(getattr(out, f), getattr(ref, f)), (mode, variant, f)
            for f in ("issue", "retire"):
                assert torch.equal(getattr(out, f)[defined], getattr(ref, f)[defined]), (mode, variant, f)
    thr = sg.sync_eval_thresholds(h, sg.THR_PERENGINE)
    with pytest.raises(sg.SyncError) as err:
        sg.sync_simulate_noalloc(h, sg.THR_PERENGINE, thr, variant=sg.SIM_UNROLLED, out=_outputs(sg, h))
    assert err.value.status == sg.ERR_ARG
    h.close()
