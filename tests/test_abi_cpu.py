"""The C ABI without a GPU: the library loads, exports every function that
include/sync.h declares, and its host-side validation returns the documented
status before any device work (no kernel is launched here)."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
import workloads

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def sg():
    from paper_2608_13757_gb300 import build
    build.build()
    import paper_2608_13757_gb300 as m
    return m


def declared_functions():
    src = open(os.path.join(ROOT, "include", "sync.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(sync_\w+)\s*\(", src)))


def test_exports_every_declared_symbol(sg):
    names = declared_functions()
    assert names == sorted(sg.EXPORTS)
    lib = ctypes.CDLL(sg.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n


def test_no_gpu_dependency_at_import(sg):
    assert sg.lib().sync_last_error() is not None


def test_launch_counter_reads_without_a_gpu(sg):
    """The launch counter is readable with no device and counts only
    launches the runtime accepted: without a device, none."""
    import torch
    n = sg.kernel_launches()
    assert isinstance(n, int) and n >= 0 and sg.kernel_launches() == n
    if not torch.cuda.is_available():
        assert n == 0


def _status(sg, batch):
    """The loader's validation on the host (sync_validate_programs runs the
    loader's per-program pass on host threads; no device needed)."""
    desc, keep = sg.batch_desc(batch)
    st = sg.lib().sync_validate_programs(ctypes.byref(desc))
    return st, sg.lib().sync_last_error().decode()




def _validated(sg):
    return {sg.OK}


def test_valid_batch_passes_validation(sg):
    st, _ = _status(sg, workloads.generate("small"))
    assert st in _validated(sg)


def test_null_arguments(sg):
    assert sg.lib().sync_load_programs(None, 0, None, None) == sg.ERR_ARG
    s = sg.Sizes()
    assert sg.lib().sync_query(None, ctypes.byref(s)) == sg.ERR_ARG
    assert sg.lib().sync_eval_thresholds(None, 0, None, None) == sg.ERR_ARG
    assert sg.lib().sync_check_minimal(None, 0, None, None, None, None) == sg.ERR_ARG
    prm = sg.SimParams()
    assert sg.lib().sync_simulate(None, 0, None, ctypes.byref(prm), 0, None, None, None, None,
                                 None, None) == sg.ERR_ARG
    assert sg.lib().sync_last_error().decode() != ""
    sg.lib().sync_free_programs(None)


def _base():
    b = workloads.ProgramBuilder(2)
    A = b.loop(0, 0, [3])
    B = b.loop(A, 5, [2, 0, 1])
    x = b.instr(A, 0, 0)
    y = b.instr(B, 0, 1)
    z = b.instr(A, 9, 1)
    b.dep(y, z, 0)
    b.dep(x, z, 1)
    return b


def _mut(fn):
    bt = _base().batch()
    fn(bt)
    return bt


@pytest.mark.parametrize("name,mutate", [
    ("root parent", lambda b: b.loop_parent.__setitem__(0, 0)),
    ("parent after child", lambda b: b.loop_parent.__setitem__(1, 2)),
    ("negative loop pos", lambda b: b.loop_pos.__setitem__(2, -1)),
    ("engine out of range", lambda b: b.instr_engine.__setitem__(0, 2)),
    ("latency 0", lambda b: b.instr_latency.__setitem__(1, 0)),
    ("negative trip", lambda b: b.trips.__setitem__(2, -1)),
    ("top loop trip 2", lambda b: b.trips.__setitem__(0, 2)),
    ("duplicate position", lambda b: b.instr_pos.__setitem__(2, 5)),
    ("instr loop out of range", lambda b: b.instr_loop.__setitem__(0, 7)),
    ("dep out of range", lambda b: b.dep_prod.__setitem__(0, 3)),
    ("negative offset", lambda b: b.dep_k.__setitem__(0, -1)),
    ("zero engines", lambda b: b.prog_n_engines.__setitem__(0, 0)),
    ("33 engines", lambda b: b.prog_n_engines.__setitem__(0, 33)),
])
def test_malformed(sg, name, mutate):
    st, msg = _status(sg, _mut(mutate))
    assert st == sg.ERR_MALFORMED, (name, st, msg)
    assert msg


def test_trip_array_length_mismatch(sg):
    bt = _base().batch()
    bt.trips = np.concatenate([bt.trips, [1]]).astype(np.int32)
    bt.trip_ptr[-1] += 1
    st, _ = _status(sg, bt)
    assert st == sg.ERR_MALFORMED


def test_depth_limit(sg):
    b = workloads.ProgramBuilder(1)
    parent = 0
    for _ in range(16):
        parent = b.loop(parent, 0, [1])
    b.instr(parent, 0, 0)
    st, _ = _status(sg, b.batch())
    assert st == sg.ERR_MALFORMED
    b = workloads.ProgramBuilder(1)
    parent = 0
    for _ in range(15):
        parent = b.loop(parent, 0, [1])
    b.instr(parent, 0, 0)
    st, _ = _status(sg, b.batch())
    assert st in _validated(sg)


@pytest.mark.parametrize("k,where,ok", [
    (0, "after", True), (1, "after", False),      # nested forward: offset 0 only
    (1, "before", True), (0, "before", False), (2, "before", False),  # backward: 1 only
])
def test_nested_offsets(sg, k, where, ok):
    b = workloads.ProgramBuilder(2)
    A = b.loop(0, 0, [3])
    B = b.loop(A, 5, [2, 2, 2])
    p = b.instr(B, 0, 0)
    c = b.instr(A, 9 if where == "after" else 1, 1)
    b.dep(p, c, k)
    st, _ = _status(sg, b.batch())
    assert (st in _validated(sg)) == ok, st
    if not ok:
        assert st == sg.ERR_NOT_ALLOCATABLE


def test_backward_offset0_same_engine_rejected(sg):
    b = workloads.ProgramBuilder(2)
    A = b.loop(0, 0, [3])
    c = b.instr(A, 0, 0)
    p = b.instr(A, 1, 0)
    b.dep(p, c, 0)
    assert _status(sg, b.batch())[0] == sg.ERR_NOT_ALLOCATABLE
    b = workloads.ProgramBuilder(2)
    A = b.loop(0, 0, [3])
    c = b.instr(A, 0, 1)
    p = b.instr(A, 1, 0)
    b.dep(p, c, 0)
    assert _status(sg, b.batch())[0] in _validated(sg)
    b = workloads.ProgramBuilder(1)
    A = b.loop(0, 0, [3])
    x = b.instr(A, 0, 0)
    b.dep(x, x, 0)
    assert _status(sg, b.batch())[0] == sg.ERR_NOT_ALLOCATABLE


def test_classification_matches_oracle(sg):
    """The loader and the oracle implement Sec. 5.2's case rules separately;
    on random programs with free offsets they accept exactly the same ones."""
    n_rej = n_ok = 0
    for seed in range(40):
        batch = workloads.random_trees(seed, 12, workloads.tree_params(any_k=1, k_max=2))
        kase = oracle.classify(batch).kase
        for p in range(batch.n_programs):
            one = batch.program(p)
            d0, d1 = batch.prog_dep_ptr[p], batch.prog_dep_ptr[p + 1]
            want_ok = bool((kase[d0:d1] != oracle.CASE_NONE).all())
            st, msg = _status(sg, one)
            assert (st in _validated(sg)) == want_ok, (seed, p, st, msg)
            if not want_ok:
                assert st == sg.ERR_NOT_ALLOCATABLE
            n_ok += want_ok
            n_rej += not want_ok
    assert n_ok > 50 and n_rej > 50


def test_overflow(sg):
    b = workloads.ProgramBuilder(1)
    A = b.loop(0, 0, [1 << 16])
    B = b.loop(A, 0, [1 << 15] * (1 << 16))
    b.instr(B, 0, 0)
    st, msg = _status(sg, b.batch())
    assert st == sg.ERR_OVERFLOW, msg
    # per-loop values N * iterations beyond INT32_MAX
    b = workloads.ProgramBuilder(2)
    A = b.loop(0, 0, [1 << 28])
    xs = [b.instr(A, i, 0) for i in range(8)]
    c = b.instr(A, 9, 1)
    b.dep(xs[0], c, 0)
    st, msg = _status(sg, b.batch())
    assert st == sg.ERR_OVERFLOW, msg
