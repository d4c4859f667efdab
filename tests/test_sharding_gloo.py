"""The multi-GPU path's host logic on CPU, with two gloo ranks.

Weak scaling (bench.shard): every rank takes its own programs.  Strong
scaling (bench.split_balanced): one batch is cut into contiguous program
ranges of about equal instance counts.  In both, each rank computes its part
with the oracle (thresholds, check, both schedules), the per-program results
gathered from the ranks in rank order equal one process's results over the
union, and bench.reduce_over_ranks gives the maximum of the ranks' measured
times and the sum of their pairs."""
import os
import socket
import time

import numpy as np
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _oracle_part(b):
    """Thresholds, check verdict and both schedules of a batch, with the
    wall time the oracle took."""
    import oracle
    t0 = time.perf_counter()
    thr = oracle.thresholds(b, oracle.PERLOOP)
    counts = oracle.check(b, thr, oracle.PERLOOP)
    sims = [oracle.simulate(b, thr, oracle.PERLOOP, v) for v in (oracle.BARRIER_FREE, oracle.BARRIER)]
    ms = 1e3 * (time.perf_counter() - t0)
    per_prog = np.stack([np.concatenate([s.makespan.astype(np.int64), s.status.astype(np.int64)]) for s in sims])
    checks = np.stack([s.checksum for s in sims])
    return thr, counts, per_prog, checks, ms


def _rank(rank, world, port, mode, out):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    import workloads
    if mode == "weak":
        first, P = bench.shard(rank, 5)
        b = workloads.generate("depth2", n_programs=P, first_program=first)
    else:
        whole = workloads.generate("chain", n_programs=600)
        first, P = bench.split_balanced(bench.instances_per_program(whole), world)[rank]
        b = workloads.generate("chain", n_programs=P, first_program=first)
    thr, counts, per_prog, checks, ms = _oracle_part(b)
    mx_ms, mx_e2e, pairs = bench.reduce_over_ranks(ms, 2.0 * (rank + 1), thr.size, "cpu")
    unsafe = bench.reduce_over_ranks(0.0, None, counts[0] + counts[1], "cpu")[2]
    gathered = [None] * world
    dist.all_gather_object(gathered, (rank, first, P, ms, int(bench.instances_per_program(b).sum()),
                                      per_prog, checks))
    out[rank] = (mx_ms, mx_e2e, pairs, unsafe, gathered)
    dist.destroy_process_group()


def _run(mode):
    world = 2
    mgr = mp.Manager()
    out = mgr.dict()
    mp.start_processes(_rank, args=(world, _free_port(), mode, out), nprocs=world, start_method="spawn")
    return dict(out)


def _check(out, union):
    import oracle
    thr, counts, per_prog, checks, _ = _oracle_part(union)
    for r, (mx_ms, mx_e2e, pairs, bad, gathered) in out.items():
        assert [g[0] for g in gathered] == [0, 1]
        assert mx_ms == max(g[3] for g in gathered)          # the slowest rank's measured time
        assert mx_e2e == 4.0
        assert pairs == thr.size and bad == 0 == counts[0] + counts[1]
        # contiguous, disjoint ranges covering the union, in rank order
        assert gathered[0][1] == 0 and gathered[1][1] == gathered[0][2]
        assert gathered[1][1] + gathered[1][2] == union.n_programs
        mk = [np.concatenate([g[5][v][:g[2]] for g in gathered]) for v in range(2)]
        st = [np.concatenate([g[5][v][g[2]:] for g in gathered]) for v in range(2)]
        ck = [np.concatenate([g[6][v] for g in gathered]) for v in range(2)]
        for v in range(2):
            assert np.array_equal(mk[v], per_prog[v][:union.n_programs])
            assert np.array_equal(st[v], per_prog[v][union.n_programs:])
            assert np.array_equal(ck[v], checks[v])
        assert (st[0] == oracle.SIM_OK).all() and (st[1] == oracle.SIM_OK).all()
    return out[0][4]


def test_weak_sharding_two_ranks_match_one_process():
    import workloads
    out = _run("weak")
    _check(out, workloads.generate("depth2", n_programs=10, first_program=0))


def test_balanced_split_two_ranks_match_one_process():
    """One skewed batch (chain programs range from a handful of instances to
    a few hundred thousand) split over two ranks: the ranks' instance counts
    are within 5% of each other, and the gathered results are one process's."""
    import bench
    import workloads
    union = workloads.generate("chain", n_programs=600)
    gathered = _check(_run("split"), union)
    inst = [g[4] for g in gathered]
    assert sum(inst) == int(bench.instances_per_program(union).sum())
    assert abs(inst[0] - inst[1]) <= 0.05 * max(inst)


def test_split_balanced_properties():
    """Contiguous, disjoint, covering ranges; every rank's work within one
    program's work of the even share; degenerate inputs."""
    import bench
    rng = np.random.default_rng(3)
    for world in (1, 2, 3, 4, 8):
        for n in (0, 1, 5, 100, 1000):
            w = rng.integers(0, 1000, size=n) ** 2
            r = bench.split_balanced(w, world)
            assert len(r) == world
            assert r[0][0] == 0 and sum(c for _, c in r) == n
            for (a, c), (a2, _) in zip(r, r[1:]):
                assert a + c == a2 and c >= 0
            if n and w.sum():
                share = w.sum() / world
                for a, c in r:
                    assert abs(int(w[a:a + c].sum()) - share) <= w.max()
