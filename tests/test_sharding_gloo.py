"""The multi-GPU path's host logic on CPU: two gloo ranks each take their own
programs (bench.shard), compute their part, and the cross-rank reduction
(bench.reduce_over_ranks) gives the same totals as one process over the
union of the programs.  Per-rank work uses the oracle on CPU."""
import os
import socket

import numpy as np
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    import oracle
    import workloads
    first, P = bench.shard(rank, 5)
    b = workloads.generate("depth2", n_programs=P, first_program=first)
    thr = oracle.thresholds(b, oracle.PERLOOP)
    bad = thr.copy()
    bad[::97] += 1                                   # planted over-synchronisation
    unsafe, over, _ = oracle.check(b, bad, oracle.PERLOOP)
    ms = 10.0 + rank                                 # stand-in step time
    mx_ms, mx_e2e, pairs = bench.reduce_over_ranks(ms, 2.0 * (rank + 1), thr.size, "cpu")
    c = bench.reduce_over_ranks(0.0, None, over, "cpu")[2]
    out[rank] = (mx_ms, mx_e2e, pairs, c, unsafe)
    dist.destroy_process_group()


def test_two_ranks_match_one_process():
    world = 2
    mgr = mp.Manager()
    out = mgr.dict()
    mp.start_processes(_rank, args=(world, _free_port(), out), nprocs=world, start_method="spawn")
    import oracle
    import workloads
    union = workloads.generate("depth2", n_programs=10, first_program=0)
    thr = oracle.thresholds(union, oracle.PERLOOP)
    expect_over = 0
    for r in range(world):
        part = workloads.generate("depth2", n_programs=5, first_program=5 * r)
        t = oracle.thresholds(part, oracle.PERLOOP)
        bad = t.copy()
        bad[::97] += 1
        expect_over += oracle.check(part, bad, oracle.PERLOOP)[1]
    for r in range(world):
        mx_ms, mx_e2e, pairs, over, unsafe = out[r]
        assert mx_ms == 11.0 and mx_e2e == 4.0
        assert pairs == thr.size
        assert over == expect_over and unsafe == 0
    # shards are disjoint and cover the union exactly
    parts = [workloads.generate("depth2", n_programs=5, first_program=5 * r) for r in range(world)]
    joined = workloads.concat(parts)
    for k, v in joined.arrays().items():
        assert np.array_equal(v, getattr(union, k)), k
