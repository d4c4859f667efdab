#!/usr/bin/env python
"""Benchmark of the barrier-free semaphore engine on one GB300 (or N, sharded).

A step is one pass of the whole hot path over one batch: threshold kernel,
minimality checker, barrier-free schedule simulation and barrier schedule
simulation.  The metric is dynamic consumer instances -- (dependency,
consumer instance) pairs -- per second, summed over all ranks.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With N > 1 the script runs under torchrun, one rank per GPU; every rank
processes its own programs (program ids rank*P .. rank*P+P-1, weak scaling),
or with --split one batch cut into contiguous program ranges of about equal
instance counts (strong scaling); no data crosses ranks.  Rank 0 prints one
JSON line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "dynamic consumer instances/sec (threshold+check+sim), bit-exact; % HBM roofline"
UNIT = "pairs/s"
WORKLOADS = {
    # name -> description for config.workload
    "small": "1 program, 2 engines, one loop of 16 iterations, 6-instruction body, 3 cross-engine "
             "dependencies (one carried at distance 1)",
    "depth2": "4096 programs, 4 engines, loop depth 2, trips U[1,64] with the inner trip redrawn per "
              "outer iteration, 16-instruction bodies, 8 dependencies per body",
    "gemm": "1 program shaped like a tiled 4096x4096x4096 GEMM: 5 engines, M/N/K nest 32x8x32, "
            "double-buffered dependencies at distance 2",
    "attention": "256 programs shaped like causal flash attention: head(32) > q-tile(64) > kv-tile "
                 "(trip = q-tile index), 5 engines, 12-instruction body, running max/sum carried deps",
    "chain": "65536 random chain programs: 2-5 engines, up to 3 loops below the top level, "
             "trips U[0,32] redrawn per parent iteration, 1-32 instructions per body, "
             "dependency density 0.3",
    "syncbound": "65536 sync-bound programs: single-instruction conditionals alternating engines, "
                 "each depending on the previous, one distance-1 dependency per loop",
}
KERNELS = ("thresholds", "check", "sim_barrier_free", "sim_barrier")
CLOCK_QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
               "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
               "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--config", default="chain")
    ap.add_argument("--programs", type=int, default=None, help="programs per rank")
    ap.add_argument("--first-program", type=int, default=0,
                    help="id of rank 0's first program (ranks follow contiguously)")
    ap.add_argument("--split", action="store_true",
                    help="strong scaling: one batch (--programs, default the config's) cut into contiguous "
                         "program ranges of about equal instance counts, one per rank")
    ap.add_argument("--mode", choices=("perloop", "count"), default="perloop")
    ap.add_argument("--pipeline", choices=("arrays", "fused"), default="arrays",
                    help="arrays: threshold kernel, checker, two simulations over the stored thresholds; "
                         "fused: the two simulations compute (and, barrier-free, check) every wait value "
                         "themselves")
    ap.add_argument("--cpu-sample", type=int, default=32768,
                    help="programs of the workload the CPU oracle baseline runs")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    return ap.parse_args()


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d.get("sm_max_mhz", 2070.0)), "measured"
    except Exception:
        return 6800.0, 2070.0, "fallback"


# --------------------------------------------------------------- clocks

class ClockSampler:
    def __init__(self, index: int):
        self.proc = None
        self.path = None
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={index}", f"--query-gpu={CLOCK_QUERY}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows)}


# ------------------------------------------------------------- GPU side

# the sources each kernel's code is compiled from (enc.h: the shared tables)
KERNEL_SOURCES = {
    "thresholds": ("k_thresholds.cu", "waitval.cuh", "enc.h"),
    "check": ("k_thresholds.cu", "waitval.cuh", "enc.h"),
    "sim_barrier_free": ("k_sweep.cu", "sweep.cuh", "k_simulate.cu", "cost.cuh", "waitval.cuh", "enc.h"),
    "sim_barrier": ("k_sweep.cu", "sweep.cuh", "k_simulate.cu", "cost.cuh", "waitval.cuh", "enc.h"),
}


def kernel_hash(kernel: str = "sim_barrier_free", read=None) -> str:
    """Hash of the sources a kernel is built from (read(name) -> bytes
    overrides reading them from the tree)."""
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kernel]:
        if read is not None:
            h.update(read(f))
            continue
        with open(os.path.join(ROOT, "paper_2608_13757_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def profile_entry(kernel: str, workload: str):
    """A kernel's record in the committed ncu summary (profiles/traffic.json),
    if it was taken on the current sources of that kernel."""
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            d = json.load(f)
        e = d.get(workload, {}).get(kernel)
        if e and e.get("source_hash") == kernel_hash(kernel):
            return e
    except Exception:
        pass
    return None


def traffic_for(kernel: str, workload: str):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on
    the current kernel sources."""
    e = profile_entry(kernel, workload)
    return e["dram_bytes_per_launch"] if e else None


def run_gpu(args, rank, world, local_rank):
    import torch
    import paper_2608_13757_gb300 as sg
    import workloads

    torch.cuda.set_device(local_rank)
    mode = sg.THR_PERLOOP if args.mode == "perloop" else sg.THR_COUNT
    total = args.programs or workloads.CONFIGS[args.config][1]
    if args.split:
        whole = workloads.generate(args.config, n_programs=total, first_program=args.first_program)
        first, P = split_balanced(instances_per_program(whole), world)[rank]
        del whole
    else:
        first, P = shard(rank, total)
    first += args.first_program
    batch = workloads.generate(args.config, n_programs=P, first_program=first)
    t0 = time.perf_counter()
    h = sg.sync_load_programs(batch, device=local_rank)
    load_s = time.perf_counter() - t0
    sz = h.sizes
    dev = torch.device("cuda", local_rank)
    thr = torch.empty(max(sz.n_pairs_padded, 4), dtype=torch.int32, device=dev)
    counts = torch.empty(2, dtype=torch.int64, device=dev)
    first_bad = torch.empty(1, dtype=torch.int64, device=dev)
    prm = sg.SimParams()
    mk = lambda: sg.SimOutputs(torch.empty(max(P, 1), dtype=torch.int32, device=dev),
                               torch.empty(max(P, 1), dtype=torch.int64, device=dev),
                               torch.empty(max(P, 1), dtype=torch.int32, device=dev))
    bf, bb = mk(), mk()
    stream = torch.cuda.current_stream()

    fused = args.pipeline == "fused"

    def step(ev=None):
        if ev: ev[0].record(stream)
        if not fused: sg.sync_eval_thresholds(h, mode, out=thr)
        if ev: ev[1].record(stream)
        if not fused: sg.sync_check_minimal(h, mode, thr, counts, first_bad)
        if ev: ev[2].record(stream)
        if fused:
            sg.sync_simulate_fused(h, mode, prm, sg.SIM_BARRIER_FREE, out=bf, check=True, counts=counts,
                                   first_bad=first_bad)
        else:
            sg.sync_simulate(h, mode, thr, prm, sg.SIM_BARRIER_FREE, out=bf)
        if ev: ev[3].record(stream)
        if fused: sg.sync_simulate_fused(h, mode, prm, sg.SIM_BARRIER, out=bb)
        else: sg.sync_simulate(h, mode, thr, prm, sg.SIM_BARRIER, out=bb)
        if ev: ev[4].record(stream)

    for _ in range(max(args.warmup, 0)):
        step()
    torch.cuda.synchronize()
    # correctness of the timed configuration: minimal thresholds, no deadlock
    ok = counts.cpu().tolist() == [0, 0] and first_bad.item() == -1 and \
        int(bf.status[:P].max().item()) == 0 and int(bb.status[:P].max().item()) == 0
    dist_barrier(world)
    clocks = ClockSampler(local_rank)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(args.steps)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    # keep the GPU busy (about 5 ms) while the host queues the timed steps, so
    # host-side launch latency never shows up as GPU time between the events
    torch.cuda._sleep(10_000_000)
    launches0 = sg.kernel_launches()
    start.record(stream)
    for k in range(args.steps):
        step(evs[k])
    end.record(stream)
    launches = sg.kernel_launches() - launches0
    torch.cuda.synchronize()
    clk = clocks.stop()
    dist_barrier(world)
    total_ms = start.elapsed_time(end)
    per_kernel = {name: 0.0 for name in KERNELS}
    for e in evs:
        for i, name in enumerate(KERNELS):
            per_kernel[name] += e[i].elapsed_time(e[i + 1])
    per_kernel = {k: v / args.steps for k, v in per_kernel.items()}
    if fused:                             # no threshold kernel or checker launched
        per_kernel["thresholds"] = per_kernel["check"] = 0.0
    out = dict(ms=total_ms / args.steps, per_kernel=per_kernel, sizes=sz, clocks=clk, ok=ok, launches=launches,
               load_s=load_s, P=P, first=first,
               num_sms=torch.cuda.get_device_properties(dev).multi_processor_count)
    if not args.no_e2e:
        out["e2e"] = run_e2e(args, sg, batch, mode, prm, dev, P)
    h.close()
    return out


def launch_step(sg, h, mode, prm, fused, bufs=None):
    """Enqueues one step's kernels on the current stream and the read-back of
    its results into pinned host buffers; returns (buffers, device tensors
    to keep alive until the stream has run them)."""
    import torch
    if fused:
        thr = None
        r1, counts, fb = sg.sync_simulate_fused(h, mode, prm, sg.SIM_BARRIER_FREE, check=True)
        r2 = sg.sync_simulate_fused(h, mode, prm, sg.SIM_BARRIER)
    else:
        thr = sg.sync_eval_thresholds(h, mode)
        counts, fb = sg.sync_check_minimal(h, mode, thr)
        r1 = sg.sync_simulate(h, mode, thr, prm, sg.SIM_BARRIER_FREE)
        r2 = sg.sync_simulate(h, mode, thr, prm, sg.SIM_BARRIER)
    res = [counts, fb, r1.makespan, r1.checksum, r1.status, r2.makespan, r2.checksum, r2.status]
    if bufs is None:
        bufs = [torch.empty(x.shape, dtype=x.dtype, pin_memory=True) for x in res]
    for b, x in zip(bufs, res):
        b.copy_(x, non_blocking=True)
    return bufs, (thr, res)


def e2e_serial(args, sg, batch, mode, prm, dev):
    """One step at a time: load (host encoding + host-to-device copies), the
    four kernels, the results read back, the device idle meanwhile."""
    import torch
    steps = max(1, min(args.steps, 3))
    times, h2d, d2h = [], 0, 0
    for i in range(steps + 1):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        h = sg.sync_load_programs(batch, device=dev.index)
        host, keep = launch_step(sg, h, mode, prm, args.pipeline == "fused")
        torch.cuda.synchronize()
        t1 = time.perf_counter()
        if i > 0:
            times.append(t1 - t0)
        h2d = h.sizes.h2d_bytes
        d2h = sum(x.numel() * x.element_size() for x in host)
        h.close()
        del keep
    return {"s": statistics.median(times), "h2d": int(h2d), "d2h": int(d2h)}


def e2e_pipelined(args, sg, batch, mode, prm, dev, steps, bufs):
    """K steps as a stream of batches: the host builds and copies step i+1's
    encoding on a second stream while the device runs step i's kernels and
    read-back; the time runs from the first load to the last result on the
    host (pipeline fill and drain included).  Handles are released after
    the last step."""
    import torch
    # the loads' stream at the highest priority: at each kernel boundary of
    # the step being simulated, the next load's kernels are dispatched first
    load_stream = torch.cuda.Stream(device=dev, priority=torch.cuda.Stream.priority_range()[1])
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    handles, keeps = [], []
    h = sg.sync_load_programs(batch, device=dev.index, stream=load_stream)
    for i in range(steps):
        handles.append(h)
        host, keep = launch_step(sg, h, mode, prm, args.pipeline == "fused", bufs[i])
        keeps.append(keep)
        if i + 1 < steps:
            h = sg.sync_load_programs(batch, device=dev.index, stream=load_stream)
    torch.cuda.synchronize()
    t1 = time.perf_counter()
    for x in handles:
        x.close()
    return (t1 - t0) / steps, handles[0].sizes.h2d_bytes


def run_e2e(args, sg, batch, mode, prm, dev, P):
    """The same step through the public API from host arrays: load (host to
    device copies), the four kernels, and the results read back to the host;
    steps pipelined (host build of the next batch beside the device's work
    on this one), and one at a time for comparison."""
    import torch
    serial = e2e_serial(args, sg, batch, mode, prm, dev)
    steps = max(8, args.steps)
    # pinned result buffers per step, allocated before the timed region
    h = sg.sync_load_programs(batch, device=dev.index)
    bufs = []
    for _ in range(steps):
        b, keep = launch_step(sg, h, mode, prm, args.pipeline == "fused")
        bufs.append(b)
    torch.cuda.synchronize()
    h.close()
    del keep
    e2e_pipelined(args, sg, batch, mode, prm, dev, steps, bufs)          # warm-up (allocator)
    s, h2d = e2e_pipelined(args, sg, batch, mode, prm, dev, steps, bufs)
    ok = bool(int(bufs[-1][4].max()) == 0 and int(bufs[-1][7].max()) == 0 and int(bufs[-1][0].sum()) == 0)
    d2h = sum(x.numel() * x.element_size() for x in bufs[-1])
    return {"s": s, "h2d": int(h2d), "d2h": int(d2h), "steps": steps, "results_ok": ok, "serial_s": serial["s"]}


def shard(rank: int, programs_per_rank: int):
    """Program ids of a rank: rank*P .. rank*P+P-1 (weak scaling, no overlap)."""
    return rank * programs_per_rank, programs_per_rank


def instances_per_program(batch):
    """Dynamic datapath instances of every program of a batch (shared trips):
    a loop's iterations are the sum of its trips, an instruction has one
    instance per iteration of its loop."""
    import numpy as np
    tp = np.asarray(batch.trip_ptr, dtype=np.int64)
    trips = np.asarray(batch.trips, dtype=np.int64)
    csum = np.concatenate([[0], np.cumsum(trips)])
    loop_total = csum[tp[1:]] - csum[tp[:-1]]
    inst = loop_total[np.asarray(batch.instr_loop, dtype=np.int64) +
                      np.repeat(np.asarray(batch.prog_loop_ptr[:-1], dtype=np.int64),
                                np.diff(batch.prog_instr_ptr))]
    isum = np.concatenate([[0], np.cumsum(inst)])
    ip = np.asarray(batch.prog_instr_ptr, dtype=np.int64)
    return isum[ip[1:]] - isum[ip[:-1]]


def split_balanced(work, world: int):
    """Contiguous program ranges [(first, count)] for `world` ranks over
    per-program `work`: rank r's range ends at the first program whose
    cumulative work reaches r+1 world-ths of the total (strong scaling: the
    ranks process one batch, each about the same number of instances)."""
    import numpy as np
    work = np.asarray(work, dtype=np.int64)
    cum = np.cumsum(work)
    total = int(cum[-1]) if cum.size else 0
    cuts = [0]
    for r in range(1, world):
        target = total * r // world
        cuts.append(max(cuts[-1], int(np.searchsorted(cum, target, side="left")) + 1 if total else 0))
    cuts.append(int(work.size))
    cuts = [min(c, int(work.size)) for c in cuts]
    return [(cuts[r], cuts[r + 1] - cuts[r]) for r in range(world)]


def reduce_over_ranks(ms: float, e2e_s, pairs: int, device):
    """(max step time, max end-to-end time, total pairs) over the ranks of the
    default process group; the only cross-rank traffic of a run."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms, e2e_s or 0.0, float(pairs)], dtype=torch.float64, device=device)
    mx = t.clone()
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    sm = t.clone()
    dist.all_reduce(sm, op=dist.ReduceOp.SUM)
    return mx[0].item(), (mx[1].item() or None), sm[2].item()


def dist_barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ------------------------------------------------------------- CPU side

def oracle_run(config, first, count, mode_name):
    """The oracle on programs first..first+count-1: thresholds, check and both
    simulations.  Returns (pairs, seconds of oracle work)."""
    import oracle
    import workloads
    mode = oracle.PERLOOP if mode_name == "perloop" else oracle.COUNT
    b = workloads.generate(config, n_programs=count, first_program=first)
    t0 = time.perf_counter()
    thr = oracle.thresholds(b, mode)
    oracle.check(b, thr, mode)
    oracle.simulate(b, thr, mode, oracle.BARRIER_FREE)
    oracle.simulate(b, thr, mode, oracle.BARRIER)
    return int(thr.size), time.perf_counter() - t0


def cpu_baseline(config, sample, mode_name):
    """Oracle on a bounded sample of the workload, spread over the host cores
    (ctypes releases the GIL inside the oracle)."""
    from concurrent.futures import ThreadPoolExecutor
    import oracle
    import workloads
    oracle.build()
    workloads.build()
    cores = len(os.sched_getaffinity(0))
    n_chunks = max(1, min(sample, cores * 4))
    bounds = [(sample * i // n_chunks, sample * (i + 1) // n_chunks) for i in range(n_chunks)]
    mode = oracle.PERLOOP if mode_name == "perloop" else oracle.COUNT
    batches = [workloads.generate(config, n_programs=b - a, first_program=a) for a, b in bounds if b > a]

    def work(b):
        thr = oracle.thresholds(b, mode)
        oracle.check(b, thr, mode)
        oracle.simulate(b, thr, mode, oracle.BARRIER_FREE)
        oracle.simulate(b, thr, mode, oracle.BARRIER)
        return int(thr.size)

    t0 = time.perf_counter()
    with ThreadPoolExecutor(max_workers=cores) as ex:
        pairs = sum(ex.map(work, batches))
    dt = time.perf_counter() - t0
    # one core on the first 1/64 of the sample (at least one program)
    one = workloads.generate(config, n_programs=max(1, sample // 64))
    t1 = time.perf_counter()
    pairs1 = work(one)
    dt1 = time.perf_counter() - t1
    return {"value": pairs / dt, "unit": UNIT, "cores": cores, "kind": "oracle",
            "single_core_value": pairs1 / dt1,
            "sample": f"programs 0..{sample - 1} of the {config} workload ({pairs} pairs), "
                      f"thresholds + check + barrier-free and barrier simulation, {dt:.2f} s wall; "
                      f"single core: programs 0..{max(1, sample // 64) - 1} ({pairs1} pairs), {dt1:.2f} s"}


def run_reference(args, rank, world):
    """The oracle as the reference arm: each step is the bounded sample."""
    if rank != 0:
        return
    import oracle
    import workloads
    oracle.build()
    workloads.build()
    for _ in range(max(args.warmup, 0)):
        cb = cpu_baseline(args.config, min(args.cpu_sample, 1024), args.mode)
    vals = []
    t0 = time.perf_counter()
    for _ in range(args.steps):
        cb = cpu_baseline(args.config, args.cpu_sample, args.mode)
        vals.append(cb["value"])
    wall = time.perf_counter() - t0
    v = statistics.median(vals)
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * wall / max(args.steps, 1),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int32",
            "data": "synthetic",
            "config": {"workload": WORKLOADS.get(args.config, args.config),
                       "sample_programs": args.cpu_sample, "threshold_mode": args.mode},
            "cpu_baseline": {**cb, "value": v},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------- main

def roofline(res, hbm_peak, peak_kind, sm_mhz, workload):
    sz, pk = res["sizes"], res["per_kernel"]
    sms = res.get("num_sms") or 152
    # algorithmic bytes per launch: thresholds written / read once (padded
    # array) plus the loop-structure arrays and tables, each once
    alg = {"thresholds": 4 * sz.n_pairs_padded + sz.struct_bytes,
           "check": 4 * sz.n_pairs_padded + sz.struct_bytes}
    kernels = {}
    for name in ("thresholds", "check"):
        if pk[name] <= 0:
            continue                      # fused pipeline: no threshold array
        t = pk[name] / 1e3
        ach = alg[name] / t / 1e9 if t > 0 else 0.0
        kernels[name] = {"bound": "hbm", "ms": pk[name], "achieved": ach, "peak": hbm_peak,
                         "unit": "GB/s", "frac": ach / hbm_peak, "alg_bytes": alg[name],
                         "out_bytes": 4 * sz.n_pairs_padded,
                         "frac_out_only": 4 * sz.n_pairs_padded / t / 1e9 / hbm_peak if t > 0 else 0.0,
                         "traffic": traffic_for(name, workload)}
        # the same time against the DRAM bytes ncu measured for this kernel
        # (a full-size capture of the current sources), when there is one
        if kernels[name]["traffic"] and t > 0:
            kernels[name]["dram_achieved"] = kernels[name]["traffic"] / t / 1e9
            kernels[name]["dram_frac"] = kernels[name]["dram_achieved"] / hbm_peak
    # simulator: integer ops of the max-plus recurrence (per instance: wait
    # cost, one max per dependency, issue, retire max, cursor, checksum terms)
    # against the SM integer lanes: SMs x 128 int32 lanes x clock (nominal
    # unit counts, not a measured peak)
    lanes_peak = sms * 128 * (sm_mhz or 2070.0) * 1e6 / 1e12
    for name in ("sim_barrier_free", "sim_barrier"):
        ops = 12 * sz.n_instances + 2 * sz.n_pairs
        t = pk[name] / 1e3
        ach = ops / t / 1e12 if t > 0 else 0.0
        kernels[name] = {"bound": "alu", "ms": pk[name], "achieved": ach, "peak": lanes_peak,
                         "unit": "Tops/s", "frac": ach / lanes_peak, "alg_ops": ops,
                         "traffic": traffic_for(name, workload)}
        # what bounds the sweep in practice: warp-instruction issue (one per
        # SM sub-partition per cycle); instructions per instance from the
        # committed capture of the same sources, times live CUDA-event time
        e = profile_entry(name, workload)
        if e and e.get("warp_inst_per_instance") and t > 0:
            wi = e["warp_inst_per_instance"] * sz.n_instances
            ipk = sms * 4 * (sm_mhz or 2070.0) * 1e6 / 1e9
            kernels[name]["issue"] = {"warp_inst_per_instance": e["warp_inst_per_instance"],
                                      "achieved": wi / t / 1e9, "peak": ipk, "unit": "Ginst/s",
                                      "frac": wi / t / 1e9 / ipk,
                                      "source": e.get("issue_source", "instructions per instance from an "
                                                                      "ncu capture of the current sources")}
    dom = max(pk, key=pk.get)
    d = dict(kernels[dom])
    d["kernel"] = dom
    d["peak_source"] = (peak_kind if d["bound"] == "hbm" else
                        f"nominal, derived: {sms} SMs x 128 int32 lanes x median SM clock (no measured integer peak)")
    return d, kernels


def main():
    args = parse()
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    local_rank = int(os.environ.get("LOCAL_RANK", 0))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    import paper_2608_13757_gb300.build as b
    b.build()
    res = run_gpu(args, rank, world, local_rank)
    ms = res["ms"]
    pairs = res["sizes"].n_pairs
    e2e_s = res["e2e"]["s"] if "e2e" in res else None
    serial_s = res["e2e"]["serial_s"] if "e2e" in res else None
    if world > 1:
        _, serial_s, _ = reduce_over_ranks(ms, serial_s, pairs, "cuda")
        ms, e2e_s, total_pairs = reduce_over_ranks(ms, e2e_s, pairs, "cuda")
    else:
        total_pairs = float(pairs)
    if rank != 0:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
        return
    hbm_peak, sm_max, peak_kind = peaks()
    clk = res["clocks"] or {}
    roof, kernels = roofline(res, hbm_peak, peak_kind, clk.get("sm_mhz"), args.config)
    line = {
        "metric": METRIC, "value": total_pairs / (ms / 1e3), "unit": UNIT, "n_gpus": world,
        "instances_per_s": (res["sizes"].n_instances * world) / (ms / 1e3),
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "strong" if args.split else "weak", "vs_baseline": None, "dtype": "int32", "data": "synthetic",
        "config": {"workload": WORKLOADS.get(args.config, args.config), "programs_per_gpu": res["P"],
                   "pairs_per_gpu": int(pairs), "instances_per_gpu": int(res["sizes"].n_instances),
                   "threshold_mode": args.mode, "pipeline": args.pipeline,
                   "l2": "inputs larger than L2 (thresholds "
                   f"{4 * res['sizes'].n_pairs_padded / 1e9:.2f} GB per pass)",
                   "parallelism": (f"one batch of {args.programs or res['P'] * world} programs split over "
                                   f"{world} GPU(s) by instance count" if args.split else
                                   f"programs sharded over {world} GPU(s)"),
                   # code-size proxy (RQ2) of rank 0's programs: looped barrier-free vs unrolled
                   "code_bytes": {"looped": int(res["sizes"].code_bytes_looped),
                                  "unrolled": int(res["sizes"].code_bytes_unrolled),
                                  "unrolled_over_looped": (res["sizes"].code_bytes_unrolled /
                                                           max(res["sizes"].code_bytes_looped, 1)),
                                  "bytes_per_instruction": 16}},
        "roofline": roof,
        "kernels": kernels,
        # the library's own count of the kernels it launched in the timed
        # region: per step thresholds, check, and per schedule the sweep, the
        # per-engine kernel for programs it hands over and, where programs are
        # cut into pieces, the piece kernels
        "gpu_launches": res["launches"],
        "results_minimal_and_deadlock_free": res["ok"],
        "load_s": res["load_s"],
        "clocks": clk or None,
    }
    if e2e_s:
        line["e2e"] = {"value": total_pairs / e2e_s, "unit": UNIT,
                       "h2d_bytes_per_step": res["e2e"]["h2d"], "d2h_bytes_per_step": res["e2e"]["d2h"],
                       "steps": res["e2e"]["steps"], "results_ok": res["e2e"]["results_ok"],
                       "pipelined": "host encoding and copies of step i+1 on a second stream beside "
                                    "the kernels and read-back of step i; fill and drain timed",
                       "serial_value": total_pairs / serial_s if serial_s else None}
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(args.config, min(args.cpu_sample, res["P"]), args.mode)
    print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
