"""A second, independent statement of the oracle's timing model, for tests.

The oracle runs an event-stepped machine over literal semaphore values.  This
module states the same timing model as memoised recursive equations over each
engine's event list, with waits expressed the specification's way: the
consumer instance waits for the retirement of the c-th instance of its
producer (c from count-mode thresholds), not for a semaphore value.  Only for
tiny programs (recursion).

Events per engine, in program order: a loop statement ("stmt"), an iteration
start ("iter"), an iteration end ("end", barrier scheme only), and the
engine's datapath instances.  Costs (barrier-free / barrier scheme):
stmt c_regop / barrier; iter c_branch + 2*c_regop / c_branch; end - / barrier;
datapath: t += the wait ops of its dependencies (barrier-free only), issue =
max(t, producer retirements), retire = max(issue + lat, previous retire),
t = issue + ii.  With per-engine trip counts each engine's event list follows
its own trips, and a wait for a producer instance its engine never runs
never ends (deadlock).  Barrier j: release = max over engines of max(t, last
retire) + c_barrier.  Unrolled (the straight-line program): as barrier-free
without stmt, iter or wait-op costs.
"""
import sys

MASK64 = (1 << 64) - 1


class Deadlock(Exception):
    pass


def _events(batch, e, barrier):
    """Per-engine event list of one-program batch (program-local ids)."""
    nl = batch.n_loops
    par = batch.loop_parent
    body = {l: [] for l in range(nl)}
    for x in range(batch.n_instrs):
        body[int(batch.instr_loop[x])].append((int(batch.instr_pos[x]), ("x", x)))
    for l in range(1, nl):
        body[int(par[l])].append((int(batch.loop_pos[l]), ("loop", l)))
    for l in body:
        body[l].sort()
    trips = {l: batch.engine_trips(0, l, e) for l in range(nl)}   # engine e's own trips
    nxt = [0] * nl
    ev = []

    def run(l, g):
        for _, (kind, i) in body[l]:
            if kind == "x":
                if int(batch.instr_engine[i]) == e:
                    ev.append(("x", i, g))
                continue
            m = i
            ev.append(("stmt", m))
            for _ in range(int(trips[m][g])):
                gm = nxt[m]
                nxt[m] += 1
                ev.append(("iter", m))
                run(m, gm)
                if barrier:
                    ev.append(("end",))

    run(0, 0)
    return ev


def simulate(batch, thr_count, params, barrier, cwait, unrolled=False, no_rhat=(), inst_wait=None,
             iter_extra=None):
    """(makespan, checksum, {(x, g): (issue, retire)}) or raises Deadlock.
    cwait: wait ops per dependency, an int or a function of the dependency.
    no_rhat: loops without a trip register (their statement costs nothing
    and their iteration starts one register op less, barrier-free).
    inst_wait: optional function of an instruction giving its total wait ops
    (replaces the sum of cwait over its dependencies); iter_extra: optional
    function (loop, engine) -> extra cycles at each iteration start of the
    loop on the engine (barrier-free)."""
    wait_ops = cwait if callable(cwait) else (lambda d: cwait)
    ne = int(batch.prog_n_engines[0])
    ev = [_events(batch, e, barrier) for e in range(ne)]
    where = {}
    for e in range(ne):
        for i, v in enumerate(ev[e]):
            if v[0] == "x":
                where[(v[1], v[2])] = (e, i)
    # pairs: dependency d, consumer instance g -> count threshold
    pair_off, off = [], 0
    loop_total = {}
    for l in range(batch.n_loops):
        loop_total[l] = None
    # consumer loop totals from the instance map
    inst_count = {}
    for (x, g) in where:
        inst_count[x] = max(inst_count.get(x, 0), g + 1)
    for d in range(batch.n_deps):
        pair_off.append(off)
        off += inst_count.get(int(batch.dep_cons[d]), 0)
    deps_of = {}
    for d in range(batch.n_deps):
        deps_of.setdefault(int(batch.dep_cons[d]), []).append(d)
    # barrier indices per engine
    bar_idx = []
    for e in range(ne):
        idx = [i for i, v in enumerate(ev[e]) if barrier and v[0] in ("stmt", "end")]
        bar_idx.append(idx)
    bar_no = [{i: j for j, i in enumerate(bar_idx[e])} for e in range(ne)]

    memo = {}
    busy = set()

    def state(e, i):
        """(t, last retire, issue, retire) after event i of engine e."""
        if i < 0:
            return (0, 0, None, None)
        key = (e, i)
        if key in memo:
            return memo[key]
        if key in busy:
            raise Deadlock()
        busy.add(key)
        t, lr, _, _ = state(e, i - 1)
        v = ev[e][i]
        if v[0] == "x":
            x, g = v[1], v[2]
            ds = deps_of.get(x, [])
            own = inst_wait(x) if inst_wait is not None else sum(wait_ops(d) for d in ds)
            tw = t + (0 if barrier or unrolled else own)
            ready = 0
            for d in ds:
                c = int(thr_count[pair_off[d] + g])
                if c <= 0:
                    continue
                p = int(batch.dep_prod[d])
                if (p, c - 1) not in where:
                    raise Deadlock()
                pe, pi = where[(p, c - 1)]
                ready = max(ready, state(pe, pi)[3])
            issue = max(tw, ready)
            retire = max(issue + int(batch.instr_latency[x]), lr)
            out = (issue + params.ii, retire, issue, retire)
        elif barrier and v[0] in ("stmt", "end"):
            j = bar_no[e][i]
            rel = 0
            for f in range(ne):
                fi = bar_idx[f][j]
                ft, flr, _, _ = state(f, fi - 1)
                rel = max(rel, ft, flr)
            out = (rel + params.c_barrier, lr, None, None)
        elif v[0] == "stmt":
            out = (t + (0 if unrolled or v[1] in no_rhat else params.c_regop), lr, None, None)
        elif unrolled:  # iteration start of the unrolled program: nothing
            out = (t, lr, None, None)
        else:  # iteration start: branch, r++ and (unless elided) r-hat++
            regops = 0 if barrier else (1 if v[1] in no_rhat else 2)
            extra = iter_extra(v[1], e) if iter_extra is not None and not barrier else 0
            out = (t + params.c_branch + regops * params.c_regop + extra, lr, None, None)
        busy.discard(key)
        memo[key] = out
        return out

    old = sys.getrecursionlimit()
    sys.setrecursionlimit(max(old, 20000))
    try:
        makespan, chk, tl = 0, 0, {}
        for e in range(ne):
            t, lr, _, _ = state(e, len(ev[e]) - 1)
            makespan = max(makespan, t, lr)
            n = 0
            for i, v in enumerate(ev[e]):
                if v[0] != "x":
                    continue
                n += 1
                _, _, iss, ret = state(e, i)
                tl[(v[1], v[2])] = (iss, ret)
                M = 0xFFFFFFFF
                a = (((iss & M) ^ ((n * 0x9E3779B9 + e) & M)) * 0x85EBCA6B) & M
                a ^= a >> 13
                b = (((ret & M) ^ ((n * 0xC2B2AE35 + e) & M)) * 0x27D4EB2F) & M
                b ^= b >> 15
                chk = (chk + ((a << 32) | b)) & MASK64
        return makespan, chk, tl
    finally:
        sys.setrecursionlimit(old)
