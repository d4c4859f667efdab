// Schedule simulator, program-order sweep: one warp per program.
//
// Under a common loop tree every engine meets the same loop statements and
// iteration boundaries, so one walker per program can visit the tree once for
// all engines (programs whose engines run their own trip counts, and
// barrier-free the programs with the barriers of the non-allocatable
// fallback, go straight to the per-engine kernel).  The body of each loop is cut at its child loops into
// straight-line segments; a segment is taken as one chunk of up to 32 datapath
// records (more chunks if longer), or -- barrier-free, for a short innermost
// body -- as several consecutive iterations at once.  The chunk's lanes are
// ordered engine-major, so each engine's events form a run of lanes:
//   - an engine's cursor obeys t' = max(t + A, B) per event (A its costs
//     and the issue interval, B the time its waits are satisfied plus the
//     issue interval), maps that compose associatively, so a segmented
//     5-step warp scan gives every event its cursor after issue, t' = issue
//     + ii; in-order retirement is a segmented max-scan of issue + latency;
//   - a wait on a semaphore whose threshold increment happened in an earlier
//     chunk reads its retire time from a ring of the semaphore's latest
//     increments (up to 32) in shared memory, or from the history array if older; an
//     increment inside the chunk is the k-th lane of the semaphore's lanes
//     (increments come in lane order), and these in-chunk waits are solved by
//     repeating the scans until no producer retires after its consumer's
//     issue (a least fixed point of the max-plus system; times only grow, a
//     cycle never settles and is a deadlock);
//   - a threshold beyond every increment up to this chunk points forward in
//     program order: the program is handed to the per-engine kernel.
// A loop whose body is one chunk runs all its iterations in a tight loop
// with the lanes' records in registers and the next iteration's thresholds
// in flight.  Barriers (barrier scheme) are a warp maximum of the engines'
// drained times.  Per-engine cursor, last retire and instance count live in
// shared memory, read by the engine's lanes and written back by the last
// lane of its run.
#pragma once

#include "cost.cuh"
#include "waitval.cuh"

namespace syncgb {
namespace {

constexpr int kWarps = 8;                   // programs (warps) per CTA
constexpr int kMaxIntra = 4;                // in-chunk waits per lane before falling back
constexpr int kMaxDeps = 2;                 // dependencies per lane held in registers
constexpr int kRingMax = 32;                // most recent increments kept per semaphore
constexpr unsigned kFull = 0xffffffffu;
constexpr int32_t kNeg = -1;                // -infinity of the cursor maps (cursors, costs >= 0)
constexpr int SIM_FALLBACK = 9;             // internal: handed to the per-engine kernel

struct Frame { int32_t loop, item, g, g_end; };

// Shared memory of one warp (program), 16-byte aligned.
__host__ __device__ __forceinline__ size_t warp_bytes(int sem_cap, int frame_depth, int ring) {
  const size_t per = (size_t)(20 + 4 * ring + 32) * sem_cap + sizeof(Frame) * (size_t)frame_depth +
                     8 * (size_t)(frame_depth + 1) + 3 * 8 + 8 + 3 * 4 * 32 + 16 + 8;
  return (per + 15) & ~(size_t)15;
}

__device__ __forceinline__ unsigned lanemask_le() {
  unsigned m;
  asm("mov.u32 %0, %%lanemask_le;" : "=r"(m));
  return m;
}
__device__ __forceinline__ unsigned long long inst_term(int32_t issue, int32_t retire, uint32_t e,
                                                        uint32_t n) {
  uint32_t x = ((uint32_t)issue ^ (n * 0x9E3779B9u + e)) * 0x85EBCA6Bu;
  x ^= x >> 13;
  uint32_t y = ((uint32_t)retire ^ (n * 0xC2B2AE35u + e)) * 0x27D4EB2Fu;
  y ^= y >> 15;
  return ((unsigned long long)x << 32) | y;
}


// Engines pay different iteration-start costs only with LICM's cached-sum
// updates (per-engine waits, barrier-free).
template <int MODE, bool BB>
__device__ __forceinline__ bool hoists(const SweepArgs& a) {
  return !BB && MODE == SYNC_THR_PERENGINE && a.prm.licm != 0;
}

struct WarpSmem {
  int32_t* t;          // [32] engine cursors
  int32_t* lr;         // [32] engine last retire
  int32_t* nn;         // [32] engine datapath instances so far
  int32_t* semv;       // [cap] increments processed
  int64_t* semhb;      // [cap] history base
  uint32_t* grp;       // [cap] lanes of the current chunk that increment it
  int32_t* tag;        // [cap] chunk that wrote grp
  int32_t* ring;       // [cap][ring] retire times of the latest increments
  uint8_t* rank_lane;  // [cap][32] lane of the chunk's k-th increment (k from 0)
  int32_t rmask;       // ring - 1
  Frame* frames;       // [depth]
  int2* lvl;           // [depth + 1] per level of the walk: {current iteration, start of its trip}
  unsigned long long* tally;  // [3] fused check: unsafe, over-synchronised, first offending pair
  int64_t* tlx;        // [2] piece runs: compact instance offset, probe (see tl_write)
};

// The timeline entry of instance o (instance layout).  Piece runs (stored
// times, PieceArgs.ptimes set) write the compact scratch instead: probe q's
// issue and retire at ptimes[2q * N + i] and ptimes[(2q + 1) * N + i], and
// (probe 0) the instance's position in its engine's stream at
// ptimes[2 * probes * N + i], i = o + the piece's compact offset.
__device__ __forceinline__ void tl_write(const SweepArgs& a, const WarpSmem& S, int64_t o, int32_t issue,
                                         int32_t retire, uint32_t nj) {
  if (a.pcs.ptimes) {
    const int64_t N = a.pcs.plen, i = o + S.tlx[0], q = S.tlx[1];
    a.pcs.ptimes[2 * q * N + i] = issue;
    a.pcs.ptimes[(2 * q + 1) * N + i] = retire;
    if (q == 0) a.pcs.ptimes[2 * (int64_t)a.pcs.probes * N + i] = (int32_t)nj;
  } else {
    a.issue[o] = issue;
    a.retire[o] = retire;
  }
}

// Fused simulation: the wait value of consumer-grouped dependency r for the
// consumer instance at global iteration gl of the loop at walk level lc
// (whose trip started at lo_c), from the walk's loop state -- the register
// form of Sec. 5.1 with r_S, r-hat_S read off the level of S.  With the
// optional check, the Eq. (1) minimum is evaluated beside it and a mismatch
// is tallied for the program.
template <int MODE>
__device__ __forceinline__ int32_t fused_wait(const SweepArgs& a, const WarpSmem& S, int r, int32_t gl, int lc,
                                              int32_t lo_c) {
  const DepInfo& D = a.dep[__ldg(a.ddep + r)];
  int32_t gs = gl, st = lo_c;
  if (D.up > 0) {
    const int2 v = S.lvl[lc - D.up];
    gs = v.x;
    st = v.y;
  }
  const int32_t T = wait_value(a, D, gs, st, MODE);
  if (a.chk_counts) {
    const int32_t m = minimum(a, D, gs, st, MODE);
    if (T != m) {
      atomicAdd(S.tally + (T < m ? 0 : 1), 1ull);
      atomicMin(S.tally + 2, (unsigned long long)(__ldg(a.dseg + r) + gl));
    }
  }
  return T;
}

// One lane's record of a chunk, with its first kMaxDeps dependencies.
struct LaneRec {
  int4 rec;                      // {global instruction, latency, dependencies, first dependency}
  int4 meta;                     // {engine, copy, first lane of the engine's run, flags}
  int4 sr;                       // {semaphore it increments or -1, stride, koff, 0}
  const int32_t* tp[kMaxDeps];   // threshold segment of dependency j
  int32_t sm[kMaxDeps];          // semaphore dependency j waits on
};

__device__ __forceinline__ void load_lane(const SweepArgs& a, const int4 ch, int lane, LaneRec& L) {
  L.rec = make_int4(0, 0, 0, 0);
  L.meta = make_int4(0, 0, lane, 0);
  L.sr = make_int4(-1, 0, 0, 0);
  if (lane < ch.y) {
    L.rec = __ldg(a.lrec + ch.x + lane);
    L.meta = __ldg(a.lmeta + ch.x + lane);
    L.sr = __ldg(a.lsem + ch.x + lane);
  }
#pragma unroll
  for (int j = 0; j < kMaxDeps; ++j) {
    L.tp[j] = a.thr;
    L.sm[j] = 0;
    if (j < L.rec.z) {
      L.tp[j] = a.thr + __ldg(a.dseg + L.rec.w + j);
      L.sm[j] = __ldg(a.dsem + L.rec.w + j);
    }
  }
}

// Thresholds of the lane's first kMaxDeps dependencies at its iteration gl
// of the loop at walk level lc (trip start lo_c): read from the threshold
// array, or (fused) from the walk's loop state.
template <int MODE, bool FUSED>
__device__ __forceinline__ void load_thr(const SweepArgs& a, const WarpSmem& S, const LaneRec& L, bool valid,
                                         int32_t gl, int lc, int32_t lo_c, int32_t (&T)[kMaxDeps]) {
#pragma unroll
  for (int j = 0; j < kMaxDeps; ++j) {
    if (FUSED) T[j] = (valid && j < L.rec.z) ? fused_wait<MODE>(a, S, L.rec.w + j, gl, lc, lo_c) : 0;
    else T[j] = (valid && j < L.rec.z) ? __ldg(L.tp[j] + gl) : 0;
  }
}

// Lanes that increment each semaphore in this chunk (`copies` iterations
// valid), published under tag ctag.
__device__ __forceinline__ void set_groups(const WarpSmem& S, const LaneRec& L, int lane, bool have,
                                           int32_t copies, int32_t ctag) {
  const bool prod = have && L.meta.y < copies && L.sr.x >= 0;
  const unsigned pm = __ballot_sync(kFull, prod);
  if (prod) {
    const unsigned peers = __match_any_sync(pm, L.sr.x);
    if (lane == __ffs(peers) - 1) { S.grp[L.sr.x] = peers; S.tag[L.sr.x] = ctag; }
    unsigned lt;
    asm("mov.u32 %0, %%lanemask_lt;" : "=r"(lt));
    S.rank_lane[L.sr.x * 32 + __popc(peers & lt)] = (uint8_t)lane;
  }
  __syncwarp();
}

// Barrier scheme, iterations of one loop through run_chunk: the lane's
// schedule of the last fully computed iteration relative to its start, and
// the in-chunk increments its waits targeted.
struct BbRep {
  bool on = false;
  int32_t sig = 0, issue = 0, retire = 0, t = 0;
};

// Barrier-free, whole iterations of one loop through run_chunk: the lane's
// issue and retire in the last computed iteration and their change since
// the one before (n: iterations computed so far).
struct BfPred {
  int n = 0;
  int32_t issue = 0, retire = 0, d_issue = 0, d_retire = 0;
};

// One chunk: `copies` iterations (g .. g+copies-1) of a segment's records,
// given the lane's record, its first thresholds T and the semaphore groups
// of this chunk (set_groups with the same copies and ctag).  Returns 0,
// SYNC_PROG_DEADLOCK or SIM_FALLBACK.  REP (barrier scheme, consecutive
// iterations of one loop): see the replay below.
template <int MODE, bool BB, bool TL, bool FUSED, bool REP = false, bool PRED = false>
__device__ __forceinline__ int run_chunk(const SweepArgs& a, const WarpSmem& S, const int4 ch, const LaneRec& L,
                                         const int32_t (&T)[kMaxDeps], int32_t g, int32_t copies,
                                         int32_t ctag, int lane, int lc, int32_t lo_c, int32_t iter_cost,
                                         unsigned long long& chk, BbRep& rp, BfPred& pd) {
  const int4 rec = L.rec, sr = L.sr;
  const bool have = lane < ch.y;
  const bool valid = have && L.meta.y < copies;
  const int32_t e = L.meta.x, head = L.meta.z;
  const int32_t gl = g + L.meta.y;
  const int32_t t_in = S.t[e], lr_in = S.lr[e], n_in = S.nn[e];
  const bool prod = valid && sr.x >= 0;
  const int32_t pub_own = prod ? S.semv[sr.x] : 0;

  // waits: increments before this chunk from the ring (or, if older, the
  // history), increments inside it by lane
  int32_t known = kNeg;                        // satisfied before this chunk (kNeg: none)
  int intra[kMaxIntra];
  int n_intra = 0;
  bool fallback = false;
  auto wait_on = [&](int32_t Tj, int32_t s) {
    if (Tj <= 0 || fallback) return;
    const int32_t pub = S.semv[s];
    if (Tj <= pub) {
      const int32_t r = pub - Tj <= S.rmask ? S.ring[s * (S.rmask + 1) + ((Tj - 1) & S.rmask)]
                                            : a.hist[S.semhb[s] + (Tj - 1)];
      known = max(known, r);
      return;
    }
    const unsigned m = S.tag[s] == ctag ? S.grp[s] : 0u;
    const int k = Tj - pub;
    if (k > __popc(m) || n_intra == kMaxIntra) { fallback = true; return; }
    const int src = S.rank_lane[s * 32 + k - 1];
#pragma unroll
    for (int i = 0; i < kMaxIntra; ++i)
      if (i == n_intra) intra[i] = src;         // static indices: intra stays in registers
    ++n_intra;
  };
#pragma unroll
  for (int j = 0; j < kMaxDeps; ++j)
    if (valid && j < rec.z) wait_on(T[j], L.sm[j]);
  for (int j = kMaxDeps; valid && j < rec.z; ++j)
    wait_on(FUSED ? fused_wait<MODE>(a, S, rec.w + j, gl, lc, lo_c) : __ldg(a.thr + __ldg(a.dseg + rec.w + j) + gl),
            __ldg(a.dsem + rec.w + j));
  if (__ballot_sync(kFull, fallback)) return SIM_FALLBACK;

  const int32_t wcost = BB ? 0 : wait_ops<MODE>(a, rec, sr.w);
  // iter_cost is the iteration-start cost of lane `lane`'s engine (engines
  // differ only by LICM's cached-sum updates); a record takes its engine's
  const int32_t ic_e = hoists<MODE, BB>(a) ? __shfl_sync(kFull, iter_cost, e) : iter_cost;
  const int32_t apre = (L.meta.w & LANE_ITER_START) ? ic_e : 0;
  const int32_t A = valid ? apre + wcost + a.prm.ii : 0;
  int32_t issue = 0, retire = 0, t_after = 0;
  // REP: every engine starts the iteration at the same cursor t_in with all
  // earlier work retired (the barriers before the loop statement and after
  // each iteration), so only in-chunk waits can bind and the schedule
  // relative to t_in depends only on which in-chunk increments the waits
  // target (their source lanes, 5 bits each, and their count): the same
  // targets as the last computed iteration give its schedule, shifted
  int32_t sig = 0;
  bool replay = false;
  if (REP) {
    sig = n_intra;
#pragma unroll
    for (int i = 0; i < kMaxIntra; ++i)
      if (i < n_intra) sig |= intra[i] << (3 + 5 * i);
    replay = rp.on && !__ballot_sync(kFull, valid && sig != rp.sig);
  }
  // PRED (barrier-free, whole iterations): extrapolate each lane's issue and
  // retire from the last two iterations and run one pass of the model on
  // it; if the pass reproduces the prediction on every lane, the prediction
  // is a fixed point of the chunk's equations -- and they have exactly one
  // (a cycle of waits admits none: along it each issue would have to follow
  // its own retirement), so it is the schedule the relaxation would reach
  bool predicted = false;
  if (PRED && pd.n >= 2) {
    const int32_t pi_ = pd.issue + pd.d_issue, pr_ = pd.retire + pd.d_retire;
    int32_t nr = kNeg;
#pragma unroll
    for (int i = 0; i < kMaxIntra; ++i) {
      const int32_t src = i < n_intra ? intra[i] : lane;
      const int32_t rv = __shfl_sync(kFull, pr_, src);
      if (i < n_intra) nr = max(nr, rv);
    }
    const int32_t ready = max(known, nr);
    int32_t Ai = A, Bi = (valid && ready >= 0) ? ready + a.prm.ii : kNeg;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t Ap = __shfl_up_sync(kFull, Ai, o), Bp = __shfl_up_sync(kFull, Bi, o);
      if (lane - o >= head) { Bi = max(Bp + Ai, Bi); Ai = Ap + Ai; }
    }
    const int32_t ta = max(t_in + Ai, Bi);
    int32_t vv = valid ? ta - a.prm.ii + rec.y : kNeg;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t vp = __shfl_up_sync(kFull, vv, o);
      if (lane - o >= head) vv = max(vv, vp);
    }
    const int32_t rt = max(lr_in, vv);
    predicted = !__ballot_sync(kFull, valid && (ta - a.prm.ii != pi_ || rt != pr_));
    if (predicted) {
      t_after = ta;
      issue = ta - a.prm.ii;
      retire = rt;
    }
  }
  if (replay) {
    issue = t_in + rp.issue;
    retire = t_in + rp.retire;
    t_after = t_in + rp.t;
  } else if (!predicted) {
  int32_t r_intra = kNeg;                      // retire of in-chunk producers (lower bound)
  const bool any_intra = __ballot_sync(kFull, n_intra > 0) != 0;
  const int passes = any_intra ? ch.y + 2 : 1;
  bool settled = false;
  for (int pass = 0; pass < passes; ++pass) {
    const int32_t ready = max(known, r_intra);
    const int32_t B0 = (valid && ready >= 0) ? ready + a.prm.ii : kNeg;
    // segmented inclusive scan of the cursor maps over the engine's run;
    // t' = max(t + A, B) with B = ready + ii gives issue = t' - ii
    int32_t Ai = A, Bi = B0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t Ap = __shfl_up_sync(kFull, Ai, o), Bp = __shfl_up_sync(kFull, Bi, o);
      if (lane - o >= head) { Bi = max(Bp + Ai, Bi); Ai = Ap + Ai; }
    }
    t_after = max(t_in + Ai, Bi);
    issue = t_after - a.prm.ii;
    int32_t v = valid ? issue + rec.y : kNeg;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t vp = __shfl_up_sync(kFull, v, o);
      if (lane - o >= head) v = max(v, vp);
    }
    retire = max(lr_in, v);
    if (!any_intra) { settled = true; break; }
    // new lower bound from the in-chunk producers' retire times; settled
    // once it binds nowhere (no issue would move)
    int32_t nr = kNeg;
#pragma unroll
    for (int i = 0; i < kMaxIntra; ++i) {
      const int32_t src = i < n_intra ? intra[i] : lane;
      const int32_t rv = __shfl_sync(kFull, retire, src);
      if (i < n_intra) nr = max(nr, rv);
    }
    if (!__ballot_sync(kFull, valid && nr > issue)) { settled = true; break; }
    r_intra = nr;
  }
  if (!settled) return SYNC_PROG_DEADLOCK;   // a cycle of waits inside the chunk
  if (REP) {
    rp.on = true;
    rp.sig = sig;
    rp.issue = issue - t_in;
    rp.retire = retire - t_in;
    rp.t = t_after - t_in;
  }
  }
  if (PRED) {
    pd.d_issue = issue - pd.issue;
    pd.d_retire = retire - pd.retire;
    pd.issue = issue;
    pd.retire = retire;
    ++pd.n;
  }

  // publish increments, instance counts, checksum terms, engine state
  const unsigned vm = __ballot_sync(kFull, valid);
  const unsigned run_le = vm & lanemask_le() & ~((1u << head) - 1u);
  const uint32_t nj = (uint32_t)n_in + __popc(run_le);   // the instance's position in its engine's stream
  if (prod) {
    // the increment this retirement makes: per-engine semaphores count the
    // engine's instances, the others a fixed number per iteration
    const int32_t n = sr.y < 0 ? (int32_t)nj : sr.y * gl + sr.z;
    S.ring[sr.x * (S.rmask + 1) + ((n - 1) & S.rmask)] = retire;
    a.hist[S.semhb[sr.x] + (n - 1)] = retire;
  }
  if (valid) {
    chk += inst_term(issue, retire, (uint32_t)e, nj);
    if (TL) tl_write(a, S, __ldg(a.inst_off + rec.x) + gl, issue, retire, nj);
  }
  __syncwarp();
  if (prod) {
    const unsigned grp = S.grp[sr.x];
    if (lane == 31 - __clz(grp)) S.semv[sr.x] = pub_own + __popc(grp);
  }
  if (have && (L.meta.w & LANE_RUN_LAST)) {
    S.t[e] = t_after;
    S.lr[e] = retire;
    S.nn[e] = n_in + __popc(run_le);
  }
  __syncwarp();
  // engines without records here still pass the iteration starts between copies
  if (copies > 1 && !((ch.w >> lane) & 1)) S.t[lane] += (copies - 1) * iter_cost;
  __syncwarp();
  return 0;
}

// All engines: the drain-and-release barrier of the barrier scheme.
__device__ __forceinline__ void barrier_all(const WarpSmem& S, int ne, int32_t c_barrier, int lane) {
  int32_t arr = lane < ne ? max(S.t[lane], S.lr[lane]) : 0;
  arr = (int32_t)__reduce_max_sync(kFull, (unsigned)arr);
  __syncwarp();
  if (lane < ne) S.t[lane] = arr + c_barrier;
  __syncwarp();
}

// Fused simulation inside a register-resident loop (levels: the loop is at
// walk level lc, its trip is [lo, hi)).  Per waited dependency, either a
// value fixed for the whole loop (S encloses the loop: fk = -1, value in fc),
// or -- S being the loop itself, so the producer sits in it -- fk = k and the
// per-loop encoding's N and N-K in fc, fn; per-engine values (fk = -2) are
// evaluated in full for every iteration.
template <int MODE>
__device__ __forceinline__ void fused_setup(const SweepArgs& a, const WarpSmem& S, int r, int32_t lo, int32_t hi,
                                            int32_t copy, int32_t copies, int lc, int32_t& fk, int32_t& fc,
                                            int32_t& fn) {
  const DepInfo& D = a.dep[__ldg(a.ddep + r)];
  if (D.up == 0) {
    fk = MODE == SYNC_THR_PERENGINE ? -2 : D.k;
    fc = D.N;
    fn = D.N - D.K;
    return;
  }
  fk = -1;
  const int2 v = S.lvl[lc - D.up];
  fc = wait_value(a, D, v.x, v.y, MODE);
  if (a.chk_counts) {
    const int32_t m = minimum(a, D, v.x, v.y, MODE);
    if (fc != m) {                 // the same mismatch at each of the lane's iterations
      atomicAdd(S.tally + (fc < m ? 0 : 1), (unsigned long long)((hi - lo - copy + copies - 1) / copies));
      atomicMin(S.tally + 2, (unsigned long long)(__ldg(a.dseg + r) + lo + copy));
    }
  }
}

template <int MODE>
__device__ __forceinline__ int32_t fused_iter(const SweepArgs& a, const WarpSmem& S, int r, int32_t fk, int32_t fc,
                                              int32_t fn, int32_t gl, int32_t lo, int lc) {
  if (fk == -1) return fc;
  if (fk == -2) return fused_wait<MODE>(a, S, r, gl, lc, lo);
  // Eq. (2) with S = this loop: r-hat_S = gl - lo + 1, expr = r_S - k
  const int32_t c = gl - lo + 1 > fk ? gl + 1 - fk : 0;
  const int32_t T = c == 0 ? 0 : MODE == SYNC_THR_PERLOOP ? fc * c - fn : c;
  if (a.chk_counts) {
    // Eq. (1): target position tS in this trip, producers through it
    const int32_t tS = gl - lo + 1 - fk;
    const int32_t cm = tS > 0 ? lo + tS : 0;
    const int32_t m = cm == 0 ? 0 : MODE == SYNC_THR_PERLOOP ? fc * cm - fn : cm;
    if (T != m) {
      atomicAdd(S.tally + (T < m ? 0 : 1), 1ull);
      atomicMin(S.tally + 2, (unsigned long long)(__ldg(a.dseg + r) + gl));
    }
  }
  return T;
}

// Iterations lo .. hi-1 of a loop whose body is one straight-line segment of
// one chunk (or, barrier-free, one multi-iteration chunk) and whose lanes
// wait on at most kMaxDeps semaphores each; the first iteration start has
// been charged.  Everything the iterations pass on stays in registers: lane
// e < ne holds engine e's cursor, last retire and instance count and hands
// them to its engine's lanes by shuffle; every lane keeps its record, its
// waited semaphores' increment counts and the next iteration's thresholds.
// Returns 0, SYNC_PROG_DEADLOCK or SIM_FALLBACK (then the program is
// abandoned, so nothing is written back).
template <int MODE, bool BB, bool TL, bool FUSED>
__device__ __forceinline__ int run_loop_regs(const SweepArgs& a, const WarpSmem& S, const ProgInfo& pi,
                                             const int4 ch, const LaneRec& L, int32_t lo, int32_t hi,
                                             int32_t ctag, int lane, int lc, int32_t iter_cost,
                                             unsigned long long& chk) {
  const int32_t ii = a.prm.ii;
  const int32_t copies = ch.z;
  const bool have = lane < ch.y;
  const int32_t e = L.meta.x, head = L.meta.z, copy = L.meta.y, lat = L.rec.y;
  const int ndep = have ? L.rec.z : 0;
  const unsigned run_from_head = ~((1u << head) - 1u);

  // semaphore groups of the chunk and the increment counts so far
  set_groups(S, L, lane, have, copies, ctag);
  uint32_t wg0 = 0, wg1 = 0;
  int32_t pub0 = 0, pub1 = 0;
  int32_t ring0 = 0, ring1 = 0;                       // ring rows of the waited semaphores
  if (ndep > 0) {
    const int32_t s = L.sm[0];
    wg0 = S.tag[s] == ctag ? S.grp[s] : 0u;
    pub0 = S.semv[s];
    ring0 = s * (S.rmask + 1);
  }
  if (ndep > 1) {
    const int32_t s = L.sm[kMaxDeps > 1 ? 1 : 0];
    wg1 = S.tag[s] == ctag ? S.grp[s] : 0u;
    pub1 = S.semv[s];
    ring1 = s * (S.rmask + 1);
  }
  const bool prod_lane = have && L.sr.x >= 0;
  const uint32_t own_grp = prod_lane ? S.grp[L.sr.x] : 0u;
  int32_t own_pub = prod_lane ? S.semv[L.sr.x] : 0;
  const int32_t own_ring = (prod_lane ? L.sr.x : 0) * (S.rmask + 1);
  const int64_t own_hist = prod_lane ? S.semhb[L.sr.x] - 1 : 0;
  const int32_t own_stride = L.sr.y, own_koff = L.sr.z;
  int64_t tl_off = 0;
  if (TL && have) tl_off = __ldg(a.inst_off + L.rec.x);

  // state lanes: engine `lane`'s run in the chunk (if any)
  const unsigned lastm = __ballot_sync(kFull, have && (L.meta.w & LANE_RUN_LAST));
  const bool present = lane < pi.ne && ((ch.w >> lane) & 1);
  int my_last = lane;
  unsigned my_run = 0;
  if (present) {
    const int rank = __popc((unsigned)ch.w & ((1u << lane) - 1u));
    my_last = (int)__fns(lastm, 0, rank + 1);
    const int first = rank == 0 ? 0 : (int)__fns(lastm, 0, rank) + 1;
    my_run = (my_last == 31 ? kFull : ((1u << (my_last + 1)) - 1u)) & ~((1u << first) - 1u);
  }
  int32_t ts = 0, lrs = 0, ns = 0;
  if (lane < pi.ne) { ts = S.t[lane]; lrs = S.lr[lane]; ns = S.nn[lane]; }

  // barrier scheme: relative schedule of the last fully computed iteration
  bool rep = false;
  int32_t rd_issue = 0, rd_retire = 0, rd_t = 0, rd_r = 0, rk0 = 0, rk1 = 0;

  const int32_t wcost = BB ? 0 : wait_ops<MODE>(a, L.rec, L.sr.w);
  // iter_cost: the iteration-start cost of lane `lane`'s engine (state
  // lanes); a record lane takes its engine's
  const int32_t ic_e = hoists<MODE, BB>(a) ? __shfl_sync(kFull, iter_cost, e) : iter_cost;
  const int32_t P = wcost + ((L.meta.w & LANE_ITER_START) ? ic_e : 0);
  const int32_t A = P + ii;                           // cursor advance of a valid lane with no wait
  int32_t T0n = 0, T1n = 0;
  int32_t fk0 = -1, fc0 = 0, fn0 = 0, fk1 = -1, fc1 = 0, fn1 = 0;   // fused: see fused_setup
  if (FUSED) {
    const bool vn = have && copy < hi - lo;
    if (vn && ndep > 0) fused_setup<MODE>(a, S, L.rec.w, lo, hi, copy, copies, lc, fk0, fc0, fn0);
    if (vn && ndep > 1) fused_setup<MODE>(a, S, L.rec.w + 1, lo, hi, copy, copies, lc, fk1, fc1, fn1);
  } else {
    const bool vn = have && copy < hi - lo;
    if (vn && ndep > 0) T0n = __ldg(L.tp[0] + lo + copy);
    if (vn && ndep > 1) T1n = __ldg(L.tp[kMaxDeps > 1 ? 1 : 0] + lo + copy);
  }
  for (int32_t g = lo; g < hi;) {
    // barrier scheme, array pipeline: a run of iterations that all replay the
    // reference (their waits target the same in-chunk increments, none past
    // the chunk's) in one pass.  Each starts at a barrier with every engine
    // at the same cursor and everything earlier retired, so iteration j of
    // the run starts at base + j*D, D = the reference's largest end (cursor
    // or last retire) past its base, plus the barrier and the iteration
    // start; its times are the reference's shifted by its start.
    if (BB && !FUSED && rep && copies == 1) {
      const unsigned vm = __ballot_sync(kFull, have);
      const int32_t inc0 = __popc(wg0 & vm), inc1 = __popc(wg1 & vm);
      const int32_t B = min(hi - g, 32);
      int jm = B;                                     // this lane: first iteration that does not replay
      if (have) {
        for (int j = 0; j < jm; ++j) {
          int k0 = 0, k1 = 0;
          if (ndep > 0) {
            const int32_t T = __ldg(L.tp[0] + g + j), pb = pub0 + j * inc0;
            if (T > pb) k0 = T - pb <= inc0 ? T - pb : -1;   // -1: past the chunk's increments
          }
          if (ndep > 1) {
            const int32_t T = __ldg(L.tp[kMaxDeps > 1 ? 1 : 0] + g + j), pb = pub1 + j * inc1;
            if (T > pb) k1 = T - pb <= inc1 ? T - pb : -1;
          }
          if (k0 != rk0 || k1 != rk1) jm = j;
        }
      }
      const int32_t J = (int32_t)__reduce_min_sync(kFull, (unsigned)jm);
      if (J > 0) {
        const int32_t base = __shfl_sync(kFull, ts, 0);
        const int32_t M = max(0, __reduce_max_sync(kFull, lane < pi.ne && present ? max(rd_t, rd_r) : 0));
        const int32_t D = M + a.prm.c_barrier + __shfl_sync(kFull, iter_cost, 0);
        const int32_t cnt = present ? __popc(vm & my_run) : 0;   // engine `lane`'s instances per iteration
        const int32_t cnt_e = __shfl_sync(kFull, cnt, e), n_e = __shfl_sync(kFull, ns, e);
        const int32_t rank = __popc(vm & lanemask_le() & run_from_head);
        if (have) {
          for (int32_t j = 0; j < J; ++j) {
            const int32_t bj = base + j * D, issue = bj + rd_issue, retire = bj + rd_retire;
            const int32_t gl = g + j;
            const uint32_t nj = (uint32_t)(n_e + j * cnt_e + rank);
            if (prod_lane) {
              const int32_t n = own_stride < 0 ? (int32_t)nj : own_stride * gl + own_koff;
              S.ring[own_ring + ((n - 1) & S.rmask)] = retire;
              a.hist[own_hist + n] = retire;
            }
            chk += inst_term(issue, retire, (uint32_t)e, nj);
            if (TL) tl_write(a, S, tl_off + gl, issue, retire, nj);
          }
        }
        pub0 += J * inc0;
        pub1 += J * inc1;
        own_pub += J * __popc(own_grp & vm);
        const int32_t blast = base + (J - 1) * D;     // the run's last iteration
        if (lane < pi.ne) {
          if (present) {
            lrs = blast + rd_r;
            ns += J * cnt;
          }
          ts = blast + M + a.prm.c_barrier + (g + J < hi ? iter_cost : 0);
        }
        __syncwarp();                                 // ring entries visible to the next iteration
        g += J;
        if (g < hi) {
          if (have && ndep > 0) T0n = __ldg(L.tp[0] + g);
          if (have && ndep > 1) T1n = __ldg(L.tp[kMaxDeps > 1 ? 1 : 0] + g);
        }
        continue;
      }
    }
    const int32_t v = min(copies, hi - g);
    int32_t T0, T1;
    if (FUSED) {
      T0 = have && copy < v && ndep > 0 ? fused_iter<MODE>(a, S, L.rec.w, fk0, fc0, fn0, g + copy, lo, lc) : 0;
      T1 = have && copy < v && ndep > 1 ? fused_iter<MODE>(a, S, L.rec.w + 1, fk1, fc1, fn1, g + copy, lo, lc) : 0;
    } else {
      T0 = T0n;
      T1 = T1n;
    }
    const int32_t gn = g + v;
    const bool valid = have && copy < v;
    if (!FUSED && gn < hi) {
      const bool vn = have && copy < hi - gn;
      if (vn && ndep > 0) T0n = __ldg(L.tp[0] + gn + copy);
      if (vn && ndep > 1) T1n = __ldg(L.tp[kMaxDeps > 1 ? 1 : 0] + gn + copy);
    }
    const unsigned vm = __ballot_sync(kFull, valid);
    const int32_t gl = g + copy;
    const int32_t t_in = __shfl_sync(kFull, ts, e), lr_in = __shfl_sync(kFull, lrs, e);
    const int32_t n_in = __shfl_sync(kFull, ns, e);

    // waits: earlier increments from the ring or history, in-chunk ones by lane
    // (barrier scheme: an increment before this iteration retired before the
    // barrier that ended the last iteration or opened the loop, so that wait
    // never binds)
    int32_t known = kNeg;
    int k0 = 0, k1 = 0;                               // in-chunk increment waited on (1-based), or 0
    bool fallback = false;
    if (valid && T0 > 0) {
      if (T0 <= pub0) {
        if (!BB) known = pub0 - T0 <= S.rmask ? S.ring[ring0 + ((T0 - 1) & S.rmask)]
                                              : a.hist[S.semhb[L.sm[0]] + (T0 - 1)];
      } else {
        k0 = T0 - pub0;
        if (k0 > __popc(wg0 & vm)) fallback = true;
      }
    }
    if (valid && T1 > 0) {
      if (T1 <= pub1) {
        if (!BB) known = max(known, pub1 - T1 <= S.rmask ? S.ring[ring1 + ((T1 - 1) & S.rmask)]
                                                         : a.hist[S.semhb[L.sm[kMaxDeps > 1 ? 1 : 0]] + (T1 - 1)]);
      } else {
        k1 = T1 - pub1;
        if (k1 > __popc(wg1 & vm)) fallback = true;
      }
    }
    if (__ballot_sync(kFull, fallback)) return SIM_FALLBACK;

    int32_t issue = 0, retire = 0, t_last = 0, r_last = 0;
    // barrier scheme: every engine starts the iteration at the same cursor
    // `base` with everything earlier retired, and only in-chunk waits can
    // bind, so an iteration whose waits target the same in-chunk increments
    // as the last fully computed one has that iteration's schedule shifted
    // by the difference of the bases
    const int32_t base = BB ? __shfl_sync(kFull, ts, 0) : 0;
    if (BB && rep && !__ballot_sync(kFull, k0 != rk0 || k1 != rk1)) {
      issue = base + rd_issue;
      retire = base + rd_retire;
      t_last = base + rd_t;
      r_last = base + rd_r;
    } else {
      const int src0 = k0 > 0 ? S.rank_lane[L.sm[0] * 32 + k0 - 1] : -1;
      const int src1 = k1 > 0 ? S.rank_lane[L.sm[kMaxDeps > 1 ? 1 : 0] * 32 + k1 - 1] : -1;
      const unsigned intra = __ballot_sync(kFull, src0 >= 0 || src1 >= 0);
      const int32_t Av = valid ? A : 0;
      int32_t r_intra = kNeg, t_after = 0;
      const int passes = intra ? ch.y + 2 : 1;
      bool settled = false;
      for (int pass = 0; pass < passes; ++pass) {
        const int32_t ready = max(known, r_intra);
        // segmented scan of t' = max(t + A, B), B = ready + ii: issue = t' - ii
        int32_t Ai = Av, Bi = (valid && ready >= 0) ? ready + ii : kNeg;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int32_t Ap = __shfl_up_sync(kFull, Ai, o), Bp = __shfl_up_sync(kFull, Bi, o);
          if (lane - o >= head) { Bi = max(Bp + Ai, Bi); Ai += Ap; }
        }
        t_after = max(t_in + Ai, Bi);
        issue = t_after - ii;
        // in-order retirement: segmented max-scan of issue + latency
        int32_t rv = valid ? issue + lat : kNeg;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int32_t vp = __shfl_up_sync(kFull, rv, o);
          if (lane - o >= head) rv = max(rv, vp);
        }
        retire = max(lr_in, rv);
        if (!intra) { settled = true; break; }
        const int32_t p0 = __shfl_sync(kFull, retire, src0 < 0 ? lane : src0);
        const int32_t p1 = __shfl_sync(kFull, retire, src1 < 0 ? lane : src1);
        const int32_t nr = max(src0 < 0 ? kNeg : p0, src1 < 0 ? kNeg : p1);
        if (!__ballot_sync(kFull, valid && nr > issue)) { settled = true; break; }   // binds nowhere
        r_intra = nr;
      }
      if (!settled) return SYNC_PROG_DEADLOCK;
      t_last = __shfl_sync(kFull, t_after, my_last);
      r_last = __shfl_sync(kFull, retire, my_last);
      if (BB) {                                       // the reference for the next iterations
        rd_issue = issue - base;
        rd_retire = retire - base;
        rd_t = t_last - base;
        rd_r = r_last - base;
        rk0 = k0;
        rk1 = k1;
        rep = true;
      }
    }

    // publish
    const uint32_t nj = (uint32_t)n_in + __popc(vm & lanemask_le() & run_from_head);
    if (valid && prod_lane) {
      const int32_t n = own_stride < 0 ? (int32_t)nj : own_stride * gl + own_koff;
      S.ring[own_ring + ((n - 1) & S.rmask)] = retire;
      a.hist[own_hist + n] = retire;
    }
    if (valid) {
      chk += inst_term(issue, retire, (uint32_t)e, nj);
      if (TL) tl_write(a, S, tl_off + gl, issue, retire, nj);
    }
    pub0 += __popc(wg0 & vm);
    pub1 += __popc(wg1 & vm);
    own_pub += __popc(own_grp & vm);
    if (present) {
      ts = t_last;
      lrs = r_last;
      ns += __popc(vm & my_run);
    } else if (v > 1 && lane < pi.ne) {
      ts += (v - 1) * iter_cost;                      // iteration starts between copies
    }
    __syncwarp();                                     // ring entries visible to the next iteration
    g = gn;
    if (BB) {
      const int32_t arr = (int32_t)__reduce_max_sync(kFull, lane < pi.ne ? (unsigned)max(ts, lrs) : 0u);
      if (lane < pi.ne) ts = arr + a.prm.c_barrier;
    }
    if (g < hi && lane < pi.ne) ts += iter_cost;
  }
  if (lane < pi.ne) { S.t[lane] = ts; S.lr[lane] = lrs; S.nn[lane] = ns; }
  if (prod_lane && lane == 31 - __clz(own_grp)) S.semv[L.sr.x] = own_pub;
  __syncwarp();
  return 0;
}

// A loop statement whose one iteration (global index g, walk level lc) runs
// a one-record chunk -- a conditional around one instruction, the common
// shape of synchronisation-bound code: the instance's cursor map applied
// directly, without scans.  Lane 0 takes the wait decisions (so a fused
// check counts each pair once); the verdicts are run_chunk's: a wait past
// the published increments hands the program over, one on its own
// increment is a cycle.
template <int MODE, bool BB, bool TL, bool FUSED>
__device__ __forceinline__ int run_single(const SweepArgs& a, const WarpSmem& S, const ProgInfo& pi,
                                          const int4 ch, int32_t g, int lane, int lc,
                                          unsigned long long& chk) {
  const int4 rec = __ldg(a.lrec + ch.x), sr = __ldg(a.lsem + ch.x);
  const int32_t e = __ldg(a.lmeta + ch.x).x;
  int32_t ready = kNeg;
  int flag = 0;                                 // 1: a cycle, 2: handed over
  if (lane == 0) {
    for (int j = 0; j < rec.z; ++j) {
      const int32_t T = FUSED ? fused_wait<MODE>(a, S, rec.w + j, g, lc, g)
                              : __ldg(a.thr + __ldg(a.dseg + rec.w + j) + g);
      if (T <= 0) continue;
      const int32_t s = __ldg(a.dsem + rec.w + j), pub = S.semv[s];
      if (T <= pub) {
        ready = max(ready, pub - T <= S.rmask ? S.ring[s * (S.rmask + 1) + ((T - 1) & S.rmask)]
                                              : a.hist[S.semhb[s] + (T - 1)]);
      } else {
        flag = max(flag, s == sr.x && T - pub == 1 ? 1 : 2);
      }
    }
  }
  flag = __shfl_sync(kFull, flag, 0);
  if (flag == 2) return SIM_FALLBACK;
  if (flag == 1) return SYNC_PROG_DEADLOCK;
  ready = __shfl_sync(kFull, ready, 0);
  const int32_t wcost = BB ? 0 : wait_ops<MODE>(a, rec, sr.w);
  const int32_t t_in = S.t[e], lr_in = S.lr[e];
  const uint32_t nj = (uint32_t)S.nn[e] + 1;
  const int32_t t_after = max(t_in + wcost + a.prm.ii, ready >= 0 ? ready + a.prm.ii : kNeg);
  const int32_t issue = t_after - a.prm.ii, retire = max(lr_in, issue + rec.y);
  __syncwarp();
  if (lane == 0) {
    if (sr.x >= 0) {
      const int32_t n = sr.y < 0 ? (int32_t)nj : sr.y * g + sr.z;
      S.ring[sr.x * (S.rmask + 1) + ((n - 1) & S.rmask)] = retire;
      a.hist[S.semhb[sr.x] + (n - 1)] = retire;
      S.semv[sr.x] += 1;
    }
    chk += inst_term(issue, retire, (uint32_t)e, nj);
    if (TL) tl_write(a, S, __ldg(a.inst_off + rec.x) + g, issue, retire, nj);
    S.t[e] = t_after;
    S.lr[e] = retire;
    S.nn[e] = (int32_t)nj;
  }
  __syncwarp();
  if (BB) barrier_all(S, pi.ne, a.prm.c_barrier, lane);
  return 0;
}

// Iterations lo .. hi-1 of a loop whose body is one straight-line segment of
// one chunk (or, barrier-free, one multi-iteration chunk); the first
// iteration start has been charged.  The lane's record and thresholds stay
// in registers; the next chunk's thresholds load while this one runs.
// `one`: with a single iteration, the chunk holding its whole body
// (zeros otherwise); a chunk of one record is applied directly.
template <int MODE, bool BB, bool TL, bool FUSED>
__device__ __forceinline__ int run_loop(const SweepArgs& a, const WarpSmem& S, const ProgInfo& pi, const int4 ch,
                                        const int4 one, int32_t lo, int32_t hi, int32_t ctag, int lane, int lc,
                                        int32_t iter_cost, unsigned long long& chk) {
  if (one.y == 1) return run_single<MODE, BB, TL, FUSED>(a, S, pi, one, lo, lane, lc, chk);
  const int32_t copies = ch.z;
  const bool have = lane < ch.y;
  LaneRec L;
  load_lane(a, ch, lane, L);
  if (!__ballot_sync(kFull, have && L.rec.z > kMaxDeps))
    return run_loop_regs<MODE, BB, TL, FUSED>(a, S, pi, ch, L, lo, hi, ctag, lane, lc, iter_cost, chk);
  set_groups(S, L, lane, have, min(copies, hi - lo), ctag);
  int32_t Tn[kMaxDeps];
  load_thr<MODE, FUSED>(a, S, L, have && L.meta.y < hi - lo, lo + L.meta.y, lc, lo, Tn);
  BbRep rp;                                     // barrier scheme: replayed iterations
  BfPred pd;                                    // barrier-free: predicted iterations
  for (int32_t g = lo; g < hi;) {
    const int32_t v = min(copies, hi - g);
    int32_t T[kMaxDeps];
#pragma unroll
    for (int j = 0; j < kMaxDeps; ++j) T[j] = Tn[j];
    const int32_t gn = g + v;
    if (gn < hi) load_thr<MODE, FUSED>(a, S, L, have && L.meta.y < hi - gn, gn + L.meta.y, lc, lo, Tn);
    if (v < copies && g > lo) set_groups(S, L, lane, have, v, ctag);   // the last, partial chunk
    if (!BB && v < copies) pd.n = 0;            // the last, partial chunk: not predicted
    const int verdict =
        run_chunk<MODE, BB, TL, FUSED, BB, !BB>(a, S, ch, L, T, g, v, ctag, lane, lc, lo, iter_cost, chk, rp, pd);
    if (verdict) return verdict;
    g = gn;
    if (BB) barrier_all(S, pi.ne, a.prm.c_barrier, lane);
    if (g < hi) {
      if (lane < pi.ne) S.t[lane] += iter_cost;
      __syncwarp();
    }
  }
  return 0;
}

// PIECE: the warp runs pieces of split programs (see PieceArgs) instead of
// whole programs: item = piece * probes + probe; the walk starts inside the
// body of the piece's loop L at its first iteration start and ends after
// its last iteration (barrier scheme: after that iteration's barrier).
template <int MODE, bool BB, bool TL, bool FUSED, bool PIECE = false>
__global__ void __launch_bounds__(kWarps * 32, 3) k_sweep(const SweepArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  WarpSmem S;
  {
    unsigned char* p = smem_raw + wib * warp_bytes(a.sem_cap, a.frame_depth, a.ring);
    // the walk-level table and check tallies go first in the barrier sweep and
    // last in the barrier-free one (a measured code-generation preference)
    S.semhb = reinterpret_cast<int64_t*>(p); p += 8 * a.sem_cap;
    if (BB) {
      S.tally = reinterpret_cast<unsigned long long*>(p); p += 3 * 8;
      S.lvl = reinterpret_cast<int2*>(p); p += 8 * (a.frame_depth + 1);
    }
    S.frames = reinterpret_cast<Frame*>(p); p += sizeof(Frame) * a.frame_depth;
    S.t = reinterpret_cast<int32_t*>(p); p += 4 * 32;
    S.lr = reinterpret_cast<int32_t*>(p); p += 4 * 32;
    S.nn = reinterpret_cast<int32_t*>(p); p += 4 * 32;
    S.semv = reinterpret_cast<int32_t*>(p); p += 4 * a.sem_cap;
    S.grp = reinterpret_cast<uint32_t*>(p); p += 4 * a.sem_cap;
    S.tag = reinterpret_cast<int32_t*>(p); p += 4 * a.sem_cap;
    S.ring = reinterpret_cast<int32_t*>(p); p += 4 * (size_t)a.ring * a.sem_cap;
    S.rank_lane = reinterpret_cast<uint8_t*>(p); p += 32 * (size_t)a.sem_cap;
    p = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(p) + 7) & ~uintptr_t(7));
    if (!BB) {
      S.tally = reinterpret_cast<unsigned long long*>(p); p += 3 * 8;
      S.lvl = reinterpret_cast<int2*>(p); p += 8 * (a.frame_depth + 1);
    }
    S.tlx = reinterpret_cast<int64_t*>(p);
    S.rmask = a.ring - 1;
  }
  const int32_t cwait = MODE == SYNC_THR_COUNT ? a.prm.c_wait_ops_count : a.prm.c_wait_ops_perloop;
  // iteration-start and statement costs of a loop; a loop flagged as
  // carrying only offset-0 dependencies keeps no trip register when the
  // elision is on (barrier-free: no r-hat := 0, no r-hat++)
  const bool elide = !BB && a.prm.trip_register_elision != 0;
  const int32_t ic_full = BB ? a.prm.c_branch : a.prm.c_branch + 2 * a.prm.c_regop;
  auto stmt_cost_of = [&](int32_t flag) { return elide && flag ? 0 : a.prm.c_regop; };

  const int32_t n_items = PIECE ? a.pcs.n_pieces * a.pcs.probes : a.n_programs;
  for (;;) {
    int slot = 0;
    if (lane == 0) slot = atomicAdd(a.next_slot, 1);
    slot = __shfl_sync(kFull, slot, 0);
    if (slot >= n_items) break;
    int piece = 0, probe = 0, p;
    PieceInfo pc;
    if (PIECE) {
      piece = slot / a.pcs.probes;
      probe = slot - piece * a.pcs.probes;
      pc = a.pcs.piece[piece];
      p = pc.prog;
    } else {
      p = __ldg(a.order + slot);
      // a split program simulated by its pieces in this call
      if (a.pcs.prog_split) {
        const int32_t sp_ = __ldg(a.pcs.prog_split + p);
        if (sp_ >= 0 && !*(volatile int32_t*)(a.pcs.fail + sp_)) continue;
      }
    }
    const ProgInfo pi = a.prog[p];
    if (PIECE) {
      // a failed validation, a probe past this program's state variables, a
      // program of the other barrier-free class, a speculative piece with no
      // run due
      if (*(volatile int32_t*)(a.pcs.fail + pc.split) || probe >= (BB || a.pcs.spec ? 1 : 2 * pi.ne)) continue;
      if (!BB && (__ldg(a.pcs.cls + pc.split) != 0) != (a.pcs.spec != 0)) continue;
      if (a.pcs.spec && !*(volatile int32_t*)(a.pcs.need + piece)) continue;
    }
    // the iteration-start cost of global loop `loop` on lane `lane`'s engine
    // (lanes past the engines: any value); flag: its trip register is elidable
    auto iter_cost_of = [&](int32_t flag, int32_t loop) {
      int32_t c = elide && flag ? ic_full - a.prm.c_regop : ic_full;
      if (hoists<MODE, BB>(a) && lane < pi.ne) c += hoist_ops<MODE, BB>(a, pi.le_base + (loop - pi.loop_base) * pi.ne + lane);
      return c;
    };
    BbRep no_rep;                     // a segment's chunk is neither replayed
    BfPred no_pred;                   // nor predicted
    // engines on their own trips (no common walk), or barrier-free with the
    // barriers of the non-allocatable fallback: the per-engine kernel (split
    // programs have neither; their time bound was checked by the validation)
    if (!PIECE && (pi.divergent || (!BB && pi.fb_iters > 0))) {
      if (lane == 0) {
        a.status[p] = SIM_FALLBACK;
        a.fallback[1 + atomicAdd(a.fallback, 1)] = p;
      }
      continue;
    }
    if (!PIECE && time_bound<MODE, BB>(pi, a.prm, cwait) > 2147483647ull) {
      if (lane == 0) { a.makespan[p] = -1; a.checksum[p] = 0; a.status[p] = SYNC_PROG_OVERFLOW; }
      continue;
    }
    // probe runs write a private history (each probe its own); the barrier
    // scheme's and the speculated pieces' single runs write the real one
    const bool probe_hist = PIECE && !BB && !a.pcs.spec;
    for (int i = lane; i < pi.nsem[MODE]; i += 32) {
      S.semv[i] = PIECE ? __ldg(a.pcs.pub + pc.pub_off[MODE] + i) : 0;
      S.semhb[i] = __ldg(a.semhb + pi.semhb_off[MODE] + i);
      if (probe_hist) S.semhb[i] += pc.hdelta[MODE] + (int64_t)probe * a.pcs.phist_len - (a.hist - a.pcs.phist);
      S.tag[i] = -1;
    }
    if (PIECE) {
      // the start state: probe `probe` raises state variable `probe` (cursors
      // 0..ne-1, then last retires) by kProbe; the barrier scheme runs from
      // a release at 0.  The instances' times go to the compact scratch.
      int32_t t0 = !BB && lane == probe ? kProbe : 0, l0 = !BB && lane + pi.ne == probe ? kProbe : 0;
      if (a.pcs.spec && lane < pi.ne) {              // a speculative piece: its guessed start
        t0 = a.pcs.xhat[(int64_t)piece * 64 + lane];
        l0 = a.pcs.xhat[(int64_t)piece * 64 + 32 + lane];
      }
      S.t[lane] = t0; S.lr[lane] = l0;
      S.nn[lane] = lane < pi.ne ? __ldg(a.pcs.pub + pc.nbase_off + lane) : 0;
      if (lane == 0) { S.tlx[0] = pc.tl[BB || a.pcs.spec ? 0 : 1]; S.tlx[1] = probe; }
    } else {
      S.t[lane] = 0; S.lr[lane] = 0; S.nn[lane] = 0;
    }
    if (FUSED && lane == 0) {
      S.lvl[0] = make_int2(0, 0);                      // the top-level loop: iteration 0 of a trip at 0
      S.tally[0] = S.tally[1] = 0;
      S.tally[2] = ~0ull;
    }
    __syncwarp();
    unsigned long long chk = 0;
    int32_t loop = PIECE ? pc.loop : pi.loop_base, item = 0, g = PIECE ? pc.g0 : 0, g_end = PIECE ? pc.g1 : 1;
    int32_t sp = 0, ctag = 0;
    int32_t iter_cost = PIECE ? iter_cost_of(__ldg(a.lflag + loop), loop) : ic_full;   // of the loop being walked
    int32_t pbeg = __ldg(a.plan_ptr + loop), pend = __ldg(a.plan_ptr + loop + 1);
    int verdict = SYNC_PROG_OK;
    if (PIECE) {                                       // the piece's first iteration starts
      __syncwarp();
      if (lane < pi.ne) S.t[lane] += iter_cost;
      __syncwarp();
    }
    for (;;) {
      if (pbeg + item == pend) {                       // end of an iteration's body
        if (sp == 0) {
          if (!PIECE) break;                           // the top-level loop runs once
          // a piece: its loop's next iteration, or the end of the piece
          if (BB) barrier_all(S, pi.ne, a.prm.c_barrier, lane);
          if (++g >= g_end) break;
          if (lane < pi.ne) S.t[lane] += iter_cost;
          __syncwarp();
          item = 0;
          continue;
        }
        if (BB) barrier_all(S, pi.ne, a.prm.c_barrier, lane);
        if (++g < g_end) {
          if (lane < pi.ne) S.t[lane] += iter_cost;
          if (FUSED && lane == 0) S.lvl[sp].x = g;
          __syncwarp();
          item = 0;
        } else {
          const Frame f = S.frames[--sp];
          loop = f.loop; item = f.item; g = f.g; g_end = f.g_end;
          iter_cost = iter_cost_of(__ldg(a.lflag + loop), loop);
          pbeg = __ldg(a.plan_ptr + loop);
          pend = __ldg(a.plan_ptr + loop + 1);
        }
        continue;
      }
      // the item and its side record (a loop statement: the child's trip
      // prefix sums and the chunks holding its whole body; a segment: its
      // first chunk), read together; then a statement's trip bounds and
      // chunks, together
      const int4 it = __ldg(a.plan + pbeg + item);
      const int4 ax = __ldg(a.paux + pbeg + item);
      if (it.x == ITEM_LOOP) {                         // a loop statement
        const int64_t rp = (int64_t)(((uint64_t)(uint32_t)ax.y << 32) | (uint32_t)ax.x);
        const int32_t lo = __ldg(a.rowptr + rp + g), hi = __ldg(a.rowptr + rp + g + 1);
        const int32_t body_chunk = BB ? ax.w : ax.z;
        const int4 chb = body_chunk >= 0 ? __ldg(a.chunk + body_chunk) : make_int4(0, 0, 0, 0);
        const int4 one = ax.w < 0 ? make_int4(0, 0, 0, 0) : BB ? chb : __ldg(a.chunk + ax.w);
        if (BB) {
          barrier_all(S, pi.ne, a.prm.c_barrier, lane);
        } else {
          if (lane < pi.ne) S.t[lane] += stmt_cost_of(it.z);
        }
        const int32_t child_ic = iter_cost_of(it.z, it.y);
        ++item;
        if (lo < hi) {
          __syncwarp();
          if (lane < pi.ne) S.t[lane] += child_ic;    // the first iteration starts
          __syncwarp();
          if (body_chunk >= 0) {
            // one iteration of one record: applied directly; otherwise a
            // loop around one chunk: all its iterations in registers
            verdict = run_loop<MODE, BB, TL, FUSED>(a, S, pi, chb, hi - lo == 1 ? one : make_int4(0, 0, 0, 0), lo,
                                                    hi, ++ctag, lane, sp + 1, child_ic, chk);
            if (verdict) break;
            continue;
          }
          const int32_t cb = __ldg(a.plan_ptr + it.y), ce = __ldg(a.plan_ptr + it.y + 1);
          if (lane == 0) S.frames[sp] = Frame{loop, item, g, g_end};
          ++sp;
          if (FUSED && lane == 0) S.lvl[sp] = make_int2(lo, lo);
          loop = it.y; item = 0; g = lo; g_end = hi;
          iter_cost = child_ic;
          pbeg = cb;
          pend = ce;
        }
        __syncwarp();
        continue;
      }
      // a straight-line segment
      if (!BB && it.w != -1) {
        // several iterations of a short innermost body at once (w >= 0), or
        // the body's closing segment joined with the next iteration's
        // opening one, whose iteration start is inside the chunk (w <= -2):
        // unless this is the trip's last iteration the walk then goes on in
        // iteration g+1 past its opening segment
        const bool joined = it.w <= -2;
        const int4 ch = __ldg(a.chunk + (joined ? -2 - it.w : it.w));
        const int32_t v = min(ch.z, g_end - g);
        LaneRec Lr;
        load_lane(a, ch, lane, Lr);
        int32_t T[kMaxDeps];
        const int32_t lo_c = FUSED ? S.lvl[sp].y : 0;
        load_thr<MODE, FUSED>(a, S, Lr, lane < ch.y && Lr.meta.y < v, g + Lr.meta.y, sp, lo_c, T);
        set_groups(S, Lr, lane, lane < ch.y, v, ++ctag);
        verdict = run_chunk<MODE, BB, TL, FUSED>(a, S, ch, Lr, T, g, v, ctag, lane, sp, lo_c, iter_cost, chk, no_rep,
                                                  no_pred);
        if (verdict) break;
        if (joined && v == 2) {
          ++g;
          if (FUSED && lane == 0) S.lvl[sp].x = g;
          __syncwarp();
          item = 1;
          continue;
        }
        g += v - 1;
        item = pend - pbeg;                            // continue at the END of iteration g
        continue;
      }
      for (int c = 0; c < it.z && !verdict; ++c) {
        const int4 ch = c == 0 ? ax : __ldg(a.chunk + it.y + c);   // the first: read with the item
        LaneRec Lr;
        load_lane(a, ch, lane, Lr);
        int32_t T[kMaxDeps];
        const int32_t lo_c = FUSED ? S.lvl[sp].y : 0;
        load_thr<MODE, FUSED>(a, S, Lr, lane < ch.y, g, sp, lo_c, T);
        set_groups(S, Lr, lane, lane < ch.y, 1, ++ctag);
        verdict = run_chunk<MODE, BB, TL, FUSED>(a, S, ch, Lr, T, g, 1, ctag, lane, sp, lo_c, iter_cost, chk, no_rep,
                                                  no_pred);
      }
      if (verdict) break;
      ++item;
    }
    if (PIECE) {
      // any verdict but OK (a deadlock, a wait reaching forward): the
      // program is simulated whole by the sweep, which reports it
      if (verdict != SYNC_PROG_OK && lane == 0) atomicExch(a.pcs.fail + pc.split, 1);
      if (lane < pi.ne) {
        int32_t* o = a.pcs.out + ((int64_t)piece * a.pcs.out_probes + probe) * 64;
        o[lane] = S.t[lane];
        o[32 + lane] = S.lr[lane];
      }
      if (a.pcs.spec && lane == 0) { a.pcs.need[piece] = 0; a.pcs.has[piece] = 1; }
      __syncwarp();
      continue;
    }
    if (verdict == SIM_FALLBACK) {
      if (lane == 0) {
        a.status[p] = SIM_FALLBACK;
        const int i = atomicAdd(a.fallback, 1);
        a.fallback[1 + i] = p;
      }
      __syncwarp();
      continue;
    }
    int32_t ms = lane < pi.ne ? max(S.t[lane], S.lr[lane]) : 0;
    ms = (int32_t)__reduce_max_sync(kFull, (unsigned)ms);
    for (int o = 16; o > 0; o >>= 1) chk += __shfl_xor_sync(kFull, chk, o);
    if (lane == 0) {
      const bool ok = verdict == SYNC_PROG_OK;
      a.makespan[p] = ok ? ms : -1;
      a.checksum[p] = ok ? chk : 0ull;
      a.status[p] = verdict;
      // fused check: the pairs of programs that ran to the end
      if (FUSED && ok && a.chk_counts) {
        if (S.tally[0]) atomicAdd(a.chk_counts + 0, S.tally[0]);
        if (S.tally[1]) atomicAdd(a.chk_counts + 1, S.tally[1]);
        if (S.tally[2] != ~0ull) atomicMin(a.chk_first, S.tally[2]);
      }
    }
    __syncwarp();
  }
}

}  // namespace
}  // namespace syncgb
