// Per-program construction of the device encoding: validation, Sec. 5.2's
// classification of every dependency, N and K (Sec. 5.5), the iteration
// spaces with their trip prefix sums, the dependency table and path pool of
// the threshold and check kernels (Eq. (1)-(3), (5)), and the simulators'
// records (op rows, sweep plan, chunks and lanes, semaphore numbering,
// Sec. 6.2's per-instruction reduction counts).
//
// One routine, run per program in two passes: COUNT validates the program
// and counts the entries it appends to each appended table; FILL (run only
// when no program failed) writes every table at the program's offsets, the
// exclusive prefix sums of the counts over the programs.  The loader runs
// both passes on host threads (sync_validate_programs runs COUNT alone).
// Every table a program owns is indexed by global ids (its loops,
// instructions, dependencies and (loop, engine) rows) or starts at its
// offsets, so programs never write each other's entries: any assignment of
// programs to threads writes the same bytes.  The routine is also valid
// device code (one thread per program); on the GPU its passes measured
// 6.8 + 12.8 ms for the 65536-program chain batch, GPU time that a stream
// of loads beside running simulations adds to every step, so the loader
// keeps them on the host cores.
#pragma once

#include "enc.h"

#ifdef __CUDACC__
#define PB_HD __host__ __device__ __forceinline__
#else
#define PB_HD inline
#endif

namespace syncgb {

constexpr int64_t kI32Max = 2147483647;
PB_HD int64_t pad4(int64_t n) { return (n + 3) & ~int64_t(3); }

// Code-size proxy: wait-value ops of a per-loop wait (Table 1) and control
// ops of a loop on one engine (r-hat := 0, branch, r++, r-hat++).
constexpr int64_t kCodeWaitOps = 5;
constexpr int64_t kCodeLoopOps = 4;

// Appended tables: entries each program appends, counted by COUNT.
enum : int32_t {
  BC_ROWPTR = 0,   // trip prefix sums (n_parent + 1 per iteration space)
  BC_ITERS,        // global loop iterations
  BC_INST,         // datapath instances
  BC_PAIRS,        // (dependency, consumer instance) pairs
  BC_PADDED,       // pairs with every dependency's segment padded to 4
  BC_DERIVED,      // derived trip-start and ancestor entries
  BC_PATH,         // path pool entries
  BC_ORD,          // ordinal pool entries (per-engine mode)
  BC_HIST,         // semaphore history slots, one count per mode
  BC_OPS = BC_HIST + kModes,  // op records (and op stops)
  BC_PLAN,         // sweep plan items (and loop-statement side records)
  BC_CHUNKS,       // sweep chunks
  BC_LANES,        // sweep lanes
  BC_SEMHB,        // semaphore history bases
  BC_JOBS,         // derive jobs
  BC_DROWS,        // rows of the derive jobs
  kBuildCounts
};

// Validation failures, in the order a program is checked; the loader
// reports the first failure of the first failing program.
enum : int32_t {
  BE_NONE = 0, BE_NO_TOP, BE_ENGINES, BE_ROOT, BE_PARENT, BE_LOOP_POS, BE_DEPTH,
  BE_TRIP_NEG, BE_TOP_TRIP, BE_ITERS, BE_TRIP_LEN, BE_ENG_TRIP_LEN, BE_ENG_TRIPS_NULL,
  BE_X_LOOP, BE_X_POS, BE_X_ENGINE, BE_X_LATENCY, BE_DUP_POS, BE_D_RANGE, BE_D_OFFSET,
  BE_BWD0, BE_FWD_K, BE_BWD_K, BE_FB_DIV, BE_N_OVERFLOW, kBuildErrors
};

// The caller's batch (sync_batch_desc), on the side that runs the pass.
struct RawBatch {
  const int32_t *prog_loop_ptr, *prog_instr_ptr, *prog_dep_ptr, *prog_n_engines;
  const int32_t *loop_parent, *loop_pos;
  const int32_t *instr_loop, *instr_pos, *instr_engine, *instr_latency;
  const int32_t *dep_prod, *dep_cons, *dep_k;
  const int64_t* trip_ptr;
  const int32_t* trips;
  const int64_t* eng_trip_ptr;
  const int32_t* eng_trips;
  const int64_t* row_base;   // [P + 1]: first (loop, engine) row of each program
  int32_t P;                 // programs the pass covers
  int32_t div;               // per-engine trip counts
  int32_t fallback;          // SYNC_NONALLOC_BARRIER
  int64_t NX, ND;
};

// A wait of the current straight-line segment (Sec. 6.2's CSE).
struct Seen {
  int32_t e, px, k, S, Pl, Pe;
};

// Scratch, indexed by global ids: per loop [NL], per instruction [NX], per
// dependency [ND], per (loop, engine) row [rows]; body items of program p
// at x0 + l0 (nx + nl - 1 of them), body offsets at l0 + p (nl + 1).
struct BuildScratch {
  int32_t *depth, *lfill;                    // [NL]
  uint8_t *needs_rhat, *fbar;                // [NL]
  int32_t* body_ptr;                         // [NL + P]
  int64_t* keys;                             // [NX + NL]
  int32_t* body;                             // [NX + NL]
  int32_t *rank, *x_ndeps, *x_dep_begin, *x_levels, *cons_next, *sem_x;   // [NX]
  int32_t *nloop_eng, *sem_row;              // [rows]
  int64_t *stot, *srp, *tstart;              // [rows] per iteration space
  uint32_t* pe_of;                           // [rows]
  uint8_t* rpflag;                           // [rows]
  int32_t* anc;                              // [rows * SYNC_MAX_DEPTH]
  uint8_t* dep_bar;                          // [ND]
  int32_t *dep_S, *dep_N, *by_cons;          // [ND]
  Seen* seen;                                // [ND]
};

// The encoding (enc.h) the pass writes; FILL writes all of it, COUNT only
// ord_off (its dedup marks).
struct BuildOut {
  LoopInfo* loop;          // [NL]
  DepInfo* dep;            // [ND]
  ProgInfo* prog;          // [P]
  int64_t* inst_off;       // [NX]
  int64_t* ord_off;        // [NX]: ordinal pool offset of a waited producer, or -1
  int4* xsem;              // [kModes][NX]
  int4* xcse;              // [NX]
  int32_t* xlvr;           // [NX]
  int64_t* seg;            // [ND + 1]
  int32_t* dep_count;      // [ND]
  int64_t* dseg;           // [ND]
  int32_t* ddep;           // [ND]
  int32_t* dsem;           // [kModes][ND]
  int32_t* lflag;          // [NL]
  int32_t* plan_ptr;       // [NL + 1]
  int32_t* op_ptr;         // [rows + 1]
  int2* rowinfo;           // [rows]
  int32_t* hoist;          // [rows]
  LoopInfo* xloops;        // [NL] (shared trips) or [rows] (per-engine trips)
  uint8_t* reads_rowptr;   // like xloops
  int32_t* rowptr;         // appended from here on
  int64_t* path;
  DeriveJob* jobs;
  int4 *ops, *plan, *paux, *chunks, *lrec, *lmeta;
  int32_t* opstop;
  int64_t* semhb;
};

// What COUNT reports per program besides the counts.
struct alignas(16) ProgSummary {
  int64_t work;            // simulated work (the simulators' program order)
  int64_t n_inst;
  int64_t code_looped, code_unrolled;   // static instructions (code-size proxy)
  int64_t n_bar_deps;      // barrier-fallback dependencies
  int64_t struct_bytes;    // path entries and rowptr spaces the threshold kernels read
  int64_t err_index;
  int32_t nsem[kModes];
  int32_t ne, depth_max, ord_overflow, err, splittable;
};

struct BuildArgs {
  RawBatch d;
  BuildScratch s;
  BuildOut o;
  const int64_t* base;     // FILL: [P][kBuildCounts] exclusive prefix sums
  int64_t* count;          // COUNT: [P][kBuildCounts]
  ProgSummary* sum;        // COUNT: [P]
};

PB_HD int32_t pb_popc(uint32_t v) {
#ifdef __CUDA_ARCH__
  return __popc(v);
#else
  return __builtin_popcount(v);
#endif
}
PB_HD int64_t pb_max(int64_t a, int64_t b) { return a > b ? a : b; }
PB_HD int64_t pb_min(int64_t a, int64_t b) { return a < b ? a : b; }

// Ascending sort of n keys: insertion sort for short bodies, heap sort
// (O(n log n), in place) for long ones.
PB_HD void pb_sort(int64_t* a, int64_t n) {
  if (n <= 32) {
    for (int64_t i = 1; i < n; ++i) {
      const int64_t v = a[i];
      int64_t j = i;
      for (; j > 0 && a[j - 1] > v; --j) a[j] = a[j - 1];
      a[j] = v;
    }
    return;
  }
  auto sift = [a](int64_t root, int64_t end) {
    while (2 * root + 1 < end) {
      int64_t c = 2 * root + 1;
      if (c + 1 < end && a[c] < a[c + 1]) ++c;
      if (a[root] >= a[c]) return;
      const int64_t t = a[root];
      a[root] = a[c];
      a[c] = t;
      root = c;
    }
  };
  for (int64_t i = n / 2; i-- > 0;) sift(i, n);
  for (int64_t end = n - 1; end > 0; --end) {
    const int64_t t = a[0];
    a[0] = a[end];
    a[end] = t;
    sift(0, end);
  }
}

template <bool FILL>
struct ProgBuilder {
  const BuildArgs& A;
  const RawBatch& d;
  const BuildScratch& S;
  const BuildOut& O;
  int32_t p, l0, x0, d0, nl, nx, nd, ne;
  int64_t row0, xbase;
  const int32_t *par, *lpos;
  int64_t c[kBuildCounts];
  int64_t inst_eng[32];      // instances per engine
  ProgInfo pi;
  ProgSummary sm;

  PB_HD ProgBuilder(const BuildArgs& a, int32_t prog) : A(a), d(a.d), S(a.s), O(a.o), p(prog) {
    l0 = d.prog_loop_ptr[p];
    x0 = d.prog_instr_ptr[p];
    d0 = d.prog_dep_ptr[p];
    nl = d.prog_loop_ptr[p + 1] - l0;
    nx = d.prog_instr_ptr[p + 1] - x0;
    nd = d.prog_dep_ptr[p + 1] - d0;
    ne = d.prog_n_engines[p];
    row0 = d.row_base[p];
    xbase = d.div ? row0 : l0;
    par = d.loop_parent + l0;
    lpos = d.loop_pos + l0;
    for (int i = 0; i < kBuildCounts; ++i) c[i] = FILL ? A.base[(int64_t)p * kBuildCounts + i] : 0;
    pi = ProgInfo{};
    sm = ProgSummary{};
  }

  PB_HD bool fail(int32_t kind, int64_t idx) {
    sm.err = kind;
    sm.err_index = idx;
    return false;
  }
  PB_HD int32_t IL(int32_t x) const { return d.instr_loop[x0 + x]; }
  PB_HD int32_t IE(int32_t x) const { return d.instr_engine[x0 + x]; }
  // row of iteration space (l, e): per (loop, engine) with per-engine trips,
  // the loop's engine-0 row otherwise
  PB_HD int64_t sr(int32_t l, int32_t e) const { return row0 + (int64_t)l * ne + (d.div ? e : 0); }
  PB_HD int64_t tot(int32_t l, int32_t e) const { return S.stot[sr(l, e)]; }
  PB_HD int32_t xid(int32_t l, int32_t e) const { return d.div ? l * ne + e : l; }
  PB_HD int32_t depth(int32_t l) const { return S.depth[l0 + l]; }

  // ------------------------------------------------------------ loops
  // FILL runs after COUNT has passed every program: the scratch COUNT left
  // for this program (depths, sorted bodies, ranks, consumer grouping) is
  // still in place, indexed by the program's own ids, so FILL skips the
  // stages that only rebuild it
  PB_HD bool loops() {
    for (int32_t x = 0; x < nx; ++x) O.ord_off[x0 + x] = -1;
    if (FILL) return true;
    if (nl < 1) return fail(BE_NO_TOP, 0);
    if (ne < 1 || ne > 32) return fail(BE_ENGINES, ne);
    if (par[0] != -1) return fail(BE_ROOT, 0);
    int32_t* dep = S.depth + l0;
    dep[0] = 0;
    for (int32_t l = 1; l < nl; ++l) {
      if (par[l] < 0 || par[l] >= l) return fail(BE_PARENT, l);
      if (lpos[l] < 0) return fail(BE_LOOP_POS, l);
      dep[l] = dep[par[l]] + 1;
      if (dep[l] > SYNC_MAX_DEPTH) return fail(BE_DEPTH, l);
      if (dep[l] > sm.depth_max) sm.depth_max = dep[l];
    }
    for (int32_t l = 0; l < nl; ++l) {
      S.needs_rhat[l0 + l] = 0;
      S.fbar[l0 + l] = 0;
    }
    return true;
  }

  // one iteration space: its trips (want of them, one per parent
  // iteration), total and trip prefix sums
  PB_HD bool add_space(int32_t l, int32_t e, const int32_t* trips, int64_t want) {
    int64_t t = 0;
    for (int64_t j = 0; j < want; ++j) {
      if (trips[j] < 0) return fail(BE_TRIP_NEG, l);
      t += trips[j];
    }
    if (l == 0 && t != 1) return fail(BE_TOP_TRIP, 0);
    if (t > kI32Max) return fail(BE_ITERS, l);
    const int64_t r = row0 + (int64_t)l * ne + e;
    S.stot[r] = t;
    S.srp[r] = c[BC_ROWPTR];
    S.rpflag[r] = 0;
    if (FILL) {
      LoopInfo L{};
      L.parent = l == 0 ? -1 : l0 + par[l];
      L.total = (int32_t)t;
      L.n_parent = (int32_t)want;
      L.depth = depth(l);
      L.rowptr_off = c[BC_ROWPTR];
      const int64_t xi = xbase + xid(l, e);
      O.xloops[xi] = L;
      int32_t* rp = O.rowptr + c[BC_ROWPTR];
      int32_t acc = 0;
      rp[0] = 0;
      for (int64_t j = 0; j < want; ++j) {
        acc += trips[j];
        rp[j + 1] = acc;
      }
      if (e == 0) O.loop[l0 + l] = L;          // engine 0's space stands for the loop
    }
    c[BC_ROWPTR] += want + 1;
    c[BC_ITERS] += t;
    return true;
  }

  PB_HD bool spaces() {
    if (!d.div) {
      for (int32_t l = 0; l < nl; ++l) {
        const int64_t gl = l0 + l;
        const int64_t t0 = d.trip_ptr[gl], t1 = d.trip_ptr[gl + 1];
        const int64_t want = l == 0 ? 1 : tot(par[l], 0);
        if (t1 - t0 != want) return fail(BE_TRIP_LEN, l);
        if (!add_space(l, 0, d.trips + t0, want)) return false;
      }
      return true;
    }
    for (int32_t l = 0; l < nl; ++l)
      for (int32_t e = 0; e < ne; ++e) {
        const int64_t r = row0 + (int64_t)l * ne + e;
        const int64_t t0 = d.eng_trip_ptr[r], t1 = d.eng_trip_ptr[r + 1];
        const int64_t want = l == 0 ? 1 : S.stot[row0 + (int64_t)par[l] * ne + e];
        if (t1 - t0 != want) return fail(BE_ENG_TRIP_LEN, l);
        if (want > 0 && !d.eng_trips) return fail(BE_ENG_TRIPS_NULL, 0);
        if (!add_space(l, e, d.eng_trips + t0, want)) return false;
      }
    return true;
  }

  PB_HD bool instrs() {
    if (FILL) return true;
    for (int32_t x = 0; x < nx; ++x) {
      const int64_t gx = x0 + x;
      if (d.instr_loop[gx] < 0 || d.instr_loop[gx] >= nl) return fail(BE_X_LOOP, x);
      if (d.instr_pos[gx] < 0) return fail(BE_X_POS, x);
      if (d.instr_engine[gx] < 0 || d.instr_engine[gx] >= ne) return fail(BE_X_ENGINE, x);
      if (d.instr_latency[gx] < 1) return fail(BE_X_LATENCY, x);
    }
    return true;
  }

  // bodies in position order (instructions >= 0, child loop l as -(l+1));
  // positions unique within a body
  PB_HD int32_t* bptr() const { return S.body_ptr + l0 + p; }
  PB_HD int32_t* body() const { return S.body + x0 + l0; }
  PB_HD bool bodies() {
    if (FILL) return true;
    int32_t* bp = bptr();
    int64_t* keys = S.keys + x0 + l0;
    int32_t* bd = body();
    for (int32_t l = 0; l <= nl; ++l) bp[l] = 0;
    for (int32_t x = 0; x < nx; ++x) bp[IL(x) + 1]++;
    for (int32_t l = 1; l < nl; ++l) bp[par[l] + 1]++;
    for (int32_t l = 0; l < nl; ++l) bp[l + 1] += bp[l];
    int32_t* fill = S.lfill + l0;
    for (int32_t l = 0; l < nl; ++l) fill[l] = bp[l];
    for (int32_t x = 0; x < nx; ++x)
      keys[fill[IL(x)]++] = ((int64_t)d.instr_pos[x0 + x] << 32) | (uint32_t)x;
    for (int32_t l = 1; l < nl; ++l)
      keys[fill[par[l]]++] = ((int64_t)lpos[l] << 32) | (uint32_t)(-(l + 1));
    for (int32_t l = 0; l < nl; ++l) {
      const int32_t b = bp[l], e = bp[l + 1];
      pb_sort(keys + b, e - b);
      for (int32_t i = b; i < e; ++i) {
        if (i > b && (keys[i] >> 32) == (keys[i - 1] >> 32)) return fail(BE_DUP_POS, l);
        bd[i] = (int32_t)(uint32_t)(keys[i] & 0xffffffffu);
      }
    }
    return true;
  }

  // N (instructions directly in a loop body on one engine) and K (rank)
  PB_HD void ranks() {
    if (FILL) return;
    for (int64_t i = 0; i < (int64_t)nl * ne; ++i) S.nloop_eng[row0 + i] = 0;
    const int32_t* bp = bptr();
    const int32_t* bd = body();
    for (int32_t l = 0; l < nl; ++l)
      for (int32_t i = bp[l]; i < bp[l + 1]; ++i) {
        const int32_t it = bd[i];
        if (it >= 0) S.rank[x0 + it] = ++S.nloop_eng[row0 + (int64_t)l * ne + IE(it)];
      }
  }

  PB_HD void aggregates() {
    pi.ne = ne;
    pi.loop_base = l0;
    pi.le_base = (int32_t)row0;
    int64_t agg = 0;                           // saturating: every term >= 0
    for (int32_t e = 0; e < ne; ++e) inst_eng[e] = 0;
    for (int32_t x = 0; x < nx; ++x) {
      const int64_t n = tot(IL(x), IE(x));
      const int64_t term = n * d.instr_latency[x0 + x];
      agg = agg > INT64_MAX - term ? INT64_MAX : agg + term;
      if (FILL) O.inst_off[x0 + x] = c[BC_INST];
      c[BC_INST] += n;
      pi.n_inst += n;
      inst_eng[IE(x)] += n;
    }
    pi.agg_lat = agg;
    for (int32_t e = 0; e < ne; ++e)
      if (inst_eng[e] > kI32Max) sm.ord_overflow = 1;
    for (int32_t e = 0; e < ne; ++e) {
      int64_t st = 0, it = 0;
      for (int32_t l = 1; l < nl; ++l) {
        st += tot(par[l], e);
        it += tot(l, e);
      }
      pi.eng_stmt += st;
      pi.eng_iter += it;
      pi.n_stmt = pb_max(pi.n_stmt, st);
      pi.n_iter = pb_max(pi.n_iter, it);
    }
    pi.divergent = d.div ? 1 : 0;
  }

  // a derive job (enc.h) at the pool's end: nrows rows, n entries, len
  // reserved, and the padding row
  PB_HD void job(int64_t path, int64_t nrows, int64_t n, int64_t len, int32_t kind, int32_t up) {
    if (FILL) {
      DeriveJob J{};
      J.out = c[BC_DERIVED]; J.row0 = c[BC_DROWS]; J.path = path; J.len = len;
      J.nrows = (int32_t)nrows; J.n = (int32_t)n; J.kind = kind; J.up = up;
      O.jobs[c[BC_JOBS]] = J;
    }
    c[BC_JOBS]++;
    c[BC_DROWS] += nrows + 1;
    c[BC_DERIVED] += len;
  }
  // iterations of the parent of iteration space (l, e): the rows of its trips
  PB_HD int64_t n_parent(int32_t l, int32_t e) const { return l == 0 ? 1 : tot(par[l], e); }
  PB_HD void push_path(int64_t v) {
    if (FILL) O.path[c[BC_PATH]] = v;
    c[BC_PATH]++;
  }

  // dependencies: innermost common loop S, the cases of Sec. 5.2, N and K,
  // and everything the threshold kernels read for them
  PB_HD bool deps() {
    for (int64_t i = 0; i < (int64_t)nl * ne; ++i) {
      S.tstart[row0 + i] = -1;
      S.pe_of[row0 + i] = 0;
      for (int32_t u = 0; u < SYNC_MAX_DEPTH; ++u) S.anc[(row0 + i) * SYNC_MAX_DEPTH + u] = -1;
    }
    for (int32_t k = 0; k < nd; ++k) {
      const int64_t gd = d0 + k;
      const int32_t px = d.dep_prod[gd], cx = d.dep_cons[gd], off = d.dep_k[gd];
      if (px < 0 || px >= nx || cx < 0 || cx >= nx) return fail(BE_D_RANGE, k);
      if (off < 0) return fail(BE_D_OFFSET, k);
      const int32_t Pl = IL(px), Cl = IL(cx);
      // climb to the innermost common loop; remember the child of it on each side
      int32_t a = Pl, b = Cl, ca = -1, cb = -1;
      while (depth(a) > depth(b)) { ca = a; a = par[a]; }
      while (depth(b) > depth(a)) { cb = b; b = par[b]; }
      while (a != b) { ca = a; a = par[a]; cb = b; b = par[b]; }
      const int32_t Sl = a;
      S.dep_S[gd] = Sl;
      const int32_t ppos = ca < 0 ? d.instr_pos[x0 + px] : lpos[ca];
      const int32_t cpos = cb < 0 ? d.instr_pos[x0 + cx] : lpos[cb];
      const bool forward = cpos > ppos;
      const bool same_engine = IE(px) == IE(cx);
      int32_t kase;
      if (ca < 0) {
        // producer directly in S: any offset; offset 0 with the consumer not
        // after the producer on the same engine can never issue (in-order)
        if (off == 0 && !forward && same_engine) return fail(BE_BWD0, k);
        kase = CASE_PS;
      } else if (forward) {
        // a larger offset targets an earlier iteration of S: with the
        // fallback, barriers at the ends of S's iterations enforce it
        if (off != 0 && !d.fallback) return fail(BE_FWD_K, k);
        kase = off == 0 ? CASE_NEST_FWD : CASE_BARRIER;
      } else {
        if (off != 1 && (!d.fallback || off == 0)) return fail(BE_BWD_K, k);
        kase = off == 1 ? CASE_NEST_BWD : CASE_BARRIER;
      }
      const int32_t ep = IE(px), ec = IE(cx);
      S.dep_bar[gd] = kase == CASE_BARRIER;
      if (kase == CASE_BARRIER) {
        // no wait value, semaphore, register or derived array: its pairs stay
        // in the threshold layout (wait value 0) and S ends its iterations
        // with all-engine barriers (none at the top level, which runs once);
        // for the threshold and check kernels a producer in S with an offset
        // no trip reaches, over a zero trip-start array (a derive job of
        // length 0 fills its region with zeros), so the masked wait value
        // (Eq. 2) and the required minimum are 0 on every pair
        if (d.div) return fail(BE_FB_DIV, k);
        if (Sl != 0) S.fbar[l0 + Sl] = 1;
        const int64_t n = tot(Cl, ec);
        if (FILL) {
          DepInfo D{};
          D.total = (int32_t)n;
          D.kase = CASE_PS;
          D.k = (int32_t)kI32Max;
          D.tstart = D.src = c[BC_DERIVED];
          D.path = c[BC_PATH];
          D.seg_off = c[BC_PADDED];
          O.dep[gd] = D;
          O.dep_count[gd] = (int32_t)n;
          O.seg[gd] = c[BC_PADDED];
        }
        job(0, 0, 0, pad4(n), DERIVE_TSTART, 0);
        c[BC_PAIRS] += n;
        c[BC_PADDED] += pad4(n);
        S.dep_N[gd] = 0;
        continue;
      }
      if (off > 0) S.needs_rhat[l0 + Sl] = 1;     // r-hat_S's no-wait check matters
      const int32_t N = S.nloop_eng[row0 + (int64_t)Pl * ne + ep];
      const int32_t K = S.rank[x0 + px];
      if ((int64_t)N * tot(Pl, ep) > kI32Max) return fail(BE_N_OVERFLOW, k);
      const int64_t n = tot(Cl, ec);            // consumer instances, on its engine
      DepInfo D{};
      D.total = (int32_t)n;
      D.up = depth(Cl) - depth(Sl);
      D.clen = depth(Pl) - depth(Sl);
      D.kase = kase;
      D.k = off; D.N = N; D.K = K;
      D.path = c[BC_PATH];
      // everything below is read on the consumer engine's iteration spaces
      // (Eq. (1) with that engine's loop-entry counts)
      for (int32_t l = Cl; l != Sl; l = par[l]) push_path(S.srp[sr(l, ec)]);
      for (int32_t l = Pl; l != Sl; l = par[l]) S.rpflag[sr(l, ec)] = 1;
      // derived arrays: trip starts of S, and the S-ancestors of the consumer loop
      const int64_t skey = sr(Sl, ec);
      if (S.tstart[skey] < 0) {
        S.tstart[skey] = c[BC_DERIVED];
        job(S.srp[skey], n_parent(Sl, ec), tot(Sl, ec), pad4(tot(Sl, ec)), DERIVE_TSTART, 1);
      }
      D.tstart = S.tstart[skey];
      if (O.ord_off[x0 + px] < 0) {
        O.ord_off[x0 + px] = c[BC_ORD];
        c[BC_ORD] += tot(Pl, ep);
      }
      D.ordp = O.ord_off[x0 + px];
      D.src = D.tstart;
      if (tot(Sl, ec) == 1) {
        // S runs once: every consumer iteration lies in S-iteration 0, whose
        // trip starts at 0; the kernels take both without reading an array
        D.src = -1;
      } else if (D.up > 0) {
        int32_t& first = S.anc[sr(Cl, ec) * SYNC_MAX_DEPTH + (D.up - 1)];
        if (first < 0) {
          first = k;
          D.src = c[BC_DERIVED];
          job(D.path, tot(Sl, ec), n, pad4(n), DERIVE_ANC, D.up);
        } else {
          D.src = FILL ? O.dep[d0 + first].src : 0;
        }
      }
      // rowptr offsets from S's child down to the producer's loop
      for (int32_t l = Pl, i = D.clen - 1; l != Sl; l = par[l], --i)
        if (FILL) O.path[c[BC_PATH] + i] = S.srp[sr(l, ec)];
      c[BC_PATH] += D.clen;
      sm.struct_bytes += 8 * (int64_t)D.clen;
      D.seg_off = c[BC_PADDED];
      if (FILL) {
        O.dep[gd] = D;
        O.dep_count[gd] = (int32_t)n;
        O.seg[gd] = c[BC_PADDED];
      }
      c[BC_PAIRS] += n;
      c[BC_PADDED] += pad4(n);
      pi.n_pairs += n;
      S.dep_N[gd] = N;
    }
    return true;
  }

  // loops whose trip register can be elided (Sec. 5.1: only offset-0
  // dependencies carried there, or none), their control counts, the
  // fallback barriers, and the code-size proxy (RQ2's code comparison): the
  // looped program holds each datapath instruction once, per waited
  // dependency the per-loop wait-value ops of Table 1 and the wait, per loop
  // and engine its control, and per engine one barrier per loop that ends
  // its iterations with a fallback barrier; the unrolled program holds one
  // instruction per instance and one static wait per waited pair
  PB_HD void control() {
    int64_t waited = 0, fb_loops = 0;
    for (int32_t l = 1; l < nl; ++l)
      if (S.fbar[l0 + l]) {
        pi.fb_iters += tot(l, 0);
        ++fb_loops;
      }
    for (int32_t k = 0; k < nd; ++k) {
      sm.n_bar_deps += S.dep_bar[d0 + k];
      waited += S.dep_bar[d0 + k] ? 0 : 1;
    }
    sm.code_looped = nx + (kCodeWaitOps + 1) * waited + (int64_t)ne * (kCodeLoopOps * (nl - 1) + fb_loops);
    sm.code_unrolled = pi.n_inst + pi.n_pairs;
    if (FILL) O.lflag[l0] = 0;
    for (int32_t l = 1; l < nl; ++l) {
      const bool keep = S.needs_rhat[l0 + l];
      if (FILL) O.lflag[l0 + l] = keep ? 0 : 1;
      if (keep) continue;
      for (int32_t e = 0; e < ne; ++e) {
        pi.el_stmt += tot(par[l], e);
        pi.el_iter += tot(l, e);
      }
    }
  }

  // per-engine waits: loops strictly between the top level and the producer's loop
  PB_HD int32_t levels(int32_t px) const {
    const int32_t v = depth(IL(px)) - 1;
    return v > 0 ? v : 0;
  }

  // waits per consumer (grouped by consumer, stable by dependency id: a
  // counting sort; a consumer's dependencies start at x_dep_begin, d0 if
  // none); returns the number of waited dependencies
  PB_HD int32_t group() {
    if (FILL) {                                    // COUNT's grouping stands; the aggregate only
      int32_t nw = 0;
      for (int32_t k = 0; k < nd; ++k) {
        const int64_t gd = d0 + k;
        if (S.dep_bar[gd]) continue;
        const int32_t cx = d.dep_cons[gd];
        pi.pair_levels += (int64_t)levels(d.dep_prod[gd]) * tot(IL(cx), IE(cx));
        ++nw;
      }
      return nw;
    }
    for (int32_t x = 0; x < nx; ++x) {
      S.x_ndeps[x0 + x] = 0;
      S.x_dep_begin[x0 + x] = d0;
      S.x_levels[x0 + x] = 0;
    }
    for (int32_t k = 0; k < nd; ++k) {
      const int64_t gd = d0 + k;
      if (S.dep_bar[gd]) continue;                 // not waited on
      const int32_t cx = d.dep_cons[gd], lev = levels(d.dep_prod[gd]);
      S.x_levels[x0 + cx] += lev;
      pi.pair_levels += (int64_t)lev * tot(IL(cx), IE(cx));
      S.x_ndeps[x0 + cx]++;
    }
    for (int32_t x = 0, at = 0; x < nx; ++x) {
      if (S.x_ndeps[x0 + x] > 0) S.x_dep_begin[x0 + x] = d0 + at;
      S.cons_next[x0 + x] = at;
      at += S.x_ndeps[x0 + x];
    }
    int32_t nw = 0;
    for (int32_t k = 0; k < nd; ++k)
      if (!S.dep_bar[d0 + k]) {
        S.by_cons[d0 + S.cons_next[x0 + d.dep_cons[d0 + k]]++] = k;
        ++nw;
      }
    return nw;
  }

  // Sec. 6.2's reductions.  CSE: per instruction, the counts its wait ops
  // are made of when the waits of one engine in one visit of a straight-
  // line segment are taken in program order (CostTables in enc.h).  LICM:
  // per (loop, engine), the producer engines whose cached path sums the
  // engine updates at the loop's iteration starts; the bound's terms.
  PB_HD void reductions() {
    if (!FILL) return;                             // nothing COUNT reports depends on them
    const int32_t* bp = bptr();
    const int32_t* bd = body();
    Seen* seen = S.seen + d0;
    for (int32_t l = 0; l < nl; ++l) {
      int32_t ns = 0;
      for (int32_t i = bp[l]; i < bp[l + 1]; ++i) {
        const int32_t x = bd[i];
        if (x < 0) { ns = 0; continue; }          // a child loop ends the segment
        const int32_t ex = IE(x);
        int4 cc = make_int4(0, 0, 0, 0);
        int32_t lvr = 0;
        for (int32_t j = 0; j < S.x_ndeps[x0 + x]; ++j) {
          const int32_t k = S.by_cons[S.x_dep_begin[x0 + x] + j];
          const int64_t gd = d0 + k;
          const int32_t px = d.dep_prod[gd], lev = levels(px);
          const Seen w{ex, px, d.dep_k[gd], S.dep_S[gd], IL(px), IE(px)};
          bool same = false, mask = false, outer = false;
          for (int32_t o = 0; o < ns; ++o) {
            const Seen& v = seen[o];
            if (v.e != ex) continue;
            same = same || (v.px == w.px && v.k == w.k);     // the same value
            mask = mask || (v.S == w.S && v.k == w.k);       // the same isGT(r-hat_S, k)
            outer = outer || (v.Pl == w.Pl && v.Pe == w.Pe); // the same outer path sum
          }
          lvr += lev > 0 ? 1 : 0;
          if (!same) {
            ++cc.x;
            if (mask) ++cc.y;
            if (!outer) { cc.z += lev > 0 ? 1 : 0; cc.w += lev; }
          }
          seen[ns++] = w;
        }
        if (FILL) {
          O.xcse[x0 + x] = cc;
          O.xlvr[x0 + x] = lvr;
        }
      }
    }
    for (int32_t k = 0; k < nd; ++k) {
      const int64_t gd = d0 + k;
      if (S.dep_bar[gd]) continue;
      const int32_t px = d.dep_prod[gd], cx = d.dep_cons[gd];
      const int32_t Pl = IL(px), ec = IE(cx);
      if (depth(Pl) > 1) pi.lv_pairs += tot(IL(cx), ec);
      for (int32_t l = par[Pl]; l > 0; l = par[l]) S.pe_of[row0 + (int64_t)l * ne + ec] |= 1u << IE(px);
    }
  }

  // semaphores that some dependency waits on, per mode, with their history
  // slots: mode 0 = one per producer instruction (one increment per
  // iteration); mode 1 = one per (loop, engine) (N increments per
  // iteration); mode 2 = one per engine (one increment per instance of the
  // engine, numbered by the instance's ordinal)
  PB_HD void semaphores(int32_t nw) {
    int32_t sem_e[32];
    for (int m = 0; m < kModes; ++m) {
      auto sem = [&](int32_t x) -> int32_t& {
        return m == 0 ? S.sem_x[x0 + x] : m == 1 ? S.sem_row[row0 + (int64_t)IL(x) * ne + IE(x)] : sem_e[IE(x)];
      };
      if (m == 0) for (int32_t x = 0; x < nx; ++x) S.sem_x[x0 + x] = -1;
      if (m == 1) for (int64_t i = 0; i < (int64_t)nl * ne; ++i) S.sem_row[row0 + i] = -1;
      if (m == 2) for (int32_t e = 0; e < ne; ++e) sem_e[e] = -1;
      int32_t nsem = 0;
      pi.semhb_off[m] = (int32_t)c[BC_SEMHB];
      for (int32_t k = 0; k < nd; ++k) {
        const int64_t gd = d0 + k;
        if (S.dep_bar[gd]) continue;                // not waited on: no semaphore of its own
        const int32_t px = d.dep_prod[gd];
        int32_t& s = sem(px);
        if (s >= 0) continue;
        s = nsem++;
        if (FILL) O.semhb[c[BC_SEMHB]] = c[BC_HIST + m];
        c[BC_SEMHB]++;
        const int32_t ep = IE(px);
        const int64_t t = tot(IL(px), ep);
        c[BC_HIST + m] += m == 0 ? t : m == 1 ? (int64_t)S.dep_N[gd] * t : inst_eng[ep];
      }
      pi.nsem[m] = nsem;
      sm.nsem[m] = nsem;
    }
    if constexpr (FILL) fill_semaphores(nw, sem_e);
  }

  // the semaphore records of the three modes (instructions, consumer-grouped
  // dependencies): per mode the semaphore and its history stride and offset
  // (one increment per iteration; N per iteration at rank K; one per
  // instance of the engine, numbered by its ordinal)
  PB_HD void fill_semaphores(int32_t nw, const int32_t* sem_e) {
    for (int32_t x = 0; x < nx; ++x) {
      const int32_t e = IE(x);
      const int64_t row = row0 + (int64_t)IL(x) * ne + e;
      const int32_t s0 = S.sem_x[x0 + x], s1 = S.sem_row[row], s2 = sem_e[e];
      O.xsem[x0 + x] = make_int4(s0, s0 >= 0 ? 1 : 0, s0 >= 0 ? 1 : 0, 0);
      O.xsem[d.NX + x0 + x] = make_int4(s1, s1 >= 0 ? S.nloop_eng[row] : 0, s1 >= 0 ? S.rank[x0 + x] : 0, 0);
      O.xsem[2 * d.NX + x0 + x] = make_int4(s2, s2 >= 0 ? -1 : 0, 0, S.x_levels[x0 + x]);
    }
    for (int32_t i = 0; i < nw; ++i) {
      const int64_t gd = d0 + S.by_cons[d0 + i];
      const int32_t px = d.dep_prod[gd], e = IE(px);
      O.dsem[d0 + i] = S.sem_x[x0 + px];
      O.dsem[d.ND + d0 + i] = S.sem_row[row0 + (int64_t)IL(px) * ne + e];
      O.dsem[2 * d.ND + d0 + i] = sem_e[e];
      O.dseg[d0 + i] = O.seg[gd];
      O.ddep[d0 + i] = (int32_t)gd;
    }
    for (int32_t i = nw; i < nd; ++i) {          // slots of barrier-fallback dependencies: unused
      for (int m = 0; m < kModes; ++m) O.dsem[(int64_t)m * d.ND + d0 + i] = -1;
      O.dseg[d0 + i] = 0;
      O.ddep[d0 + i] = d0 + i;
    }
  }

  // per-(loop, engine) op records: own instructions and child loops in body
  // order, then an END record; the next LOOP or END record at or after each
  PB_HD void op_rows() {
    const int32_t* bp = bptr();
    const int32_t* bd = body();
    if constexpr (!FILL) {
      // every instruction on its engine's row, every child loop and an END
      // record on each engine's row
      for (int32_t l = 0; l < nl; ++l) {
        int32_t nloops = 0;
        for (int32_t i = bp[l]; i < bp[l + 1]; ++i) nloops += bd[i] < 0 ? 1 : 0;
        c[BC_OPS] += (bp[l + 1] - bp[l] - nloops) + (int64_t)ne * (nloops + 1);
      }
      return;
    }
    // one pass over each body: an engine's rows follow each other, so each
    // item goes to its engine's write position (a child loop to every
    // engine's); a LOOP or END record closes the instructions before it
    // (their op stop is that record)
    int64_t pos[32], pend[32];
    int32_t cnt[32];
    for (int32_t l = 0; l < nl; ++l) {
      int32_t nloops = 0;
      for (int32_t e = 0; e < ne; ++e) cnt[e] = 0;
      for (int32_t i = bp[l]; i < bp[l + 1]; ++i) {
        const int32_t it = bd[i];
        if (it < 0) ++nloops; else ++cnt[IE(it)];
      }
      int64_t at = c[BC_OPS];
      for (int32_t e = 0; e < ne; ++e) {
        O.op_ptr[row0 + (int64_t)l * ne + e] = (int32_t)at;
        pos[e] = pend[e] = at;
        at += cnt[e] + nloops + 1;
      }
      auto close = [&](int32_t e, int64_t q) {
        for (int64_t r = pend[e]; r <= q; ++r) O.opstop[r] = (int32_t)q;
        pend[e] = q + 1;
      };
      for (int32_t i = bp[l]; i < bp[l + 1]; ++i) {
        const int32_t it = bd[i];
        if (it < 0) {
          const int32_t m = -it - 1;
          for (int32_t e = 0; e < ne; ++e) {
            const int64_t rp = S.srp[sr(m, e)], q = pos[e]++;
            O.ops[q] = make_int4(OP_LOOP, (int32_t)(row0 + (int64_t)m * ne), (int32_t)(uint32_t)(rp & 0xffffffffu),
                                 (int32_t)(rp >> 32));
            close(e, q);
          }
        } else {
          O.ops[pos[IE(it)]++] = make_int4(x0 + it, d.instr_latency[x0 + it], S.x_ndeps[x0 + it],
                                           S.x_dep_begin[x0 + it]);
        }
      }
      const int32_t flags = (nloops > 0 ? 1 : 0) | (O.lflag[l0 + l] ? 2 : 0) | (S.fbar[l0 + l] ? 4 : 0);
      for (int32_t e = 0; e < ne; ++e) {
        const int64_t row = row0 + (int64_t)l * ne + e, q = pos[e];
        O.ops[q] = make_int4(OP_END, 0, 0, 0);
        close(e, q);
        const int32_t nh = pb_popc(S.pe_of[row]);
        pi.licm_upd += (int64_t)nh * tot(l, e);
        O.rowinfo[row] = make_int2((int32_t)q, flags);
        O.hoist[row] = nh;
      }
      c[BC_OPS] = at;
    }
  }

  // one sweep chunk: n <= 32 lanes `recs` (program-local instructions,
  // already engine-major, their engines `engs`) with their iteration copies
  // (nullptr: all copy 0)
  PB_HD void add_chunk(const int32_t* recs, const int32_t* engs, const int32_t* copies, int32_t n,
                       int32_t ncopies) {
    const int64_t base = c[BC_LANES];
    int32_t emask = 0, head = 0;
    for (int32_t i = 0; i < n; ++i) {
      const int32_t x = recs[i], e = engs[i];
      const int32_t cp = copies ? copies[i] : 0;
      if (cp == ncopies - 1) emask |= (int32_t)(1u << e);   // engines in the last copy
      if (i > 0 && engs[i - 1] != e) head = i;         // first lane of the engine's run
      const bool last = i + 1 == n || engs[i + 1] != e;
      const bool first_in_copy = cp > 0 && (i == head || copies[i - 1] != cp);
      if (FILL) {
        O.lrec[c[BC_LANES]] = make_int4(x0 + x, d.instr_latency[x0 + x], S.x_ndeps[x0 + x], S.x_dep_begin[x0 + x]);
        O.lmeta[c[BC_LANES]] =
            make_int4(e, cp, head, (first_in_copy ? LANE_ITER_START : 0) | (last ? LANE_RUN_LAST : 0));
      }
      c[BC_LANES]++;
    }
    if (FILL) O.chunks[c[BC_CHUNKS]] = make_int4((int32_t)base, n, ncopies, emask);
    c[BC_CHUNKS]++;
  }

  PB_HD void add_item(int4 v) {
    if (FILL) O.plan[c[BC_PLAN]] = v;
    c[BC_PLAN]++;
  }

  // program-order sweep plan: per loop, its body cut at child loops into
  // straight-line segments, each segment in chunks of <= 32 engine-sorted lanes
  PB_HD void plan() {
    const int32_t* bp = bptr();
    const int32_t* bd = body();
    for (int32_t l = 0; l < nl; ++l) {
      if (FILL) O.plan_ptr[l0 + l] = (int32_t)c[BC_PLAN];
      int32_t seg0 = bp[l], nseg = 0, nloops = 0;   // current segment: body[seg0 .. i)
      for (int32_t i = bp[l]; i <= bp[l + 1]; ++i) {
        const bool at_end = i == bp[l + 1];
        const int32_t it = at_end ? -1 : bd[i];
        if (!at_end && it >= 0) continue;
        if (i > seg0) {
          ++nseg;
          const int64_t first_chunk = c[BC_CHUNKS];
          for (int32_t b = seg0; b < i; b += 32) {
            // up to 32 records, engine-major and in body order within an
            // engine (a counting sort by engine)
            const int32_t n = (int32_t)pb_min(32, i - b);
            if constexpr (!FILL) {                // COUNT: the chunk's size only
              c[BC_LANES] += n;
              c[BC_CHUNKS]++;
              continue;
            }
            int32_t cnt[33], piece[32], peng[32], eng[32];
            for (int32_t e = 0; e <= ne; ++e) cnt[e] = 0;
            for (int32_t j = 0; j < n; ++j) ++cnt[(eng[j] = IE(bd[b + j])) + 1];
            for (int32_t e = 0; e < ne; ++e) cnt[e + 1] += cnt[e];
            for (int32_t j = 0; j < n; ++j) {
              const int32_t q = cnt[eng[j]]++;
              piece[q] = bd[b + j];
              peng[q] = eng[j];
            }
            add_chunk(piece, peng, nullptr, n, 1);
          }
          add_item(make_int4(ITEM_SEG, (int32_t)first_chunk, (int32_t)(c[BC_CHUNKS] - first_chunk), -1));
        }
        seg0 = i + 1;
        if (!at_end) {
          ++nloops;
          const int32_t m = -it - 1;
          add_item(make_int4(ITEM_LOOP, l0 + m, FILL ? O.lflag[l0 + m] : 0, 0));
        }
      }
      // a short body with no child loop: a template of several iterations
      const int32_t L = bp[l + 1] - bp[l];
      if (nloops == 0 && nseg == 1 && L >= 1 && L <= 16) {
        const int32_t k = 32 / L;
        if constexpr (!FILL) {                    // COUNT: every record in each of k copies
          c[BC_LANES] += (int64_t)k * L;
          c[BC_CHUNKS]++;
          continue;
        }
        int32_t recs[32], engs[32], copies[32], n = 0, be[16];
        for (int32_t i = 0; i < L; ++i) be[i] = IE(bd[bp[l] + i]);
        for (int32_t e = 0; e < ne; ++e)
          for (int32_t cp = 0; cp < k; ++cp)
            for (int32_t i = 0; i < L; ++i)
              if (be[i] == e) { recs[n] = bd[bp[l] + i]; engs[n] = e; copies[n++] = cp; }
        if (FILL) O.plan[c[BC_PLAN] - 1].w = (int32_t)c[BC_CHUNKS];
        add_chunk(recs, engs, copies, n, k);
      }
    }
    // a body that opens with instructions (A) before its first child loop
    // and closes with instructions (B) after its last: one more chunk, B
    // (copy 0) with the next iteration's A (copy 1), for the barrier-free
    // walk of every iteration but a trip's last; the B item, the body's
    // last, names it (w = -2 - chunk).  These chunks follow all the
    // program's others, which the barrier sweep keeps contiguous.
    const int64_t plan_end = c[BC_PLAN];
    for (int32_t l = 1; l < nl; ++l) {
      const int32_t b0 = bp[l], b1 = bp[l + 1];
      int32_t fa = b0;
      while (fa < b1 && bd[fa] >= 0) ++fa;            // the first child loop
      if (fa == b1) continue;                         // none
      int32_t lb = b1;
      while (bd[lb - 1] >= 0) --lb;                   // just past the last one
      const int32_t na = fa - b0, nb = b1 - lb;
      if (na < 1 || nb < 1 || na + nb > 32) continue;
      if constexpr (!FILL) {
        c[BC_LANES] += na + nb;
        c[BC_CHUNKS]++;
        continue;
      }
      // B's records (copy 0), then A's (copy 1), sorted stably by engine
      int32_t rec[32], eng[32], cnt[33], recs[32], engs[32], copies[32];
      int32_t n = 0;
      for (int32_t i = lb; i < b1; ++i) { rec[n] = bd[i]; eng[n++] = IE(bd[i]); }
      for (int32_t i = b0; i < fa; ++i) { rec[n] = bd[i]; eng[n++] = IE(bd[i]); }
      for (int32_t e = 0; e <= ne; ++e) cnt[e] = 0;
      for (int32_t j = 0; j < n; ++j) ++cnt[eng[j] + 1];
      for (int32_t e = 0; e < ne; ++e) cnt[e + 1] += cnt[e];
      for (int32_t j = 0; j < n; ++j) {
        const int32_t q = cnt[eng[j]]++;
        recs[q] = rec[j];
        engs[q] = eng[j];
        copies[q] = j < nb ? 0 : 1;
      }
      const int64_t last_item = (l + 1 < nl ? (int64_t)O.plan_ptr[l0 + l + 1] : plan_end) - 1;
      O.plan[last_item].w = -2 - (int32_t)c[BC_CHUNKS];
      add_chunk(recs, engs, copies, n, 2);
    }
  }

  // per plan item, what the walker reads beside it: for a loop statement
  // the child's rowptr offset and the chunk that holds its whole body
  // (barrier-free: the multi-iteration template if there is one), or -1;
  // for a segment the record of its first chunk
  PB_HD void loop_statements(int64_t plan_first) {
    if constexpr (FILL) {
      for (int64_t i = plan_first; i < c[BC_PLAN]; ++i) {
        const int4 v = O.plan[i];
        if (v.x != ITEM_LOOP) {                   // a segment: its first chunk's record
          O.paux[i] = O.chunks[v.y];
          continue;
        }
        const int32_t m = v.y - l0;
        const int64_t b = O.plan_ptr[l0 + m];
        const int64_t e = m + 1 < nl ? (int64_t)O.plan_ptr[l0 + m + 1] : c[BC_PLAN];
        int32_t bf = -1, bb = -1;
        if (e - b == 1 && O.plan[b].x == ITEM_SEG) {
          if (O.plan[b].z == 1) bf = bb = O.plan[b].y;
          if (O.plan[b].w >= 0) bf = O.plan[b].w;
        }
        const int64_t rp = S.srp[sr(m, 0)];
        O.paux[i] = make_int4((int32_t)(uint32_t)(rp & 0xffffffffu), (int32_t)(rp >> 32), bf, bb);
      }
    }
  }

  // the rowptr spaces the threshold kernels read (nested producers' loops)
  PB_HD void reads() {
    for (int32_t l = 0; l < nl; ++l)
      for (int32_t e = 0; e < (d.div ? ne : 1); ++e) {
        const int64_t r = row0 + (int64_t)l * ne + e;
        if (FILL) O.reads_rowptr[xbase + xid(l, e)] = S.rpflag[r];
        if (S.rpflag[r]) sm.struct_bytes += 4 * ((l == 0 ? 1 : S.stot[sr(par[l], e)]) + 1);
      }
  }

  PB_HD void run() {
    bool ok = loops() && spaces() && instrs() && bodies();
    if (ok) {
      ranks();
      aggregates();
      ok = deps();
    }
    if (ok) {
      control();
      const int32_t nw = group();
      reductions();
      semaphores(nw);
      op_rows();
      const int64_t plan_first = c[BC_PLAN];
      plan();
      loop_statements(plan_first);
      reads();
    }
    if constexpr (FILL) {
      O.prog[p] = pi;
      if (p == d.P - 1) {                        // the closing entries of the offset tables
        O.seg[d.ND] = c[BC_PADDED];
        O.op_ptr[d.row_base[d.P]] = (int32_t)c[BC_OPS];
        O.plan_ptr[d.prog_loop_ptr[d.P]] = (int32_t)c[BC_PLAN];
      }
    } else {
      for (int i = 0; i < kBuildCounts; ++i) A.count[(int64_t)p * kBuildCounts + i] = ok ? c[i] : 0;
      sm.ne = ne;
      sm.n_inst = pi.n_inst;
      sm.work = pi.n_inst + pi.n_pairs + (pi.n_stmt + pi.n_iter) * pi.ne;
      sm.splittable = !d.div && pi.fb_iters == 0;
      A.sum[p] = sm;
    }
  }
};

// Tile tables (k_tiles.cu) of the threshold kernels (segment starts) and
// the derive kernel (job rows).
cudaError_t launch_tile_tables(const int64_t* seg, int64_t n_deps, int32_t* tile_first, int64_t n_first_tiles,
                               const DeriveJob* jobs, int64_t n_jobs, int32_t* tile_job, int64_t n_job_tiles,
                               int num_sms, cudaStream_t s);

}  // namespace syncgb
