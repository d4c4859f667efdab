/*
 * CPU oracle for barrier-free semaphore thresholds (arxiv 2608.13757).
 *
 * TEST INFRASTRUCTURE.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may call this file.  The product path never
 * links it, and it shares no source with the GPU library.
 *
 * Everything is a plain, slow, per-program walk of the loop tree in program
 * order.  What each function follows:
 *
 *  - Program model (Sec. 4.1): structured control flow where every construct
 *    is a loop, conditionals are loops of trip 0 or 1 and the program is a
 *    top-level loop run once; instructions are indexed by iteration vectors of
 *    1-based per-level iteration counts, outermost first.
 *  - orc_thresholds_bruteforce / orc_thresholds: the dependency-satisfaction
 *    condition, Eq. (1) (Sec. 4.2): the target is t = v_cns - delta, where
 *    delta is nonzero only on the innermost common loop S (Sec. 5.1, "carried
 *    at S", offset k); the consumer needs no wait if some t_j <= 0, otherwise
 *    it waits for the number of producer instances whose common-loop
 *    iteration vector is lexicographically <= t.  The brute-force form
 *    compares vectors pairwise; the counting form counts producer instances
 *    per iteration of S and prefix-sums.
 *  - orc_register_replay: the registers of Sec. 5.1 (trip register r-hat,
 *    monotone register r; "entry" read as iteration start) and the masked wait
 *    values of Eq. (2), Eq. (3) and Eq. (5), in natural-number arithmetic as
 *    in the implementation model (Appendix A.5), replayed per engine exactly
 *    as the regOps of Fig. 7 and Fig. 8 place them.
 *  - orc_classify: the allocatable cases of Sec. 5.2 (producer in S with any
 *    offset; producer nested and forward with offset 0; nested and backward
 *    with offset 1), forward/backward by position in S's body (a nested item
 *    counts at the position of the child loop holding it; two instructions of
 *    different engines in the same straight-line region of S count as
 *    forward), and N, K of the per-loop allocation (Sec. 5.5).
 *  - orc_check: the minimality criterion -- a threshold below Eq. (1)'s value
 *    lets the consumer issue early (unsafe), above it over-synchronises
 *    (Sec. 4, consequences in Sec. 7.6).
 *  - orc_simulate: the timing model below, run as an event-stepped machine
 *    over literal semaphores: waits of the form sem >= threshold before issue,
 *    increments at retirement (Sec. 3.3, Appendix A.5), in-order issue and
 *    in-order retirement per engine (Sec. 3.2, Appendix A.2), all counters
 *    and registers starting at zero (Appendix A.6).
 *
 * Timing model.  The paper gives no latencies or costs, so this model is the
 * oracle's own statement; its constants are parameters, and the model is
 * pinned by closed forms and invariants in the tests rather than by numbers
 * printed in the paper.  Integer cycles.  Each engine keeps a cursor t
 * (starting at 0) and walks the common loop tree with the shared trip counts
 * (or its own, with per-engine trips):
 *  - loop statement reached:   barrier-free: t += c_regop (r-hat := 0);
 *                              barrier scheme: an all-engine barrier;
 *  - iteration start:          barrier-free: t += c_branch + 2*c_regop
 *                              (branch, r++, r-hat++); barrier: t += c_branch;
 *    with trip-register elision, a loop at which only offset-0 dependencies
 *    are carried (or none) keeps no r-hat (Sec. 5.1): barrier-free, its
 *    statement costs 0 and each iteration start c_branch + c_regop;
 *  - iteration end:            barrier scheme: an all-engine barrier;
 *                              barrier-free: the same barrier at the end
 *                              of each iteration of a loop that carries a
 *                              barrier-fallback dependency (Sec. 5.2's
 *                              fallback to the barrier scheme, batch
 *                              nonalloc_policy 1), none otherwise;
 *  - datapath instruction x with dependency set D(x) (barrier-fallback
 *    dependencies left out: they are not waited on):
 *      barrier-free: t += sum over D(x) of the wait-value ops (Table 1):
 *        c_wait_ops_count (count), c_wait_ops_perloop (per-loop), or
 *        c_wait_ops_perloop + c_wait_ops_perengine_level * max(0, depth(P)
 *        - 1) (per-engine, Sec. 6.1: one N_l*(r_l - 1) term per loop
 *        strictly between the top level and the producer's loop P);
 *      issue  = max(t, time each waited semaphore reached its threshold);
 *      retire = max(issue + latency, previous retire on this engine);
 *      t = issue + ii;
 *  - barrier: arrival a_e = max(t_e, last retire on e) (drain); release =
 *    max_e a_e + c_barrier (handshake, reset, handshake); every t_e = release;
 *  - the top-level loop has no statement, branch or barrier costs;
 *  - makespan = max over engines of max(t_e, last retire on e).
 *  - unrolled variant (the straight-line program of Sec. 3.3 the loops would
 *    unroll to): as barrier-free with no loop statement, iteration start or
 *    wait-value costs; per-engine semaphores with static waits.
 *  - ALU reductions of Sec. 6.2 (barrier-free; both off by default):
 *    licm (per-engine waits only): the term of every loop l strictly between
 *      the top level and the producer's loop P in the per-engine path sum
 *      changes only when l starts an iteration, so it is kept in a cached
 *      partial sum updated there: at each iteration start of l, engine e pays
 *      c_wait_ops_perengine_level once per producer engine e' such that some
 *      per-engine wait on e (a consumer on e) has its producer on e' and P
 *      strictly below l; such a wait then costs c_wait_ops_perloop plus
 *      c_regop (the read of the cached sum) instead of c_wait_ops_perloop +
 *      c_wait_ops_perengine_level * levels (no read without levels);
 *    cse: on one engine, within one visit of a straight-line segment of a
 *      loop body (the items between two child loops, in one iteration), the
 *      waits are taken in program order (an instruction's dependencies in
 *      dependency order); a wait on the same producer with the same offset as
 *      an earlier one reuses its value and costs 0; otherwise the mask
 *      isGT(r-hat_S, k) of an earlier wait with the same S and k is reused
 *      (min(c_regop, wait-value ops) less), and, per-engine, the outer
 *      partial sum of an earlier wait with the same producer loop and
 *      producer engine (its levels term, or with licm its read) is reused.
 * A semaphore's value reaches v at the retire time of its v-th increment
 * (increments of one semaphore all come from one engine, in retire order;
 * a per-engine semaphore is incremented by every retirement on its engine).
 * Under the barrier scheme the waits stay in place; after a barrier they can
 * only be already satisfied or concern the current barrier interval.
 * The bound counts the wait ops before the reductions of Sec. 6.2; with licm
 * (per-engine, barrier-free) it adds c_wait_ops_perengine_level for every
 * cached-sum update (per iteration of l on e, per producer engine counted
 * above) and c_regop for every pair of a per-engine wait with levels.  CSE
 * only removes costs and changes no bound.
 * Checksum: the sum (mod 2^64) over datapath instances of
 *   (a << 32) | b, with 32-bit arithmetic mod 2^32,
 *   a = (issue ^ (n*0x9E3779B9 + e)) * 0x85EBCA6B, a ^= a >> 13,
 *   b = (retire ^ (n*0xC2B2AE35 + e)) * 0x27D4EB2F, b ^= b >> 15,
 * where e is the engine and n the instance's 1-based ordinal among engine
 * e's datapath instances.  Status: 4 when the static time bound
 *   sum_x inst(x)*(lat(x)+ii+wait ops(x)) + E*(stmts*c_regop + iters*(c_branch+2*c_regop))
 *   + (iterations of loops with fallback barriers)*c_barrier
 * (barrier-free; unrolled: without the control and wait terms), or
 *   sum_x inst(x)*(lat(x)+ii) + E*iters*c_branch + (stmts+iters)*c_barrier
 * (barrier scheme) exceeds INT32_MAX; 7 when no engine can make progress
 * before the end; for both, makespan = -1 and checksum = 0.
 */
#include "oracle.h"

#include <stdlib.h>
#include <string.h>

typedef unsigned __int128 u128;

/* ----------------------------------------------------------- program view */

typedef struct {
  int32_t ne, nl, nx, nd;
  const int32_t *par, *lpos, *xl, *xp, *xe, *xlat, *dp, *dc, *dk;
  const int64_t *tptr;               /* per loop: first trip of the current view */
  const int32_t *trips;
  int32_t maxdepth;
  int32_t *depth;
  int64_t *total;                    /* per loop: iterations in the current view */
  /* per-engine trips: rows (loop, engine) of this program, their totals,
   * and the engine whose trips the view (tptr, trips, total) shows */
  int div, view;
  const int64_t *etptr;
  int64_t *etot, *vtptr;
  int32_t *body_ptr, *body;          /* items by position: x >= 0, or -(loop+1) */
  int32_t *prod_ptr, *prod_dep;      /* dependencies grouped by producer */
  int32_t *cons_ptr, *cons_dep;      /* dependencies grouped by consumer */
  int policy;                        /* the batch's nonalloc_policy */
} prog_t;

static void prog_close(prog_t *P) {
  free(P->etot); free(P->vtptr);
  free(P->depth); free(P->total); free(P->body_ptr); free(P->body);
  free(P->prod_ptr); free(P->prod_dep); free(P->cons_ptr); free(P->cons_dep);
  memset(P, 0, sizeof *P);
}

static int cmp_i64(const void *a, const void *b) {
  int64_t x = *(const int64_t *)a, y = *(const int64_t *)b;
  return x < y ? -1 : x > y;
}

static int group(int32_t n, int32_t m, const int32_t *key, int32_t **ptr, int32_t **idx) {
  *ptr = (int32_t *)calloc((size_t)n + 1, sizeof(int32_t));
  *idx = (int32_t *)malloc(((size_t)m + 1) * sizeof(int32_t));
  if (!*ptr || !*idx) return ORC_ERR_OOM;
  for (int32_t i = 0; i < m; ++i) (*ptr)[key[i] + 1]++;
  for (int32_t i = 0; i < n; ++i) (*ptr)[i + 1] += (*ptr)[i];
  int32_t *fill = (int32_t *)malloc(((size_t)n + 1) * sizeof(int32_t));
  if (!fill) return ORC_ERR_OOM;
  memcpy(fill, *ptr, ((size_t)n + 1) * sizeof(int32_t));
  for (int32_t i = 0; i < m; ++i) (*idx)[fill[key[i]]++] = i;
  free(fill);
  return ORC_OK;
}

/* Per-engine trips: show engine e's trips and totals through tptr, trips
 * and total (no-op for shared trips). */
static void prog_view(prog_t *P, int32_t e) {
  if (!P->div || P->view == e) return;
  for (int32_t l = 0; l < P->nl; ++l) {
    P->vtptr[l] = P->etptr[(int64_t)l * P->ne + e];
    P->total[l] = P->etot[(int64_t)l * P->ne + e];
  }
  P->view = e;
}

/* iterations of loop l on engine e */
static int64_t tot_on(const prog_t *P, int32_t l, int32_t e) {
  return P->div ? P->etot[(int64_t)l * P->ne + e] : P->total[l];
}

/* trip of loop m on engine e during global iteration g of its parent there */
static int32_t trip_on(const prog_t *P, int32_t m, int32_t e, int64_t g) {
  return P->div ? P->trips[P->etptr[(int64_t)m * P->ne + e] + g] : P->trips[P->tptr[m] + g];
}

/* pairs of dependency d: its consumer's instances */
static int64_t cons_total(const prog_t *P, int32_t d) {
  return tot_on(P, P->xl[P->dc[d]], P->xe[P->dc[d]]);
}

/* instances of instruction x */
static int64_t inst_total(const prog_t *P, int32_t x) { return tot_on(P, P->xl[x], P->xe[x]); }

static int prog_open(const orc_batch *b, int32_t p, prog_t *P) {
  memset(P, 0, sizeof *P);
  int32_t l0 = b->prog_loop_ptr[p], x0 = b->prog_instr_ptr[p], d0 = b->prog_dep_ptr[p];
  P->nl = b->prog_loop_ptr[p + 1] - l0;
  P->nx = b->prog_instr_ptr[p + 1] - x0;
  P->nd = b->prog_dep_ptr[p + 1] - d0;
  P->ne = b->prog_n_engines[p];
  P->policy = b->nonalloc_policy;
  if (P->nl < 1 || P->nx < 0 || P->nd < 0 || P->ne < 1 || P->ne > 32) return ORC_ERR_MALFORMED;
  P->par = b->loop_parent + l0; P->lpos = b->loop_pos + l0;
  P->xl = b->instr_loop + x0; P->xp = b->instr_pos + x0;
  P->xe = b->instr_engine + x0; P->xlat = b->instr_latency + x0;
  P->dp = b->dep_prod + d0; P->dc = b->dep_cons + d0; P->dk = b->dep_k + d0;
  P->tptr = b->trip_ptr + l0; P->trips = b->trips;
  int32_t nl = P->nl, nx = P->nx, nd = P->nd;
  P->depth = (int32_t *)calloc((size_t)nl, sizeof(int32_t));
  P->total = (int64_t *)calloc((size_t)nl, sizeof(int64_t));
  if (!P->depth || !P->total) return ORC_ERR_OOM;
  /* the loop tree, parents listed before children */
  if (P->par[0] != -1) return ORC_ERR_MALFORMED;
  for (int32_t l = 1; l < nl; ++l) {
    if (P->par[l] < 0 || P->par[l] >= l || P->lpos[l] < 0) return ORC_ERR_MALFORMED;
    P->depth[l] = P->depth[P->par[l]] + 1;
    if (P->depth[l] > P->maxdepth) P->maxdepth = P->depth[l];
  }
  /* trips: one per iteration of the parent; the top-level loop runs once */
  if (b->eng_trip_ptr) {
    /* per-engine rows: (loop l, engine e) is row rb + l*ne + e */
    int64_t rb = 0;
    for (int32_t q = 0; q < p; ++q)
      rb += (int64_t)(b->prog_loop_ptr[q + 1] - b->prog_loop_ptr[q]) * b->prog_n_engines[q];
    int32_t ne = P->ne;
    P->div = 1;
    P->etptr = b->eng_trip_ptr + rb;
    P->etot = (int64_t *)calloc((size_t)nl * ne, sizeof(int64_t));
    P->vtptr = (int64_t *)calloc((size_t)nl, sizeof(int64_t));
    if (!P->etot || !P->vtptr || !b->eng_trips) return P->etot && P->vtptr ? ORC_ERR_ARG : ORC_ERR_OOM;
    for (int32_t l = 0; l < nl; ++l)
      for (int32_t e = 0; e < ne; ++e) {
        const int64_t *r = P->etptr + (int64_t)l * ne + e;
        int64_t n = r[1] - r[0];
        int64_t want = l == 0 ? 1 : P->etot[(int64_t)P->par[l] * ne + e];
        if (n != want) return ORC_ERR_MALFORMED;
        int64_t s = 0;
        for (int64_t j = 0; j < n; ++j) {
          int32_t t = b->eng_trips[r[0] + j];
          if (t < 0) return ORC_ERR_MALFORMED;
          s += t;
        }
        if (l == 0 && s != 1) return ORC_ERR_MALFORMED;
        P->etot[(int64_t)l * ne + e] = s;
      }
    P->trips = b->eng_trips;
    P->tptr = P->vtptr;
    P->view = -1;
    prog_view(P, 0);
  } else {
    for (int32_t l = 0; l < nl; ++l) {
      int64_t n = P->tptr[l + 1] - P->tptr[l];
      int64_t want = l == 0 ? 1 : P->total[P->par[l]];
      if (n != want) return ORC_ERR_MALFORMED;
      int64_t s = 0;
      for (int64_t j = 0; j < n; ++j) {
        int32_t t = P->trips[P->tptr[l] + j];
        if (t < 0) return ORC_ERR_MALFORMED;
        s += t;
      }
      if (l == 0 && s != 1) return ORC_ERR_MALFORMED;
      P->total[l] = s;
    }
  }
  for (int32_t x = 0; x < nx; ++x) {
    if (P->xl[x] < 0 || P->xl[x] >= nl || P->xp[x] < 0) return ORC_ERR_MALFORMED;
    if (P->xe[x] < 0 || P->xe[x] >= P->ne || P->xlat[x] < 1) return ORC_ERR_MALFORMED;
  }
  for (int32_t d = 0; d < nd; ++d) {
    if (P->dp[d] < 0 || P->dp[d] >= nx || P->dc[d] < 0 || P->dc[d] >= nx || P->dk[d] < 0)
      return ORC_ERR_MALFORMED;
  }
  /* body items sorted by position */
  int32_t nitems = nx + nl - 1;
  int64_t *keys = (int64_t *)malloc(((size_t)nitems + 1) * sizeof(int64_t));
  P->body_ptr = (int32_t *)calloc((size_t)nl + 1, sizeof(int32_t));
  P->body = (int32_t *)malloc(((size_t)nitems + 1) * sizeof(int32_t));
  if (!keys || !P->body_ptr || !P->body) { free(keys); return ORC_ERR_OOM; }
  for (int32_t x = 0; x < nx; ++x) P->body_ptr[P->xl[x] + 1]++;
  for (int32_t l = 1; l < nl; ++l) P->body_ptr[P->par[l] + 1]++;
  for (int32_t l = 0; l < nl; ++l) P->body_ptr[l + 1] += P->body_ptr[l];
  int32_t *fill = (int32_t *)malloc(((size_t)nl + 1) * sizeof(int32_t));
  if (!fill) { free(keys); return ORC_ERR_OOM; }
  memcpy(fill, P->body_ptr, (size_t)nl * sizeof(int32_t));
  /* key: position in the high half, item code in the low half */
  for (int32_t x = 0; x < nx; ++x)
    keys[fill[P->xl[x]]++] = ((int64_t)P->xp[x] << 32) | (uint32_t)x;
  for (int32_t l = 1; l < nl; ++l)
    keys[fill[P->par[l]]++] = ((int64_t)P->lpos[l] << 32) | (uint32_t)(-(l + 1));
  free(fill);
  int rc = ORC_OK;
  for (int32_t l = 0; l < nl && rc == ORC_OK; ++l) {
    int32_t a = P->body_ptr[l], e = P->body_ptr[l + 1];
    qsort(keys + a, (size_t)(e - a), sizeof(int64_t), cmp_i64);
    for (int32_t i = a; i < e; ++i) {
      if (i > a && (keys[i] >> 32) == (keys[i - 1] >> 32)) rc = ORC_ERR_MALFORMED;
      P->body[i] = (int32_t)(uint32_t)(keys[i] & 0xFFFFFFFFu);
    }
  }
  free(keys);
  if (rc) return rc;
  if ((rc = group(nx, nd, P->dp, &P->prod_ptr, &P->prod_dep))) return rc;
  if ((rc = group(nx, nd, P->dc, &P->cons_ptr, &P->cons_dep))) return rc;
  return ORC_OK;
}

/* --------------------------------------------------------------- walking */

typedef struct walker walker;
struct walker {
  prog_t *P;
  int64_t *gl;    /* per level on the current path: global iteration index */
  int64_t *vl;    /* per level on the current path: 1-based index in the trip */
  int64_t *next;  /* per loop: global index of its next iteration */
  void (*visit)(walker *w, int32_t x);
  void *ctx;
};

static void walk_body(walker *w, int32_t l) {
  prog_t *P = w->P;
  for (int32_t i = P->body_ptr[l]; i < P->body_ptr[l + 1]; ++i) {
    int32_t it = P->body[i];
    if (it >= 0) { w->visit(w, it); continue; }
    int32_t m = -it - 1, dm = P->depth[m];
    int32_t trip = P->trips[P->tptr[m] + w->gl[P->depth[l]]];
    for (int32_t q = 1; q <= trip; ++q) {
      w->gl[dm] = w->next[m]++;
      w->vl[dm] = q;
      walk_body(w, m);
    }
  }
}

static int walk(prog_t *P, void (*visit)(walker *, int32_t), void *ctx) {
  walker w;
  w.P = P; w.visit = visit; w.ctx = ctx;
  w.gl = (int64_t *)calloc((size_t)P->maxdepth + 1, sizeof(int64_t));
  w.vl = (int64_t *)calloc((size_t)P->maxdepth + 1, sizeof(int64_t));
  w.next = (int64_t *)calloc((size_t)P->nl, sizeof(int64_t));
  if (!w.gl || !w.vl || !w.next) { free(w.gl); free(w.vl); free(w.next); return ORC_ERR_OOM; }
  w.gl[0] = 0; w.vl[0] = 1; w.next[0] = 1;
  walk_body(&w, 0);
  free(w.gl); free(w.vl); free(w.next);
  return ORC_OK;
}

/* innermost common loop of loops a and b; *ca / *cb receive the child of it
 * on the path down to a / b, or -1 when a / b is that loop itself */
static int32_t common_loop(const prog_t *P, int32_t a, int32_t b, int32_t *ca, int32_t *cb) {
  *ca = -1; *cb = -1;
  while (P->depth[a] > P->depth[b]) { *ca = a; a = P->par[a]; }
  while (P->depth[b] > P->depth[a]) { *cb = b; b = P->par[b]; }
  while (a != b) { *ca = a; a = P->par[a]; *cb = b; b = P->par[b]; }
  return a;
}

typedef struct { int32_t S, P, kase, N, K; } dep_class;

static dep_class classify(const prog_t *P, int32_t d) {
  dep_class c;
  int32_t p = P->dp[d], x = P->dc[d], k = P->dk[d];
  int32_t cp, cx;
  c.S = common_loop(P, P->xl[p], P->xl[x], &cp, &cx);
  c.P = P->xl[p];
  int32_t ppos = cp < 0 ? P->xp[p] : P->lpos[cp];
  int32_t xpos = cx < 0 ? P->xp[x] : P->lpos[cx];
  int forward = xpos > ppos;
  if (cp < 0 && cx < 0 && P->xe[p] != P->xe[x]) {
    /* both directly in S on different engines: same straight-line region
     * unless a child loop of S sits between them */
    int32_t lo = ppos < xpos ? ppos : xpos, hi = ppos < xpos ? xpos : ppos, between = 0;
    for (int32_t i = P->body_ptr[c.S]; i < P->body_ptr[c.S + 1]; ++i) {
      int32_t it = P->body[i];
      if (it < 0 && P->lpos[-it - 1] > lo && P->lpos[-it - 1] < hi) between = 1;
    }
    if (!between) forward = 1;
  }
  if (cp < 0) {
    c.kase = (k == 0 && !forward && P->xe[p] == P->xe[x]) ? ORC_CASE_NONE : ORC_CASE_PS;
  } else if (forward) {
    c.kase = k == 0 ? ORC_CASE_NEST_FWD : P->policy ? ORC_CASE_BARRIER : ORC_CASE_NONE;
  } else {
    c.kase = k == 1 ? ORC_CASE_NEST_BWD : (P->policy && k >= 2) ? ORC_CASE_BARRIER : ORC_CASE_NONE;
  }
  c.N = 0; c.K = 1;
  for (int32_t y = 0; y < P->nx; ++y) {
    if (P->xl[y] != c.P || P->xe[y] != P->xe[p]) continue;
    c.N++;
    if (P->xp[y] < P->xp[p]) c.K++;
  }
  return c;
}

/* per-loop encoding of a completion count (Eq. 4/5); -1 if it leaves int32 */
static int64_t perloop_value(int64_t c, int32_t N, int32_t K) {
  if (c <= 0) return 0;
  int64_t v = (int64_t)N * c - (int64_t)(N - K);
  return v > INT32_MAX ? -1 : v;
}

/* Encodes a completion count c in `mode`; `ord` (per-engine mode only) lists
 * the engine ordinal of each of the producer's instances in program order. */
static int store(int32_t *out, int64_t i, int mode, int64_t c, const dep_class *dc,
                 const int64_t *ord) {
  int64_t v;
  if (mode == ORC_PERLOOP) v = perloop_value(c, dc->N, dc->K);
  else if (mode == ORC_PERENGINE) v = c > 0 ? ord[c - 1] : 0;
  else v = c;
  if (v < 0 || v > INT32_MAX) return ORC_ERR_OVERFLOW;
  out[i] = (int32_t)v;
  return ORC_OK;
}

/* ---------------------------------------------- per-engine stream ordinals */

/* Walk the program in program order, counting each engine's datapath
 * instances: ord[ioff[x] + g] is the 1-based position of instruction x's
 * instance at global iteration g of its loop in the dynamic stream of x's
 * engine (Sec. 6.1: a per-engine counter reaches it when that instance
 * retires, retirement being in order on an engine). */
typedef struct {
  int64_t *ord, *ioff, *count;
} ord_ctx;

static void ord_visit(walker *w, int32_t x) {
  ord_ctx *O = (ord_ctx *)w->ctx;
  prog_t *P = w->P;
  int32_t e = P->xe[x];
  O->ord[O->ioff[x] + w->gl[P->depth[P->xl[x]]]] = ++O->count[e];
}

/* *ord_out / *ioff_out: malloc'd tables (caller frees) */
static int engine_ordinals(prog_t *P, int64_t **ord_out, int64_t **ioff_out) {
  ord_ctx O;
  O.ioff = (int64_t *)malloc(((size_t)P->nx + 1) * sizeof(int64_t));
  O.count = (int64_t *)calloc((size_t)P->ne, sizeof(int64_t));
  if (!O.ioff || !O.count) { free(O.ioff); free(O.count); return ORC_ERR_OOM; }
  int64_t n = 0;
  for (int32_t x = 0; x < P->nx; ++x) { O.ioff[x] = n; n += P->total[P->xl[x]]; }
  O.ioff[P->nx] = n;
  O.ord = (int64_t *)malloc(((size_t)n + 1) * sizeof(int64_t));
  if (!O.ord) { free(O.ioff); free(O.count); return ORC_ERR_OOM; }
  int rc = walk(P, ord_visit, &O);
  free(O.count);
  if (rc) { free(O.ord); free(O.ioff); return rc; }
  *ord_out = O.ord;
  *ioff_out = O.ioff;
  return ORC_OK;
}

/* ------------------------------------------------------------------ sizes */

int orc_sizes(const orc_batch *b, int64_t *n_pairs, int64_t *n_instances) {
  if (!b || b->n_programs < 0) return ORC_ERR_ARG;
  int64_t np = 0, ni = 0;
  for (int32_t p = 0; p < b->n_programs; ++p) {
    prog_t P;
    int rc = prog_open(b, p, &P);
    if (rc) { prog_close(&P); return rc; }
    for (int32_t d = 0; d < P.nd; ++d) np += cons_total(&P, d);
    for (int32_t x = 0; x < P.nx; ++x) ni += inst_total(&P, x);
    prog_close(&P);
  }
  if (n_pairs) *n_pairs = np;
  if (n_instances) *n_instances = ni;
  return ORC_OK;
}

int orc_code_size(const orc_batch *b, int64_t *looped, int64_t *unrolled) {
  if (!b || !looped || !unrolled || b->n_programs < 0) return ORC_ERR_ARG;
  int64_t lp = 0, un = 0;
  for (int32_t p = 0; p < b->n_programs; ++p) {
    prog_t P;
    int rc = prog_open(b, p, &P);
    if (rc) { prog_close(&P); return rc; }
    int8_t *bar_loop = (int8_t *)calloc((size_t)P.nl, 1);
    if (!bar_loop) { prog_close(&P); return ORC_ERR_OOM; }
    lp += P.nx;
    for (int32_t x = 0; x < P.nx; ++x) un += inst_total(&P, x);
    for (int32_t d = 0; d < P.nd; ++d) {
      dep_class c = classify(&P, d);
      if (c.kase == ORC_CASE_BARRIER) {            /* no wait: a barrier ends S's iterations */
        if (c.S != 0) bar_loop[c.S] = 1;
        continue;
      }
      lp += 5 + 1;                                  /* wait-value ops and the wait */
      un += cons_total(&P, d);                      /* one static wait per pair */
    }
    for (int32_t l = 1; l < P.nl; ++l) lp += (int64_t)P.ne * (4 + bar_loop[l]);
    free(bar_loop);
    prog_close(&P);
  }
  *looped = lp;
  *unrolled = un;
  return ORC_OK;
}

int orc_classify(const orc_batch *b, int32_t *S, int32_t *Pl, int32_t *kase, int32_t *N,
                 int32_t *K) {
  if (!b || b->n_programs < 0) return ORC_ERR_ARG;
  for (int32_t p = 0; p < b->n_programs; ++p) {
    prog_t P;
    int rc = prog_open(b, p, &P);
    if (rc) { prog_close(&P); return rc; }
    int32_t d0 = b->prog_dep_ptr[p];
    for (int32_t d = 0; d < P.nd; ++d) {
      dep_class c = classify(&P, d);
      if (S) S[d0 + d] = c.S;
      if (Pl) Pl[d0 + d] = c.P;
      if (kase) kase[d0 + d] = c.kase;
      if (N) N[d0 + d] = c.N;
      if (K) K[d0 + d] = c.K;
    }
    prog_close(&P);
  }
  return ORC_OK;
}

/* --------------------------------------------- Eq. (1), brute-force form */

typedef struct {
  int64_t n, cap, vn, vcap;
  int32_t *x;
  int64_t *g, *voff, *vec;
} inst_list;

static void bf_visit(walker *w, int32_t x) {
  inst_list *L = (inst_list *)w->ctx;
  int32_t dx = w->P->depth[w->P->xl[x]];
  if (L->n == L->cap) {
    L->cap = L->cap ? 2 * L->cap : 256;
    L->x = (int32_t *)realloc(L->x, (size_t)L->cap * sizeof(int32_t));
    L->g = (int64_t *)realloc(L->g, (size_t)L->cap * sizeof(int64_t));
    L->voff = (int64_t *)realloc(L->voff, (size_t)L->cap * sizeof(int64_t));
  }
  while (L->vn + dx + 1 > L->vcap) {
    L->vcap = L->vcap ? 2 * L->vcap : 1024;
    L->vec = (int64_t *)realloc(L->vec, (size_t)L->vcap * sizeof(int64_t));
  }
  L->x[L->n] = x;
  L->g[L->n] = w->gl[dx];
  L->voff[L->n] = L->vn;
  for (int32_t i = 0; i <= dx; ++i) L->vec[L->vn++] = w->vl[i];
  L->n++;
}

/* Eq. (1) by definition for every dependency of the program, in the pair
 * layout of the current view */
static int prog_bruteforce(prog_t *P, int mode, int32_t *out) {
  inst_list L;
  memset(&L, 0, sizeof L);
  int rc = walk(P, bf_visit, &L);
  int64_t *ord = NULL, *ioff = NULL;
  if (rc == ORC_OK && mode == ORC_PERENGINE) rc = engine_ordinals(P, &ord, &ioff);
  int64_t *t = (int64_t *)malloc(((size_t)P->maxdepth + 1) * sizeof(int64_t));
  if (!t && rc == ORC_OK) rc = ORC_ERR_OOM;
  int64_t base = 0;
  for (int32_t d = 0; d < P->nd && rc == ORC_OK; ++d) {
    dep_class dc = classify(P, d);
    int32_t dS = P->depth[dc.S];
    for (int64_t i = 0; i < L.n && rc == ORC_OK; ++i) {
      if (L.x[i] != P->dc[d]) continue;
      /* target t = v restricted to the common loops, minus k on S */
      for (int32_t j = 0; j <= dS; ++j) t[j] = L.vec[L.voff[i] + j];
      t[dS] -= P->dk[d];
      int64_t c = 0;
      if (t[dS] > 0) {
        for (int64_t q = 0; q < L.n; ++q) {
          if (L.x[q] != P->dp[d]) continue;
          int cmp = 0;
          for (int32_t j = 0; j <= dS && cmp == 0; ++j) {
            int64_t a = L.vec[L.voff[q] + j];
            cmp = a < t[j] ? -1 : a > t[j];
          }
          if (cmp <= 0) ++c;
        }
      }
      rc = store(out, base + L.g[i], mode, c, &dc, ord ? ord + ioff[P->dp[d]] : NULL);
    }
    base += P->total[P->xl[P->dc[d]]];
  }
  free(ord); free(ioff);
  free(t); free(L.x); free(L.g); free(L.voff); free(L.vec);
  return rc;
}

/* Per-engine trips: every dependency is evaluated in its consumer engine's
 * view (the loop-entry counts of Eq. (1) are the consumer engine's); f
 * computes all dependencies of one view, and each keeps the segment of the
 * view of its consumer's engine. */
static int per_consumer_view(prog_t *P, int mode, int32_t *out,
                             int (*f)(prog_t *, int, int32_t *)) {
  if (!P->div) return f(P, mode, out);
  if (mode == ORC_PERENGINE) return ORC_ERR_ARG;
  int rc = ORC_OK;
  for (int32_t e = 0; e < P->ne && rc == ORC_OK; ++e) {
    prog_view(P, e);
    int64_t nv = 0;
    for (int32_t d = 0; d < P->nd; ++d) nv += P->total[P->xl[P->dc[d]]];
    int32_t *tmp = (int32_t *)malloc(((size_t)nv + 1) * sizeof(int32_t));
    if (!tmp) return ORC_ERR_OOM;
    rc = f(P, mode, tmp);
    int64_t src = 0, dst = 0;
    for (int32_t d = 0; d < P->nd && rc == ORC_OK; ++d) {
      int64_t n = P->total[P->xl[P->dc[d]]];
      if (P->xe[P->dc[d]] == e) memcpy(out + dst, tmp + src, (size_t)n * sizeof(int32_t));
      src += n;
      dst += cons_total(P, d);
    }
    free(tmp);
  }
  prog_view(P, 0);
  return rc;
}

int orc_thresholds_bruteforce(const orc_batch *b, int mode, int32_t *out) {
  if (!b || !out || (mode != ORC_COUNT && mode != ORC_PERLOOP && mode != ORC_PERENGINE)) return ORC_ERR_ARG;
  int64_t base = 0;
  for (int32_t p = 0; p < b->n_programs; ++p) {
    prog_t P;
    int rc = prog_open(b, p, &P);
    if (rc == ORC_OK) rc = per_consumer_view(&P, mode, out + base, prog_bruteforce);
    for (int32_t d = 0; d < P.nd && rc == ORC_OK; ++d) base += cons_total(&P, d);
    prog_close(&P);
    if (rc) return rc;
  }
  return ORC_OK;
}

/* ------------------------------------------------ Eq. (1), counting form */

typedef struct {
  int32_t *dS;             /* per dep: depth of S */
  int64_t **cnt;           /* per dep: producer instances per global S-iteration */
  int64_t **pg, **pv;      /* per dep, per consumer instance: S-iteration, its index in the trip */
  int64_t *seen;
} cnt_ctx;

static void cnt_visit(walker *w, int32_t x) {
  cnt_ctx *C = (cnt_ctx *)w->ctx;
  prog_t *P = w->P;
  for (int32_t i = P->prod_ptr[x]; i < P->prod_ptr[x + 1]; ++i) {
    int32_t d = P->prod_dep[i];
    C->cnt[d][w->gl[C->dS[d]]]++;
  }
  for (int32_t i = P->cons_ptr[x]; i < P->cons_ptr[x + 1]; ++i) {
    int32_t d = P->cons_dep[i];
    int64_t j = C->seen[d]++;
    C->pg[d][j] = w->gl[C->dS[d]];
    C->pv[d][j] = w->vl[C->dS[d]];
  }
}

/* thresholds of one program, written at out[0 ..) in pair layout */
static int prog_thresholds(prog_t *P, int mode, int32_t *out) {
  int32_t nd = P->nd;
  cnt_ctx C;
  dep_class *cls = (dep_class *)malloc(((size_t)nd + 1) * sizeof(dep_class));
  C.dS = (int32_t *)malloc(((size_t)nd + 1) * sizeof(int32_t));
  C.cnt = (int64_t **)calloc((size_t)nd + 1, sizeof(int64_t *));
  C.pg = (int64_t **)calloc((size_t)nd + 1, sizeof(int64_t *));
  C.pv = (int64_t **)calloc((size_t)nd + 1, sizeof(int64_t *));
  C.seen = (int64_t *)calloc((size_t)nd + 1, sizeof(int64_t));
  int rc = (!cls || !C.dS || !C.cnt || !C.pg || !C.pv || !C.seen) ? ORC_ERR_OOM : ORC_OK;
  for (int32_t d = 0; d < nd && rc == ORC_OK; ++d) {
    cls[d] = classify(P, d);
    C.dS[d] = P->depth[cls[d].S];
    int64_t ncons = P->total[P->xl[P->dc[d]]];
    C.cnt[d] = (int64_t *)calloc((size_t)P->total[cls[d].S] + 1, sizeof(int64_t));
    C.pg[d] = (int64_t *)malloc(((size_t)ncons + 1) * sizeof(int64_t));
    C.pv[d] = (int64_t *)malloc(((size_t)ncons + 1) * sizeof(int64_t));
    if (!C.cnt[d] || !C.pg[d] || !C.pv[d]) rc = ORC_ERR_OOM;
  }
  if (rc == ORC_OK) rc = walk(P, cnt_visit, &C);
  int64_t *ord = NULL, *ioff = NULL;
  if (rc == ORC_OK && mode == ORC_PERENGINE) rc = engine_ordinals(P, &ord, &ioff);
  int64_t base = 0;
  for (int32_t d = 0; d < nd && rc == ORC_OK; ++d) {
    int64_t nS = P->total[cls[d].S];
    for (int64_t g = 1; g < nS; ++g) C.cnt[d][g] += C.cnt[d][g - 1];  /* inclusive sums */
    int64_t ncons = P->total[P->xl[P->dc[d]]];
    for (int64_t j = 0; j < ncons && rc == ORC_OK; ++j) {
      int64_t tS = C.pv[d][j] - P->dk[d];
      /* t lies in the same trip of S as v when tS >= 1, so its global index is
       * the consumer's S-iteration minus k */
      int64_t c = tS <= 0 ? 0 : C.cnt[d][C.pg[d][j] - P->dk[d]];
      rc = store(out, base + j, mode, c, &cls[d], ord ? ord + ioff[P->dp[d]] : NULL);
    }
    base += ncons;
  }
  free(ord); free(ioff);
  for (int32_t d = 0; d < nd; ++d) {
    if (C.cnt) free(C.cnt[d]);
    if (C.pg) free(C.pg[d]);
    if (C.pv) free(C.pv[d]);
  }
  free(cls); free(C.dS); free(C.cnt); free(C.pg); free(C.pv); free(C.seen);
  return rc;
}

int orc_thresholds(const orc_batch *b, int mode, int32_t *out) {
  if (!b || !out || (mode != ORC_COUNT && mode != ORC_PERLOOP && mode != ORC_PERENGINE)) return ORC_ERR_ARG;
  int64_t base = 0;
  for (int32_t p = 0; p < b->n_programs; ++p) {
    prog_t P;
    int rc = prog_open(b, p, &P);
    if (rc == ORC_OK) rc = per_consumer_view(&P, mode, out + base, prog_thresholds);
    for (int32_t d = 0; d < P.nd && rc == ORC_OK; ++d) base += cons_total(&P, d);
    prog_close(&P);
    if (rc) return rc;
  }
  return ORC_OK;
}

/* ------------------------------------------------------ register replay */

typedef struct {
  prog_t *P;
  int32_t e, mode;
  int64_t *r, *rh;        /* monotone and trip registers per loop */
  dep_class *cls;
  int64_t *pair_off;      /* per dep, program-local */
  int32_t *out;
  int rc;
} replay_ctx;

static int64_t nat_sub(int64_t a, int64_t b) { return a > b ? a - b : 0; }

static void replay_body(replay_ctx *R, int32_t l) {
  prog_t *P = R->P;
  for (int32_t i = P->body_ptr[l]; i < P->body_ptr[l + 1]; ++i) {
    int32_t it = P->body[i];
    if (it >= 0) {
      if (P->xe[it] != R->e) continue;
      for (int32_t j = P->cons_ptr[it]; j < P->cons_ptr[it + 1]; ++j) {
        int32_t d = P->cons_dep[j];
        const dep_class *c = &R->cls[d];
        int64_t slot = R->pair_off[d] + (R->r[P->xl[it]] - 1);
        if (c->kase == ORC_CASE_NONE) { R->out[slot] = -1; continue; }
        if (c->kase == ORC_CASE_BARRIER) { R->out[slot] = 0; continue; }   /* no wait emitted */
        int64_t k = P->dk[d];
        int64_t mask = R->rh[c->S] > k ? 1 : 0;                              /* Eq. (2) */
        int64_t expr = c->kase == ORC_CASE_PS ? nat_sub(R->r[c->S], k) : R->r[c->P];
        int64_t w = R->mode == ORC_COUNT
                        ? mask * expr                                            /* Eq. (3) */
                        : mask * nat_sub((int64_t)c->N * expr, c->N - c->K);     /* Eq. (5) */
        if (w > INT32_MAX) { R->rc = ORC_ERR_OVERFLOW; w = -1; }
        R->out[slot] = (int32_t)w;
      }
      continue;
    }
    int32_t m = -it - 1;
    R->rh[m] = 0;                                          /* [r-hat_m := 0] */
    int32_t trip = P->trips[P->tptr[m] + (R->r[l] - 1)];
    for (int32_t q = 0; q < trip; ++q) {
      R->r[m]++;                                           /* [r_m++, r-hat_m++] */
      R->rh[m]++;
      replay_body(R, m);
    }
  }
}

int orc_register_replay(const orc_batch *b, int mode, int32_t *out) {
  if (!b || !out || (mode != ORC_COUNT && mode != ORC_PERLOOP)) return ORC_ERR_ARG;
  int64_t base = 0;
  for (int32_t p = 0; p < b->n_programs; ++p) {
    prog_t P;
    int rc = prog_open(b, p, &P);
    replay_ctx R;
    memset(&R, 0, sizeof R);
    if (rc == ORC_OK) {
      R.P = &P; R.mode = mode; R.out = out;
      R.r = (int64_t *)calloc((size_t)P.nl, sizeof(int64_t));
      R.rh = (int64_t *)calloc((size_t)P.nl, sizeof(int64_t));
      R.cls = (dep_class *)malloc(((size_t)P.nd + 1) * sizeof(dep_class));
      R.pair_off = (int64_t *)malloc(((size_t)P.nd + 1) * sizeof(int64_t));
      if (!R.r || !R.rh || !R.cls || !R.pair_off) rc = ORC_ERR_OOM;
    }
    if (rc == ORC_OK) {
      int64_t off = base;
      for (int32_t d = 0; d < P.nd; ++d) {
        R.cls[d] = classify(&P, d);
        R.pair_off[d] = off;
        off += cons_total(&P, d);
      }
      for (int32_t e = 0; e < P.ne; ++e) {
        prog_view(&P, e);                   /* engine e walks its own trips */
        memset(R.r, 0, (size_t)P.nl * sizeof(int64_t));
        memset(R.rh, 0, (size_t)P.nl * sizeof(int64_t));
        R.e = e;
        R.rh[0] = 0; R.r[0]++; R.rh[0]++;     /* the top-level loop is entered once */
        replay_body(&R, 0);
      }
      rc = R.rc;
      base = off;
    }
    free(R.r); free(R.rh); free(R.cls); free(R.pair_off);
    prog_close(&P);
    if (rc) return rc;
  }
  return ORC_OK;
}

/* ------------------------------------------------------------ the check */

int orc_check(const orc_batch *b, int mode, const int32_t *thr, uint64_t counts[2],
              int64_t *first_bad) {
  if (!b || !thr || !counts || !first_bad ||
      (mode != ORC_COUNT && mode != ORC_PERLOOP && mode != ORC_PERENGINE))
    return ORC_ERR_ARG;
  counts[0] = counts[1] = 0;
  *first_bad = -1;
  int64_t base = 0;
  for (int32_t p = 0; p < b->n_programs; ++p) {
    prog_t P;
    int rc = prog_open(b, p, &P);
    int64_t np = 0;
    for (int32_t d = 0; d < P.nd && rc == ORC_OK; ++d) np += cons_total(&P, d);
    int32_t *want = (int32_t *)malloc(((size_t)np + 1) * sizeof(int32_t));
    if (rc == ORC_OK && !want) rc = ORC_ERR_OOM;
    if (rc == ORC_OK) rc = per_consumer_view(&P, mode, want, prog_thresholds);
    int64_t i = 0;
    for (int32_t d = 0; d < P.nd && rc == ORC_OK; ++d) {
      int64_t n = cons_total(&P, d);
      /* a barrier enforces a barrier-fallback dependency: its minimum is 0 */
      int bar = classify(&P, d).kase == ORC_CASE_BARRIER;
      for (int64_t j = 0; j < n; ++j, ++i) {
        int32_t got = thr[base + i], need = bar ? 0 : want[i];
        if (got == need) continue;
        counts[got < need ? 0 : 1]++;
        if (*first_bad < 0) *first_bad = base + i;
      }
    }
    free(want);
    prog_close(&P);
    if (rc) return rc;
    base += np;
  }
  return ORC_OK;
}

/* ------------------------------------------------------- the timing model */

enum { E_RUN = 0, E_BAR = 1, E_DONE = 2 };
enum { S_PROGRESS = 0, S_BLOCKED = 1, S_BARRIER = 2, S_DONE = 3 };

typedef struct { int32_t loop, item; int64_t g, g_end; } frame;

typedef struct {
  frame *st;
  int32_t sp, state, bar_passed;
  int64_t *next;               /* per loop: global index of its next iteration */
  int64_t t, lastret, arrival, n;
  uint64_t chk;
} engine;

typedef struct {
  prog_t *P;
  const orc_sim_params *prm;
  int mode, barrier;
  int64_t *wcost;              /* per instruction: wait-value ops before issue */
  int64_t *iter_cost;          /* per (loop l, engine e), at l*ne + e: iteration start */
  int64_t *stmt_cost;          /* per loop: loop statement */
  const int32_t *thr;          /* program's pairs */
  int64_t *pair_off;           /* per dep */
  int32_t *own_sem, *dep_sem;  /* semaphore incremented by x / waited by d */
  int64_t *value;              /* per semaphore: increments so far */
  int64_t **times;             /* per waited semaphore: retire time of each increment */
  int32_t *issue, *retire;     /* program's instances, or NULL */
  int64_t *inst_off;           /* per instruction, program-local */
  int8_t *dep_bar;             /* per dep: barrier fallback (no wait) */
  int8_t *loop_bar;            /* per loop: all-engine barrier at the end of each iteration */
} sim_ctx;

static uint64_t inst_term(int64_t issue, int64_t retire, int32_t e, int64_t n) {
  uint32_t a = ((uint32_t)issue ^ ((uint32_t)n * 0x9E3779B9u + (uint32_t)e)) * 0x85EBCA6Bu;
  a ^= a >> 13;
  uint32_t b = ((uint32_t)retire ^ ((uint32_t)n * 0xC2B2AE35u + (uint32_t)e)) * 0x27D4EB2Fu;
  b ^= b >> 15;
  return ((uint64_t)a << 32) | b;
}

static int64_t max64(int64_t a, int64_t b) { return a > b ? a : b; }

static int step(sim_ctx *X, engine *E, int32_t e) {
  prog_t *P = X->P;
  const orc_sim_params *q = X->prm;
  frame *f = &E->st[E->sp - 1];
  int32_t blen = P->body_ptr[f->loop + 1] - P->body_ptr[f->loop];
  if (f->item == blen) {                       /* end of an iteration's body */
    if (f->loop == 0) { E->state = E_DONE; return S_DONE; }
    if ((X->barrier || X->loop_bar[f->loop]) && !E->bar_passed) {
      E->arrival = max64(E->t, E->lastret);
      E->state = E_BAR;
      return S_BARRIER;
    }
    E->bar_passed = 0;
    if (++f->g < f->g_end) {                   /* next iteration starts */
      E->t += X->iter_cost[(int64_t)f->loop * P->ne + e];
      E->next[f->loop]++;
      f->item = 0;
    } else {
      E->sp--;                                 /* loop exit */
    }
    return S_PROGRESS;
  }
  int32_t it = P->body[P->body_ptr[f->loop] + f->item];
  if (it < 0) {                                /* a loop statement */
    if (X->barrier && !E->bar_passed) {
      E->arrival = max64(E->t, E->lastret);
      E->state = E_BAR;
      return S_BARRIER;
    }
    E->bar_passed = 0;
    int32_t m = -it - 1;
    if (!X->barrier) E->t += X->stmt_cost[m];
    int32_t trip = trip_on(P, m, e, f->g);
    f->item++;
    if (trip > 0) {
      frame *c = &E->st[E->sp++];
      c->loop = m; c->item = 0;
      c->g = E->next[m]; c->g_end = c->g + trip;
      E->next[m]++;
      E->t += X->iter_cost[(int64_t)m * P->ne + e];
    }
    return S_PROGRESS;
  }
  if (P->xe[it] != e) { f->item++; return S_PROGRESS; }
  /* datapath instruction `it` in iteration f->g of its loop */
  int64_t tw = E->t + (X->barrier ? 0 : X->wcost[it]);
  int64_t ready = 0;
  for (int32_t j = P->cons_ptr[it]; j < P->cons_ptr[it + 1]; ++j) {
    int32_t d = P->cons_dep[j];
    if (X->dep_bar[d]) continue;               /* enforced by a barrier, not waited on */
    int32_t T = X->thr[X->pair_off[d] + f->g];
    if (T <= 0) continue;
    int32_t s = X->dep_sem[d];
    if (X->value[s] < T) return S_BLOCKED;     /* sem >= T does not hold yet */
    ready = max64(ready, X->times[s][T - 1]);
  }
  int64_t issue = max64(tw, ready);
  int64_t retire = max64(issue + P->xlat[it], E->lastret);
  E->t = issue + q->ii;
  E->lastret = retire;
  int32_t s = X->own_sem[it];
  if (X->times[s]) X->times[s][X->value[s]] = retire;
  X->value[s]++;
  E->n++;
  E->chk += inst_term(issue, retire, e, E->n);
  if (X->issue) {
    X->issue[X->inst_off[it] + f->g] = (int32_t)issue;
    X->retire[X->inst_off[it] + f->g] = (int32_t)retire;
  }
  f->item++;
  return S_PROGRESS;
}

static int sim_program(prog_t *P, int mode, const int32_t *thr, const orc_sim_params *q,
                       int variant, int32_t *makespan, uint64_t *checksum, int32_t *status,
                       int32_t *issue, int32_t *retire) {
  int32_t nl = P->nl, nx = P->nx, nd = P->nd, ne = P->ne;
  int barrier = variant == ORC_BARRIER;
  int unrolled = variant == ORC_UNROLLED;       /* straight-line: no control or wait-value ops */
  /* wait-value ops of each dependency (Table 1; per-engine: O(D), Sec. 6.1) */
  int64_t *wcost = (int64_t *)calloc((size_t)nx + 1, sizeof(int64_t));
  /* the same without the reductions of Sec. 6.2: the static bound's term */
  int64_t *wfull = (int64_t *)calloc((size_t)nx + 1, sizeof(int64_t));
  if (!wfull) { free(wcost); return ORC_ERR_OOM; }
  int8_t *dep_bar = (int8_t *)calloc((size_t)nd + 1, sizeof(int8_t));
  int8_t *loop_bar = (int8_t *)calloc((size_t)nl, sizeof(int8_t));
  if (!wcost || !dep_bar || !loop_bar) { free(wcost); free(wfull); free(dep_bar); free(loop_bar); return ORC_ERR_OOM; }
  /* barrier fallback (Sec. 5.2): no wait; a barrier ends every iteration of
   * the carrying loop S (none at the top level, which runs once) */
  int any_bar = 0;
  for (int32_t d = 0; d < nd; ++d) {
    dep_class c = classify(P, d);
    if (c.kase != ORC_CASE_BARRIER) continue;
    dep_bar[d] = 1;
    any_bar = 1;
    if (c.S != 0) loop_bar[c.S] = 1;
  }
  if (any_bar && unrolled) { free(wcost); free(wfull); free(dep_bar); free(loop_bar); return ORC_ERR_ARG; }
  /* Each loop body is walked in item order; a child loop ends a straight-
   * line segment.  Every waited dependency of a consumer costs its wait-value
   * ops, reduced by the CSE rules (see the header) against the earlier waits
   * of the same engine in the same segment. */
  typedef struct { int32_t e, p, k, S, Pl, pe; } wait_key;
  wait_key *seen = (wait_key *)malloc(((size_t)nd + 1) * sizeof(wait_key));
  if (!seen) { free(wcost); free(wfull); free(dep_bar); free(loop_bar); return ORC_ERR_OOM; }
  const int64_t cw = mode == ORC_COUNT ? q->c_wait_ops_count : q->c_wait_ops_perloop;
  for (int32_t l = 0; l < nl && !unrolled; ++l) {
    int32_t nseen = 0;
    for (int32_t i = P->body_ptr[l]; i < P->body_ptr[l + 1]; ++i) {
      int32_t x = P->body[i];
      if (x < 0) { nseen = 0; continue; }        /* a child loop ends the segment */
      for (int32_t j = P->cons_ptr[x]; j < P->cons_ptr[x + 1]; ++j) {
        int32_t d = P->cons_dep[j];
        if (dep_bar[d]) continue;
        dep_class dc = classify(P, d);
        wait_key w = { P->xe[x], P->dp[d], P->dk[d], dc.S, dc.P, P->xe[P->dp[d]] };
        int32_t lev = mode == ORC_PERENGINE ? P->depth[dc.P] - 1 : 0;
        if (lev < 0) lev = 0;
        /* the outer part of a per-engine wait: its levels, or the cached read */
        int64_t outer = mode != ORC_PERENGINE ? 0
                        : q->licm ? (lev > 0 ? q->c_regop : 0)
                                  : (int64_t)q->c_wait_ops_perengine_level * lev;
        int64_t c = cw + outer;
        wfull[x] += cw + (mode == ORC_PERENGINE ? (int64_t)q->c_wait_ops_perengine_level * lev : 0);
        if (q->cse) {
          int same = 0, mask = 0, part = 0;
          for (int32_t s2 = 0; s2 < nseen; ++s2) {
            if (seen[s2].e != w.e) continue;
            if (seen[s2].p == w.p && seen[s2].k == w.k) same = 1;
            if (seen[s2].S == w.S && seen[s2].k == w.k) mask = 1;
            if (seen[s2].Pl == w.Pl && seen[s2].pe == w.pe) part = 1;
          }
          int64_t m = q->c_regop < cw ? q->c_regop : cw;
          c = same ? 0 : cw - (mask ? m : 0) + (part ? 0 : outer);
          seen[nseen++] = w;
        }
        wcost[x] += c;
      }
    }
  }
  free(seen);
  /* per loop: the register ops of its statement (r-hat := 0) and of each
   * iteration start (branch, r++, r-hat++); with trip-register elision a
   * loop that carries only offset-0 dependencies (or none) has no r-hat
   * (Sec. 5.1), barrier-free */
  int64_t *iter_cost = (int64_t *)calloc((size_t)nl, sizeof(int64_t));
  int64_t *stmt_cost = (int64_t *)calloc((size_t)nl, sizeof(int64_t));
  int8_t *needs_rhat = (int8_t *)calloc((size_t)nl, sizeof(int8_t));
  if (!iter_cost || !stmt_cost || !needs_rhat) {
    free(iter_cost); free(stmt_cost); free(needs_rhat); free(wcost); free(wfull); free(dep_bar); free(loop_bar);
    return ORC_ERR_OOM;
  }
  for (int32_t d = 0; d < nd; ++d)     /* a barrier-fallback dependency reads no register */
    if (P->dk[d] > 0 && !dep_bar[d]) needs_rhat[classify(P, d).S] = 1;
  /* LICM (per-engine, barrier-free): cached path sums kept per (loop l,
   * engine e), one per producer engine e' (bit e' of pe_of[l*ne + e]) */
  uint32_t *pe_of = (uint32_t *)calloc((size_t)nl * ne, sizeof(uint32_t));
  int64_t licm_updates = 0, lv_pairs = 0;        /* for the static bound */
  if (!pe_of) {
    free(iter_cost); free(stmt_cost); free(needs_rhat); free(wcost); free(wfull); free(dep_bar); free(loop_bar);
    return ORC_ERR_OOM;
  }
  int licm = q->licm && mode == ORC_PERENGINE && !barrier && !unrolled;
  for (int32_t d = 0; d < nd && licm; ++d) {
    if (dep_bar[d]) continue;
    int32_t Pl = P->xl[P->dp[d]];
    if (P->depth[Pl] > 1) lv_pairs += cons_total(P, d);
    for (int32_t l = P->par[Pl]; l > 0; l = P->par[l])
      pe_of[(int64_t)l * ne + P->xe[P->dc[d]]] |= 1u << P->xe[P->dp[d]];
  }
  for (int32_t l = 0; l < nl; ++l) {
    int elide = q->trip_register_elision && !needs_rhat[l];
    iter_cost[l] = unrolled ? 0 : barrier ? q->c_branch : q->c_branch + (elide ? 1 : 2) * (int64_t)q->c_regop;
    stmt_cost[l] = unrolled || elide ? 0 : q->c_regop;
  }
  /* per (loop, engine): the iteration start, plus the cached-sum updates */
  int64_t *iter_cost_e = (int64_t *)calloc((size_t)nl * ne + 1, sizeof(int64_t));
  if (!iter_cost_e) {
    free(pe_of); free(iter_cost); free(stmt_cost); free(needs_rhat); free(wcost); free(wfull); free(dep_bar); free(loop_bar);
    return ORC_ERR_OOM;
  }
  for (int32_t l = 0; l < nl; ++l)
    for (int32_t e = 0; e < ne; ++e) {
      int32_t n = __builtin_popcount(pe_of[(int64_t)l * ne + e]);
      iter_cost_e[(int64_t)l * ne + e] = iter_cost[l] + (int64_t)q->c_wait_ops_perengine_level * n;
      licm_updates += (int64_t)n * tot_on(P, l, e);
    }
  free(pe_of);
  free(needs_rhat);
  /* the static time bound */
  u128 bound = 0, ctl = 0;
  int64_t stmts = 0, iters = 0;      /* summed over the engines */
  for (int32_t e = 0; e < ne; ++e)
    for (int32_t l = 1; l < nl; ++l) {
      stmts += tot_on(P, P->par[l], e);
      iters += tot_on(P, l, e);
      ctl += (u128)tot_on(P, P->par[l], e) * (u128)stmt_cost[l] + (u128)tot_on(P, l, e) * (u128)iter_cost[l];
    }
  for (int32_t x = 0; x < nx; ++x) {        /* wait ops before the reductions of Sec. 6.2 */
    int64_t per = (int64_t)P->xlat[x] + q->ii;
    if (!barrier) per += wfull[x];
    bound += (u128)inst_total(P, x) * (u128)per;
  }
  free(wfull);
  wfull = NULL;
  if (barrier) {                     /* shared trips: every engine has the same counts */
    bound += (u128)iters * (u128)q->c_branch;
    bound += (u128)(stmts / ne + iters / ne) * (u128)q->c_barrier;
  } else {
    bound += ctl;
    for (int32_t l = 1; l < nl; ++l)  /* the fallback barriers: one per iteration of a flagged loop */
      if (loop_bar[l]) bound += (u128)P->total[l] * (u128)q->c_barrier;
    if (licm)                         /* cached-sum updates and reads */
      bound += (u128)licm_updates * (u128)q->c_wait_ops_perengine_level + (u128)lv_pairs * (u128)q->c_regop;
  }
  if (bound > (u128)INT32_MAX) {
    free(iter_cost_e);
    free(wcost); free(iter_cost); free(stmt_cost); free(dep_bar); free(loop_bar);
    *makespan = -1; *checksum = 0; *status = ORC_SIM_OVERFLOW;
    return ORC_OK;
  }
  sim_ctx X;
  memset(&X, 0, sizeof X);
  X.P = P; X.prm = q; X.mode = mode; X.barrier = barrier; X.wcost = wcost; X.thr = thr;
  X.iter_cost = iter_cost_e; X.stmt_cost = stmt_cost;
  X.issue = issue; X.retire = retire;
  X.dep_bar = dep_bar; X.loop_bar = loop_bar;
  int32_t nsem = mode == ORC_COUNT ? nx : mode == ORC_PERLOOP ? nl * ne : ne;
  X.pair_off = (int64_t *)malloc(((size_t)nd + 1) * sizeof(int64_t));
  X.inst_off = (int64_t *)malloc(((size_t)nx + 1) * sizeof(int64_t));
  X.own_sem = (int32_t *)malloc(((size_t)nx + 1) * sizeof(int32_t));
  X.dep_sem = (int32_t *)malloc(((size_t)nd + 1) * sizeof(int32_t));
  X.value = (int64_t *)calloc((size_t)nsem + 1, sizeof(int64_t));
  X.times = (int64_t **)calloc((size_t)nsem + 1, sizeof(int64_t *));
  int64_t *incs = (int64_t *)calloc((size_t)nsem + 1, sizeof(int64_t));
  engine *E = (engine *)calloc((size_t)ne, sizeof(engine));
  int rc = (!X.pair_off || !X.inst_off || !X.own_sem || !X.dep_sem || !X.value || !X.times ||
            !incs || !E) ? ORC_ERR_OOM : ORC_OK;
  if (rc == ORC_OK) {
    int64_t off = 0;
    for (int32_t d = 0; d < nd; ++d) { X.pair_off[d] = off; off += cons_total(P, d); }
    off = 0;
    for (int32_t x = 0; x < nx; ++x) {
      X.inst_off[x] = off; off += inst_total(P, x);
      X.own_sem[x] = mode == ORC_COUNT ? x : mode == ORC_PERLOOP ? P->xl[x] * ne + P->xe[x] : P->xe[x];
      incs[X.own_sem[x]] += inst_total(P, x);
    }
    for (int32_t d = 0; d < nd; ++d) {
      int32_t p = P->dp[d];
      X.dep_sem[d] = mode == ORC_COUNT ? p : mode == ORC_PERLOOP ? P->xl[p] * ne + P->xe[p] : P->xe[p];
      int32_t s = X.dep_sem[d];
      if (!dep_bar[d] && !X.times[s]) {
        X.times[s] = (int64_t *)malloc(((size_t)incs[s] + 1) * sizeof(int64_t));
        if (!X.times[s]) rc = ORC_ERR_OOM;
      }
    }
  }
  for (int32_t e = 0; e < ne && rc == ORC_OK; ++e) {
    E[e].st = (frame *)calloc((size_t)P->maxdepth + 1, sizeof(frame));
    E[e].next = (int64_t *)calloc((size_t)nl, sizeof(int64_t));
    if (!E[e].st || !E[e].next) { rc = ORC_ERR_OOM; break; }
    E[e].st[0].loop = 0; E[e].st[0].item = 0; E[e].st[0].g = 0; E[e].st[0].g_end = 1;
    E[e].sp = 1;
    E[e].next[0] = 1;
  }
  int deadlock = 0;
  while (rc == ORC_OK) {
    int progress = 0, ndone = 0, nbar = 0;
    for (int32_t e = 0; e < ne; ++e) {
      if (E[e].state != E_RUN) continue;
      int s;
      while ((s = step(&X, &E[e], e)) == S_PROGRESS) progress = 1;
      if (s == S_BARRIER || s == S_DONE) progress = 1;
    }
    for (int32_t e = 0; e < ne; ++e) {
      ndone += E[e].state == E_DONE;
      nbar += E[e].state == E_BAR;
    }
    if (ndone == ne) break;
    if (nbar == ne) {                           /* every engine drained: release */
      int64_t rel = 0;
      for (int32_t e = 0; e < ne; ++e) rel = max64(rel, E[e].arrival);
      rel += q->c_barrier;
      for (int32_t e = 0; e < ne; ++e) { E[e].t = rel; E[e].state = E_RUN; E[e].bar_passed = 1; }
      progress = 1;
    }
    if (!progress) { deadlock = 1; break; }
  }
  if (rc == ORC_OK) {
    if (deadlock) {
      *makespan = -1; *checksum = 0; *status = ORC_SIM_DEADLOCK;
    } else {
      int64_t ms = 0;
      uint64_t chk = 0;
      for (int32_t e = 0; e < ne; ++e) {
        ms = max64(ms, max64(E[e].t, E[e].lastret));
        chk += E[e].chk;
      }
      *makespan = (int32_t)ms; *checksum = chk; *status = ORC_SIM_OK;
    }
  }
  for (int32_t e = 0; E && e < ne; ++e) { free(E[e].st); free(E[e].next); }
  for (int32_t s = 0; X.times && s < nsem; ++s) free(X.times[s]);
  free(E); free(incs); free(X.pair_off); free(X.inst_off); free(X.own_sem); free(X.dep_sem);
  free(X.value); free(X.times); free(wcost); free(iter_cost); free(stmt_cost);
  free(iter_cost_e); free(dep_bar); free(loop_bar);
  return rc;
}

int orc_simulate(const orc_batch *b, int mode, const int32_t *thr, const orc_sim_params *prm,
                 int variant, int32_t *makespan, uint64_t *checksum, int32_t *status,
                 int32_t *issue, int32_t *retire) {
  if (!b || !thr || !prm || !makespan || !checksum || !status) return ORC_ERR_ARG;
  if ((mode != ORC_COUNT && mode != ORC_PERLOOP && mode != ORC_PERENGINE) ||
      (variant != ORC_BARRIER_FREE && variant != ORC_BARRIER && variant != ORC_UNROLLED) ||
      (variant == ORC_UNROLLED && mode != ORC_PERENGINE) || (!issue) != (!retire))
    return ORC_ERR_ARG;
  int64_t pbase = 0, ibase = 0;
  for (int32_t p = 0; p < b->n_programs; ++p) {
    prog_t P;
    int rc = prog_open(b, p, &P);
    /* per-engine trips: no common barrier sequence, no per-engine positions */
    if (rc == ORC_OK && P.div && (variant != ORC_BARRIER_FREE || mode == ORC_PERENGINE)) rc = ORC_ERR_ARG;
    for (int32_t d = 0; d < P.nd && rc == ORC_OK && P.div; ++d)   /* no common barriers */
      if (classify(&P, d).kase == ORC_CASE_BARRIER) rc = ORC_ERR_ARG;
    if (rc == ORC_OK)
      rc = sim_program(&P, mode, thr + pbase, prm, variant, makespan + p, checksum + p,
                       status + p, issue ? issue + ibase : NULL, retire ? retire + ibase : NULL);
    for (int32_t d = 0; d < P.nd && rc == ORC_OK; ++d) pbase += cons_total(&P, d);
    for (int32_t x = 0; x < P.nx && rc == ORC_OK; ++x) ibase += inst_total(&P, x);
    prog_close(&P);
    if (rc) return rc;
  }
  return ORC_OK;
}
