/*
 * Seeded synthetic batches of structured multi-engine programs.
 *
 * This file is the shared INPUT generator: it builds loop trees, per-engine
 * instruction placements, dependency lists and per-parent-iteration trip
 * counts.  It contains none of the synchronisation method's arithmetic (no
 * thresholds, no iteration-vector decoding, no timing); it only decides the
 * shape of the workload.  Both the CPU oracle and the GPU library consume its
 * output.
 *
 * Program model (the paper's structured control flow, Sec. 4.1): every
 * construct is a loop; a conditional is a loop whose trip is 0 or 1; loop 0 of
 * each program is the top-level loop, which runs once.  A loop body is an
 * ordered list of items (datapath instructions and child loops), ordered by
 * their `pos` value.  Trip counts are given per parent iteration: for loop l,
 * trips[trip_ptr[l] + j] is the trip of l during the j-th (0-based, global)
 * iteration of its parent.  Trip counts are shared by all engines.
 *
 * Random numbers: splitmix64 (Steele, Lea, Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA 2014), one stream per program seeded
 * with seed ^ (program_id * golden gamma); bounded integers by Lemire's
 * multiply-shift reduction of the top 32 bits.
 *
 * Dependency generation keeps every generated dependency inside the paper's
 * allocatable subset (Sec. 5.2) and makes every producer instance a
 * dependency points at precede its consumer in program order, so generated
 * batches never deadlock under either synchronisation scheme.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#include "synth.h"

/* ------------------------------------------------------------------ utils */

typedef struct { int32_t *a; int64_t n, cap; } vi;
typedef struct { int64_t *a; int64_t n, cap; } vl;

static int g_oom = 0;

static void vi_push(vi *v, int32_t x) {
  if (v->n == v->cap) {
    int64_t c = v->cap ? v->cap * 2 : 64;
    int32_t *p = (int32_t *)realloc(v->a, (size_t)c * sizeof *p);
    if (!p) { g_oom = 1; return; }
    v->a = p; v->cap = c;
  }
  v->a[v->n++] = x;
}
static void vl_push(vl *v, int64_t x) {
  if (v->n == v->cap) {
    int64_t c = v->cap ? v->cap * 2 : 64;
    int64_t *p = (int64_t *)realloc(v->a, (size_t)c * sizeof *p);
    if (!p) { g_oom = 1; return; }
    v->a = p; v->cap = c;
  }
  v->a[v->n++] = x;
}
static void vi_free(vi *v) { free(v->a); v->a = NULL; v->n = v->cap = 0; }

typedef struct { uint64_t s; } rng_t;

static uint64_t rng_next(rng_t *r) {
  uint64_t z = (r->s += 0x9E3779B97F4A7C15ULL);
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}
/* uniform integer in [lo, hi] */
static int32_t rng_uni(rng_t *r, int32_t lo, int32_t hi) {
  uint64_t x = rng_next(r) >> 32;
  uint64_t span = (uint64_t)((int64_t)hi - (int64_t)lo + 1);
  return (int32_t)((int64_t)lo + (int64_t)((x * span) >> 32));
}
static rng_t rng_for(uint64_t seed, int64_t pid, uint64_t stream) {
  rng_t r;
  r.s = seed ^ ((uint64_t)pid * 0x9E3779B97F4A7C15ULL) ^ (stream * 0xD1B54A32D192ED03ULL);
  (void)rng_next(&r);
  return r;
}

/* ------------------------------------------------------- program builder */

enum { TRIP_FIXED = 0, TRIP_UNIFORM = 1, TRIP_TRIANGULAR = 2 };

typedef struct {
  int32_t ne;
  vi lpar, lpos, tkind, ta, tb;  /* loops */
  vi xl, xp, xe, xlat;           /* instructions */
  vi dp, dc, dk;                 /* dependencies */
} pbuild;

static void pb_init(pbuild *b, int32_t ne) {
  memset(b, 0, sizeof *b);
  b->ne = ne;
  /* loop 0: the top-level loop, runs once */
  vi_push(&b->lpar, -1); vi_push(&b->lpos, 0);
  vi_push(&b->tkind, TRIP_FIXED); vi_push(&b->ta, 1); vi_push(&b->tb, 1);
}
static void pb_free(pbuild *b) {
  vi_free(&b->lpar); vi_free(&b->lpos); vi_free(&b->tkind); vi_free(&b->ta); vi_free(&b->tb);
  vi_free(&b->xl); vi_free(&b->xp); vi_free(&b->xe); vi_free(&b->xlat);
  vi_free(&b->dp); vi_free(&b->dc); vi_free(&b->dk);
}
static int32_t pb_loop(pbuild *b, int32_t parent, int32_t pos, int32_t kind, int32_t a, int32_t bb) {
  int32_t id = (int32_t)b->lpar.n;
  vi_push(&b->lpar, parent); vi_push(&b->lpos, pos);
  vi_push(&b->tkind, kind); vi_push(&b->ta, a); vi_push(&b->tb, bb);
  return id;
}
static int32_t pb_instr(pbuild *b, int32_t loop, int32_t pos, int32_t eng, int32_t lat) {
  int32_t id = (int32_t)b->xl.n;
  vi_push(&b->xl, loop); vi_push(&b->xp, pos); vi_push(&b->xe, eng); vi_push(&b->xlat, lat);
  return id;
}
static void pb_dep(pbuild *b, int32_t prod, int32_t cons, int32_t k) {
  vi_push(&b->dp, prod); vi_push(&b->dc, cons); vi_push(&b->dk, k);
}

/* ---------------------------------------------------------- batch builder */

typedef struct {
  vi prog_loop_ptr, prog_instr_ptr, prog_dep_ptr, prog_ne;
  vi loop_parent, loop_pos, instr_loop, instr_pos, instr_engine, instr_latency;
  vi dep_prod, dep_cons, dep_k;
  vl trip_ptr; vi trips;
} bbuild;

/* Append one program; draws its trip counts from `tr`. */
static void bb_emit(bbuild *B, pbuild *b, rng_t *tr) {
  int32_t nl = (int32_t)b->lpar.n;
  vi_push(&B->prog_ne, b->ne);
  for (int32_t l = 0; l < nl; ++l) { vi_push(&B->loop_parent, b->lpar.a[l]); vi_push(&B->loop_pos, b->lpos.a[l]); }
  for (int64_t x = 0; x < b->xl.n; ++x) {
    vi_push(&B->instr_loop, b->xl.a[x]); vi_push(&B->instr_pos, b->xp.a[x]);
    vi_push(&B->instr_engine, b->xe.a[x]); vi_push(&B->instr_latency, b->xlat.a[x]);
  }
  for (int64_t d = 0; d < b->dp.n; ++d) {
    vi_push(&B->dep_prod, b->dp.a[d]); vi_push(&B->dep_cons, b->dc.a[d]); vi_push(&B->dep_k, b->dk.a[d]);
  }
  /* Trips, in loop index order (parents precede children).  `wt[l]` holds the
   * 1-based position of each global iteration of l inside its trip; only the
   * triangular rule reads it (a child whose trip equals the parent's index). */
  int64_t *total = (int64_t *)calloc((size_t)nl, sizeof(int64_t));
  vi *wt = (vi *)calloc((size_t)nl, sizeof(vi));
  if (!total || !wt) { g_oom = 1; free(total); free(wt); return; }
  for (int32_t l = 0; l < nl; ++l) {
    vl_push(&B->trip_ptr, B->trips.n);
    int64_t nparent = l == 0 ? 1 : total[b->lpar.a[l]];
    for (int64_t j = 0; j < nparent; ++j) {
      int32_t t;
      switch (b->tkind.a[l]) {
        case TRIP_UNIFORM: t = rng_uni(tr, b->ta.a[l], b->tb.a[l]); break;
        case TRIP_TRIANGULAR: t = wt[b->lpar.a[l]].a[j]; break;
        default: t = b->ta.a[l]; break;
      }
      vi_push(&B->trips, t);
      for (int32_t i = 1; i <= t; ++i) vi_push(&wt[l], i);
      total[l] += t;
    }
  }
  for (int32_t l = 0; l < nl; ++l) vi_free(&wt[l]);
  free(wt); free(total);
  vi_push(&B->prog_loop_ptr, (int32_t)B->loop_parent.n);
  vi_push(&B->prog_instr_ptr, (int32_t)B->instr_loop.n);
  vi_push(&B->prog_dep_ptr, (int32_t)B->dep_prod.n);
}

/* -------------------------------------------------------------- configs */

/* 1 program, 2 engines (PE=0, DMA=1), one loop of trip 16, 6-instruction
 * body, 3 cross-engine deps, one of them loop-carried at distance 1. */
/* An instruction with a drawn engine and then a drawn latency.  Each draw is
 * its own statement: the order of evaluation of a call's arguments is
 * unspecified in C, so two draws in one argument list would give different
 * programs on different compilers or targets. */
static int32_t pb_instr_drawn(pbuild *b, int32_t loop, int32_t pos, rng_t *r, int32_t e_lo, int32_t e_hi,
                              int32_t lat_lo, int32_t lat_hi) {
  const int32_t e = rng_uni(r, e_lo, e_hi);
  const int32_t lat = rng_uni(r, lat_lo, lat_hi);
  return pb_instr(b, loop, pos, e, lat);
}

static void gen_small(pbuild *b, rng_t *r) {
  enum { PE = 0, DMA = 1 };
  pb_init(b, 2);
  int32_t L = pb_loop(b, 0, 0, TRIP_FIXED, 16, 16);
  int32_t ld_a = pb_instr(b, L, 0, DMA, rng_uni(r, 1, 64));
  int32_t ld_b = pb_instr(b, L, 1, DMA, rng_uni(r, 1, 64));
  int32_t mm = pb_instr(b, L, 2, PE, rng_uni(r, 1, 64));
  int32_t mm2 = pb_instr(b, L, 3, PE, rng_uni(r, 1, 64));
  int32_t st = pb_instr(b, L, 4, DMA, rng_uni(r, 1, 64));
  (void)pb_instr(b, L, 5, DMA, rng_uni(r, 1, 64));
  pb_dep(b, ld_b, mm, 0);
  pb_dep(b, mm, st, 0);
  pb_dep(b, mm2, ld_a, 1);
}

/* 4 engines, outer loop A (trip U[1,64]) holding 8 instructions, inner loop
 * B (trip redrawn U[1,64] per A-iteration), 8 more instructions; B holds 16
 * instructions.  8 deps per body, 2 of them loop-carried (distance 1..2). */
static void gen_depth2(pbuild *b, rng_t *r) {
  pb_init(b, 4);
  int32_t A = pb_loop(b, 0, 0, TRIP_UNIFORM, 1, 64);
  int32_t a[16], bx[16];
  for (int i = 0; i < 8; ++i) a[i] = pb_instr_drawn(b, A, i, r, 0, 3, 1, 256);
  int32_t B = pb_loop(b, A, 8, TRIP_UNIFORM, 1, 64);
  for (int i = 8; i < 16; ++i) a[i] = pb_instr_drawn(b, A, i + 1, r, 0, 3, 1, 256);
  for (int i = 0; i < 16; ++i) bx[i] = pb_instr_drawn(b, B, i, r, 0, 3, 1, 256);
  /* B body: 6 same-iteration deps (producer earlier), 2 carried at 1..2 */
  for (int i = 0; i < 6; ++i) {
    int32_t c = rng_uni(r, 1, 15), p = rng_uni(r, 0, c - 1);
    pb_dep(b, bx[p], bx[c], 0);
  }
  for (int i = 0; i < 2; ++i) {
    int32_t c = rng_uni(r, 0, 15), p = rng_uni(r, 0, 15);
    pb_dep(b, bx[p], bx[c], rng_uni(r, 1, 2));
  }
  /* A body: 6 same-iteration deps, either both in A (producer earlier) or
   * producer in B and consumer after B; 2 carried: both in A at 1..2, or
   * producer in B and consumer before B at distance 1. */
  for (int i = 0; i < 6; ++i) {
    if (rng_uni(r, 0, 1)) {
      int32_t c = rng_uni(r, 1, 15), p = rng_uni(r, 0, c - 1);
      pb_dep(b, a[p], a[c], 0);
    } else {
      const int32_t pi = rng_uni(r, 0, 15);
      const int32_t ci = rng_uni(r, 8, 15);
      pb_dep(b, bx[pi], a[ci], 0);
    }
  }
  for (int i = 0; i < 2; ++i) {
    if (rng_uni(r, 0, 1)) {
      const int32_t pi = rng_uni(r, 0, 15);
      const int32_t ci = rng_uni(r, 0, 15);
      const int32_t k = rng_uni(r, 1, 2);
      pb_dep(b, a[pi], a[ci], k);
    } else {
      const int32_t pi = rng_uni(r, 0, 15);
      const int32_t ci = rng_uni(r, 0, 7);
      pb_dep(b, bx[pi], a[ci], 1);
    }
  }
}

/* Tiled 4096^3 GEMM shape: 5 engines, M(32) > N(8) > K(32) with 128x512x128
 * tiles.  K body: 16 A-tile load descriptors + 128 B-row descriptors on DMA-in
 * and 4 matmuls (one per 128-column slab) on PE.  N body after K: 4 ACT, 4
 * vector, 128 DMA-out descriptors.  Double buffering shows up as distance-2
 * dependencies on K (load buffers) and on N (PSUM and output buffers). */
static void gen_gemm(pbuild *b, rng_t *r) {
  enum { DIN = 0, PE = 1, ACT = 2, VEC = 3, DOUT = 4 };
  pb_init(b, 5);
  int32_t M = pb_loop(b, 0, 0, TRIP_FIXED, 32, 32);
  int32_t N = pb_loop(b, M, 0, TRIP_FIXED, 8, 8);
  int32_t K = pb_loop(b, N, 0, TRIP_FIXED, 32, 32);
  int32_t A[16], Bd[128], P[4], C[4], V[4], O[128];
  for (int i = 0; i < 16; ++i) A[i] = pb_instr(b, K, i, DIN, rng_uni(r, 32, 256));
  for (int i = 0; i < 128; ++i) Bd[i] = pb_instr(b, K, 16 + i, DIN, rng_uni(r, 32, 256));
  for (int i = 0; i < 4; ++i) P[i] = pb_instr(b, K, 144 + i, PE, rng_uni(r, 64, 128));
  for (int i = 0; i < 4; ++i) C[i] = pb_instr(b, N, 1 + i, ACT, rng_uni(r, 16, 64));
  for (int i = 0; i < 4; ++i) V[i] = pb_instr(b, N, 5 + i, VEC, rng_uni(r, 16, 64));
  for (int i = 0; i < 128; ++i) O[i] = pb_instr(b, N, 9 + i, DOUT, rng_uni(r, 32, 256));
  for (int j = 0; j < 4; ++j) {
    pb_dep(b, A[15], P[j], 0);            /* A tile loaded before any matmul   */
    pb_dep(b, Bd[32 * j + 31], P[j], 0);  /* slab j of B loaded                */
    pb_dep(b, P[j], Bd[32 * j], 2);       /* WAR on the double-buffered slab   */
    pb_dep(b, P[j], C[j], 0);             /* PSUM of slab j after the K loop   */
    pb_dep(b, C[j], V[j], 0);
    pb_dep(b, V[j], O[32 * j], 0);
    pb_dep(b, O[32 * j + 31], C[j], 2);   /* output staging buffer reuse       */
    pb_dep(b, C[j], P[j], 2);             /* PSUM reuse two N-iterations later */
  }
  pb_dep(b, P[3], A[0], 2);               /* WAR on the double-buffered A tile */
}

/* Causal flash attention, seq 8192, 32 heads, 128-row tiles: 5 engines,
 * head(32) > q-tile(64) > kv-tile with trip = q-tile index (1..64). */
static void gen_attention(pbuild *b, rng_t *r) {
  enum { DIN = 0, PE = 1, ACT = 2, VEC = 3, DOUT = 4 };
  pb_init(b, 5);
  int32_t H = pb_loop(b, 0, 0, TRIP_FIXED, 32, 32);
  int32_t Q = pb_loop(b, H, 0, TRIP_FIXED, 64, 64);
  int32_t ldq = pb_instr(b, Q, 0, DIN, rng_uni(r, 32, 256));
  int32_t KV = pb_loop(b, Q, 1, TRIP_TRIANGULAR, 0, 0);
  int32_t nrm = pb_instr(b, Q, 2, VEC, rng_uni(r, 16, 64));
  int32_t out = pb_instr(b, Q, 3, DOUT, rng_uni(r, 32, 256));
  int32_t ldk = pb_instr(b, KV, 0, DIN, rng_uni(r, 32, 256));
  int32_t ldv = pb_instr(b, KV, 1, DIN, rng_uni(r, 32, 256));
  int32_t qk = pb_instr(b, KV, 2, PE, rng_uni(r, 64, 128));
  int32_t rmax = pb_instr(b, KV, 3, VEC, rng_uni(r, 16, 64));
  int32_t ex = pb_instr(b, KV, 4, ACT, rng_uni(r, 16, 64));
  int32_t rsum = pb_instr(b, KV, 5, VEC, rng_uni(r, 16, 64));
  int32_t resc = pb_instr(b, KV, 6, VEC, rng_uni(r, 16, 64));
  int32_t pv = pb_instr(b, KV, 7, PE, rng_uni(r, 64, 128));
  int32_t acc = pb_instr(b, KV, 8, VEC, rng_uni(r, 16, 64));
  int32_t bka = pb_instr(b, KV, 9, ACT, rng_uni(r, 16, 64));
  int32_t bkp = pb_instr(b, KV, 10, PE, rng_uni(r, 64, 128));
  int32_t bko = pb_instr(b, KV, 11, DOUT, rng_uni(r, 32, 256));
  pb_dep(b, ldk, qk, 0);
  pb_dep(b, qk, rmax, 0);
  pb_dep(b, rmax, ex, 0);
  pb_dep(b, ex, rsum, 0);
  pb_dep(b, rmax, resc, 0);
  pb_dep(b, ex, pv, 0);
  pb_dep(b, ldv, pv, 0);
  pb_dep(b, pv, acc, 0);
  pb_dep(b, resc, acc, 0);
  pb_dep(b, rmax, rmax, 1);   /* running max  */
  pb_dep(b, rsum, rsum, 1);   /* running sum  */
  pb_dep(b, acc, acc, 1);     /* running output accumulator */
  pb_dep(b, qk, ldk, 2);      /* K buffer double buffering */
  pb_dep(b, pv, ldv, 2);      /* V buffer double buffering */
  pb_dep(b, ex, bka, 0);
  pb_dep(b, pv, bkp, 0);
  pb_dep(b, acc, bko, 0);
  pb_dep(b, ldq, qk, 0);      /* Q tile loaded before the kv loop uses it */
  pb_dep(b, acc, nrm, 0);     /* after the kv loop */
  pb_dep(b, rsum, nrm, 0);
  pb_dep(b, nrm, out, 0);
  pb_dep(b, qk, ldq, 1);      /* Q buffer reuse: previous q-tile's kv loop done */
  pb_dep(b, out, nrm, 1);     /* output buffer reuse */
}

/* Random chain programs: engines U{2..5}; U{0..3} nested loops below the
 * top-level loop as a chain (one child per level at a random body position);
 * trips redrawn U[0,32] per parent iteration; U[1,32] instructions per body;
 * each instruction consumes one dependency with probability 0.3, producer
 * uniform over the program's instructions. */
static void gen_chain(pbuild *b, rng_t *r) {
  int32_t ne = rng_uni(r, 2, 5);
  int32_t d = rng_uni(r, 0, 3);
  pb_init(b, ne);
  int32_t lev_loop[4], lev_child_pos[4], nb[4];
  lev_loop[0] = 0;
  for (int i = 0; i <= d; ++i) {
    nb[i] = rng_uni(r, 1, 32);
    lev_child_pos[i] = i < d ? rng_uni(r, 0, nb[i]) : -1;
    if (i < d) lev_loop[i + 1] = pb_loop(b, lev_loop[i], lev_child_pos[i], TRIP_UNIFORM, 0, 32);
  }
  /* instruction j of level i sits at position j, or j+1 past the child */
  int32_t first[5];
  first[0] = 0;
  for (int i = 0; i <= d; ++i) {
    first[i + 1] = first[i] + nb[i];
    for (int j = 0; j < nb[i]; ++j) {
      int32_t pos = (i < d && j >= lev_child_pos[i]) ? j + 1 : j;
      (void)pb_instr_drawn(b, lev_loop[i], pos, r, 0, ne - 1, 1, 256);
    }
  }
  int32_t nx = first[d + 1];
  for (int32_t x = 0; x < nx; ++x) {
    if (rng_uni(r, 0, 999) >= 300) continue;
    int32_t p = rng_uni(r, 0, nx - 1);
    int32_t la = 0, lb = 0;
    while (x >= first[la + 1]) ++la;
    while (p >= first[lb + 1]) ++lb;
    int32_t px = b->xp.a[x], pp = b->xp.a[p];
    int32_t k;
    if (lb <= la) {
      /* producer's loop encloses the consumer: the order in the producer's
       * loop body decides whether the same iteration is still ahead */
      int32_t cons_pos = la == lb ? px : lev_child_pos[lb];
      k = cons_pos > pp ? rng_uni(r, 0, 2) : rng_uni(r, 1, 2);
    } else {
      /* producer nested below the consumer's loop */
      k = px > lev_child_pos[la] ? 0 : 1;
    }
    pb_dep(b, p, x, k);
  }
}

/* Synchronisation-bound chain (AddManyLoop-like): every body is a sequence of
 * single-instruction conditionals (trip-1 loops), engines alternate with the
 * static instruction index; each instruction depends on the previous one, and
 * each chain loop carries one distance-1 dependency from its last conditional
 * to its first. */
static void gen_syncbound(pbuild *b, rng_t *r) {
  int32_t ne = rng_uni(r, 2, 5);
  int32_t d = rng_uni(r, 0, 3);
  pb_init(b, ne);
  int32_t lev_loop[4], nb[4], child_at[4];
  int32_t lev_first_x[4], lev_last_x[4];
  lev_loop[0] = 0;
  for (int i = 0; i <= d; ++i) { nb[i] = rng_uni(r, 1, 2); child_at[i] = i < d ? rng_uni(r, 0, nb[i]) : -1; }
  /* preorder construction: level i body = conds, with the chain child at slot child_at[i] */
  int32_t prev = -1, counter = 0;
  /* iterative preorder over the chain: emit level i conds before the child,
   * descend, then the conds after the child (on the way back up) */
  int32_t before_done[4];
  for (int i = 0; i <= d; ++i) {
    lev_first_x[i] = -1; lev_last_x[i] = -1;
    int32_t upto = i < d ? child_at[i] : nb[i];
    for (int j = 0; j < upto; ++j) {
      int32_t c = pb_loop(b, lev_loop[i], j, TRIP_FIXED, 1, 1);
      int32_t x = pb_instr(b, c, 0, counter++ % ne, rng_uni(r, 1, 256));
      if (prev >= 0) pb_dep(b, prev, x, 0);
      if (lev_first_x[i] < 0) lev_first_x[i] = x;
      lev_last_x[i] = x;
      prev = x;
    }
    before_done[i] = upto;
    if (i < d) lev_loop[i + 1] = pb_loop(b, lev_loop[i], child_at[i], TRIP_UNIFORM, 0, 32);
  }
  for (int i = d - 1; i >= 0; --i) {
    for (int j = before_done[i]; j < nb[i]; ++j) {
      int32_t c = pb_loop(b, lev_loop[i], j + 1, TRIP_FIXED, 1, 1);
      int32_t x = pb_instr(b, c, 0, counter++ % ne, rng_uni(r, 1, 256));
      if (prev >= 0) pb_dep(b, prev, x, 0);
      if (lev_first_x[i] < 0) lev_first_x[i] = x;
      lev_last_x[i] = x;
      prev = x;
    }
  }
  for (int i = 1; i <= d; ++i)
    if (lev_first_x[i] >= 0) pb_dep(b, lev_last_x[i], lev_first_x[i], 1);
}

/* General random loop trees for tests (branching, conditionals, sparse
 * positions, several dependencies per consumer).  With p->any_k set the
 * offsets are drawn freely and may fall outside the allocatable subset. */
static void gen_tree(pbuild *b, rng_t *r, const synth_tree_params *p) {
  int32_t ne = rng_uni(r, p->engines_lo, p->engines_hi);
  pb_init(b, ne);
  int32_t nloops = 1 + rng_uni(r, p->loops_lo, p->loops_hi);
  int32_t *depth = (int32_t *)calloc((size_t)nloops, sizeof(int32_t));
  int32_t *nitems = (int32_t *)calloc((size_t)nloops, sizeof(int32_t));
  int32_t *nbody = (int32_t *)calloc((size_t)nloops, sizeof(int32_t));
  if (!depth || !nitems || !nbody) { g_oom = 1; free(depth); free(nitems); free(nbody); return; }
  /* parents first; position assigned later by a random permutation of items */
  int32_t *par = (int32_t *)calloc((size_t)nloops, sizeof(int32_t));
  par[0] = -1;
  for (int32_t l = 1; l < nloops; ++l) {
    int32_t q, tries = 0;
    do { q = rng_uni(r, 0, l - 1); } while (depth[q] >= p->max_depth && ++tries < 64);
    if (depth[q] >= p->max_depth) q = 0;
    par[l] = q; depth[l] = depth[q] + 1; nitems[q]++;
  }
  for (int32_t l = 0; l < nloops; ++l) { nbody[l] = rng_uni(r, p->body_lo, p->body_hi); nitems[l] += nbody[l]; }
  /* per loop: shuffled slots 0..nitems-1; children take the first slots in
   * creation order, instructions the rest; positions are 3*slot + jitter */
  int32_t **slots = (int32_t **)calloc((size_t)nloops, sizeof(int32_t *));
  int32_t *used = (int32_t *)calloc((size_t)nloops, sizeof(int32_t));
  for (int32_t l = 0; l < nloops; ++l) {
    slots[l] = (int32_t *)malloc((size_t)(nitems[l] + 1) * sizeof(int32_t));
    for (int32_t i = 0; i < nitems[l]; ++i) slots[l][i] = i;
    for (int32_t i = nitems[l] - 1; i > 0; --i) {
      int32_t j = rng_uni(r, 0, i);
      int32_t t = slots[l][i]; slots[l][i] = slots[l][j]; slots[l][j] = t;
    }
  }
  for (int32_t l = 1; l < nloops; ++l) {
    int32_t q = par[l];
    int32_t pos = 3 * slots[q][used[q]++] + rng_uni(r, 0, 2);
    int32_t kind = TRIP_UNIFORM, a = p->trip_lo, bb = p->trip_hi;
    if (rng_uni(r, 0, 999) < p->cond_permille) { a = 0; bb = 1; }
    pb_loop(b, q, pos, kind, a, bb);
  }
  for (int32_t l = 0; l < nloops; ++l)
    for (int32_t i = 0; i < nbody[l]; ++i) {
      int32_t pos = 3 * slots[l][used[l]++] + rng_uni(r, 0, 2);
      (void)pb_instr_drawn(b, l, pos, r, 0, ne - 1, p->lat_lo, p->lat_hi);
    }
  int32_t nx = (int32_t)b->xl.n;
  /* dependencies */
  for (int32_t x = 0; x < nx && nx > 0; ++x) {
    if (rng_uni(r, 0, 999) >= p->dep_permille) continue;
    int32_t nd = rng_uni(r, 1, p->max_deps_per_cons < 1 ? 1 : p->max_deps_per_cons);
    for (int32_t t = 0; t < nd; ++t) {
      int32_t pr = rng_uni(r, 0, nx - 1);
      int32_t k;
      if (p->any_k) {
        k = rng_uni(r, 0, p->k_max);
      } else {
        /* common enclosing loop of the two instructions and the body item of
         * that loop which holds each of them */
        int32_t lx = b->xl.a[x], lp = b->xl.a[pr];
        int32_t ax = lx, ap = lp, cx = -1, cp = -1;
        while (depth[ax] > depth[ap]) { cx = ax; ax = par[ax]; }
        while (depth[ap] > depth[ax]) { cp = ap; ap = par[ap]; }
        while (ax != ap) { cx = ax; ax = par[ax]; cp = ap; ap = par[ap]; }
        int32_t xpos = cx < 0 ? b->xp.a[x] : b->lpos.a[cx];
        int32_t ppos = cp < 0 ? b->xp.a[pr] : b->lpos.a[cp];
        if (cp < 0) {
          /* producer directly in the common loop: any distance, but distance 0
           * only when the producer is earlier in that body */
          int32_t hi = p->k_max < 1 ? 1 : p->k_max;
          k = xpos > ppos ? rng_uni(r, 0, p->k_max) : rng_uni(r, 1, hi);
        } else if (p->nest_far_permille > 0 && rng_uni(r, 0, 999) < p->nest_far_permille) {
          k = xpos > ppos ? rng_uni(r, 1, p->k_max + 1) : rng_uni(r, 2, p->k_max + 2);
        } else {
          k = xpos > ppos ? 0 : 1;
        }
      }
      pb_dep(b, pr, x, k);
    }
  }
  for (int32_t l = 0; l < nloops; ++l) free(slots[l]);
  free(slots); free(used); free(par); free(depth); free(nitems); free(nbody);
}

/* ------------------------------------------------------------------- API */

static void out_take(bbuild *B, synth_batch *o) {
  o->n_programs = (int32_t)B->prog_ne.n;
  o->n_loops = B->loop_parent.n;
  o->n_instrs = B->instr_loop.n;
  o->n_deps = B->dep_prod.n;
  o->n_trips = B->trips.n;
  o->prog_loop_ptr = B->prog_loop_ptr.a; o->prog_instr_ptr = B->prog_instr_ptr.a;
  o->prog_dep_ptr = B->prog_dep_ptr.a; o->prog_n_engines = B->prog_ne.a;
  o->loop_parent = B->loop_parent.a; o->loop_pos = B->loop_pos.a;
  o->instr_loop = B->instr_loop.a; o->instr_pos = B->instr_pos.a;
  o->instr_engine = B->instr_engine.a; o->instr_latency = B->instr_latency.a;
  o->dep_prod = B->dep_prod.a; o->dep_cons = B->dep_cons.a; o->dep_k = B->dep_k.a;
  o->trip_ptr = B->trip_ptr.a; o->trips = B->trips.a;
}

static int generate(int32_t cfg, uint64_t seed, int64_t first, int64_t count,
                    const synth_tree_params *tp, synth_batch *out) {
  if (!out || count < 0 || first < 0) return SYNTH_ERR_ARG;
  if (cfg == SYNTH_TREE && !tp) return SYNTH_ERR_ARG;
  if (cfg < SYNTH_TREE || cfg > SYNTH_SYNCBOUND) return SYNTH_ERR_ARG;
  memset(out, 0, sizeof *out);
  g_oom = 0;
  bbuild B;
  memset(&B, 0, sizeof B);
  vi_push(&B.prog_loop_ptr, 0); vi_push(&B.prog_instr_ptr, 0); vi_push(&B.prog_dep_ptr, 0);
  for (int64_t i = 0; i < count && !g_oom; ++i) {
    int64_t pid = first + i;
    rng_t rs = rng_for(seed, pid, 1), rt = rng_for(seed, pid, 2);
    pbuild b;
    switch (cfg) {
      case SYNTH_SMALL: gen_small(&b, &rs); break;
      case SYNTH_DEPTH2: gen_depth2(&b, &rs); break;
      case SYNTH_GEMM: gen_gemm(&b, &rs); break;
      case SYNTH_ATTENTION: gen_attention(&b, &rs); break;
      case SYNTH_CHAIN: gen_chain(&b, &rs); break;
      case SYNTH_SYNCBOUND: gen_syncbound(&b, &rs); break;
      default: gen_tree(&b, &rs, tp); break;
    }
    bb_emit(&B, &b, &rt);
    pb_free(&b);
  }
  vl_push(&B.trip_ptr, B.trips.n);
  out_take(&B, out);
  if (g_oom) { synth_free(out); return SYNTH_ERR_OOM; }
  return SYNTH_OK;
}

int synth_generate(int32_t cfg, uint64_t seed, int64_t first_program, int64_t n_programs,
                   synth_batch *out) {
  if (cfg == SYNTH_TREE) return SYNTH_ERR_ARG;
  return generate(cfg, seed, first_program, n_programs, NULL, out);
}

int synth_generate_tree(const synth_tree_params *params, uint64_t seed, int64_t first_program,
                        int64_t n_programs, synth_batch *out) {
  return generate(SYNTH_TREE, seed, first_program, n_programs, params, out);
}

void synth_free(synth_batch *b) {
  if (!b) return;
  free(b->prog_loop_ptr); free(b->prog_instr_ptr); free(b->prog_dep_ptr); free(b->prog_n_engines);
  free(b->loop_parent); free(b->loop_pos); free(b->instr_loop); free(b->instr_pos);
  free(b->instr_engine); free(b->instr_latency); free(b->dep_prod); free(b->dep_cons);
  free(b->dep_k); free(b->trip_ptr); free(b->trips);
  memset(b, 0, sizeof *b);
}
