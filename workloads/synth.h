/*
 * Seeded synthetic program batches (shared input generator; holds none of the
 * synchronisation method's arithmetic).  Arrays are structure-of-arrays,
 * int32 unless noted, with program-local loop and instruction ids.
 */
#ifndef SYNTH_H
#define SYNTH_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
  SYNTH_TREE = 0,        /* general random trees (synth_generate_tree)          */
  SYNTH_SMALL = 1,       /* 1 program, 2 engines, trip-16 loop, 6 instructions   */
  SYNTH_DEPTH2 = 2,      /* depth-2 nest, U[1,64] trips, 16-instruction bodies   */
  SYNTH_GEMM = 3,        /* tiled 4096^3 GEMM, M/N/K = 32/8/32                   */
  SYNTH_ATTENTION = 4,   /* causal flash attention, head/q-tile/kv-tile          */
  SYNTH_CHAIN = 5,       /* random chain programs, trips U[0,32], density 0.3    */
  SYNTH_SYNCBOUND = 6    /* single-instruction conditionals, sync-bound          */
};

enum { SYNTH_OK = 0, SYNTH_ERR_ARG = 1, SYNTH_ERR_OOM = 2 };

typedef struct {
  int32_t n_programs;
  int64_t n_loops, n_instrs, n_deps, n_trips;
  int32_t *prog_loop_ptr, *prog_instr_ptr, *prog_dep_ptr; /* [n_programs+1] */
  int32_t *prog_n_engines;                                /* [n_programs]   */
  int32_t *loop_parent, *loop_pos;                        /* [n_loops]      */
  int32_t *instr_loop, *instr_pos, *instr_engine, *instr_latency; /* [n_instrs] */
  int32_t *dep_prod, *dep_cons, *dep_k;                   /* [n_deps]       */
  int64_t *trip_ptr;                                      /* [n_loops+1]    */
  int32_t *trips;                                         /* [n_trips]      */
} synth_batch;

typedef struct {
  int32_t engines_lo, engines_hi;
  int32_t max_depth;            /* nesting levels below the top-level loop      */
  int32_t loops_lo, loops_hi;   /* number of loops besides the top-level one    */
  int32_t body_lo, body_hi;     /* instructions directly in each loop body      */
  int32_t trip_lo, trip_hi;     /* trip drawn per parent iteration              */
  int32_t cond_permille;        /* chance that a loop is a conditional (0..1)   */
  int32_t lat_lo, lat_hi;
  int32_t dep_permille;         /* chance that an instruction is a consumer     */
  int32_t max_deps_per_cons;
  int32_t k_max;
  int32_t any_k;                /* 1: offsets drawn freely (may be non-allocatable) */
  int32_t nest_far_permille;    /* chance that a nested producer gets an offset
                                   beyond the allocatable one (forward 1..k_max+1,
                                   backward 2..k_max+2): a barrier-fallback case */
} synth_tree_params;

/* Programs first_program .. first_program+n_programs-1 of a fixed config; a
 * program's content depends only on (cfg, seed, its id). */
int synth_generate(int32_t cfg, uint64_t seed, int64_t first_program, int64_t n_programs,
                   synth_batch *out);
int synth_generate_tree(const synth_tree_params *params, uint64_t seed, int64_t first_program,
                        int64_t n_programs, synth_batch *out);
void synth_free(synth_batch *b);

#ifdef __cplusplus
}
#endif
#endif
