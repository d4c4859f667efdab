/*
 * CPU oracle for barrier-free semaphore thresholds -- TEST INFRASTRUCTURE.
 *
 * Only the test suite, the smoke check and the benchmark's CPU-baseline leg
 * may call this code.  It shares nothing with the GPU library: its own types,
 * its own walk of the loop tree, its own arithmetic.
 *
 * Pair layout: dependency-major in batch dependency order; inside dependency
 * d, one entry per dynamic instance of the consumer, in the order the
 * consumer's loop iterates (its global iteration index g = 0, 1, ...).  No
 * padding.
 *
 * Instance layout (issue/retire outputs): instruction-major in batch
 * instruction order; instruction x has one entry per global iteration of its
 * loop.
 */
#ifndef SYNC_ORACLE_H
#define SYNC_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
  int32_t n_programs;
  const int32_t *prog_loop_ptr, *prog_instr_ptr, *prog_dep_ptr, *prog_n_engines;
  const int32_t *loop_parent, *loop_pos;
  const int32_t *instr_loop, *instr_pos, *instr_engine, *instr_latency;
  const int32_t *dep_prod, *dep_cons, *dep_k;
  const int64_t *trip_ptr;
  const int32_t *trips;
  /* optional per-engine trip counts (NULL: every engine runs `trips`): one
   * row per (program, loop, engine), programs in order, then loops, then
   * engines; a row holds the loop's trips on that engine during each global
   * iteration of its parent on that engine.  When set, `trips` is unused. */
  const int64_t *eng_trip_ptr;
  const int32_t *eng_trips;
  /* 0: every dependency is taken as a semaphore wait; 1: the fallback of
   * Sec. 5.2 to the barrier scheme for the non-allocatable dependencies a
   * barrier enforces (ORC_CASE_BARRIER below) */
  int32_t nonalloc_policy;
} orc_batch;

enum { ORC_OK = 0, ORC_ERR_ARG = 1, ORC_ERR_MALFORMED = 2, ORC_ERR_NOT_ALLOCATABLE = 3,
       ORC_ERR_OVERFLOW = 4, ORC_ERR_OOM = 6 };

/* threshold modes: the producer-completion count c (Eq. 3), the per-loop
 * semaphore value T = N*c - (N-K), 0 when c = 0 (Eq. 5), or the per-engine
 * semaphore value (Sec. 6.1): one counter per engine counts every retirement
 * on that engine, so the wait is for the 1-based ordinal of the producer's
 * c-th instance in its engine's dynamic instruction stream, 0 when c = 0 */
enum { ORC_COUNT = 0, ORC_PERLOOP = 1, ORC_PERENGINE = 2 };

/* allocatable cases of Sec. 5.2; with nonalloc_policy 1, ORC_CASE_BARRIER is
 * a producer nested below S with a forward offset >= 1 or a backward offset
 * >= 2 (its target lies in an earlier iteration of S, so an all-engine
 * barrier at the end of every iteration of S enforces it); ORC_CASE_NONE is
 * what remains outside the cases */
enum { ORC_CASE_PS = 0, ORC_CASE_NEST_FWD = 1, ORC_CASE_NEST_BWD = 2, ORC_CASE_NONE = 3,
       ORC_CASE_BARRIER = 4 };

/* simulator variants (UNROLLED: the straight-line program, per-engine
 * thresholds, no loop-control or wait-value operations) and per-program
 * status codes */
enum { ORC_BARRIER_FREE = 0, ORC_BARRIER = 1, ORC_UNROLLED = 2 };
enum { ORC_SIM_OK = 0, ORC_SIM_OVERFLOW = 4, ORC_SIM_DEADLOCK = 7 };

typedef struct {
  int32_t ii;                 /* issue interval of a datapath instruction      */
  int32_t c_branch;           /* loop branch at each iteration start          */
  int32_t c_regop;            /* one register operation                        */
  int32_t c_wait_ops_count;   /* wait-value ops per dependency, count mode     */
  int32_t c_wait_ops_perloop; /* wait-value ops per dependency, per-loop mode  */
  int32_t c_barrier;          /* all-engine barrier handshake + reset          */
  int32_t c_wait_ops_perengine_level; /* per-engine mode: per enclosing loop level */
  int32_t trip_register_elision; /* 1: no r-hat for loops carrying only offset-0 deps */
  int32_t licm;               /* 1: loop-invariant code motion of the per-engine
                                 path sums (Sec. 6.2), see oracle.c */
  int32_t cse;                /* 1: common-subexpression elimination of wait
                                 values within a straight-line segment (Sec. 6.2) */
} orc_sim_params;

/* Per-engine trip counts (control-flow divergence, Sec. 7.5): each engine
 * walks the common loop tree with its own trips.  A dependency's pairs are
 * its consumer's instances, and Eq. (1) is evaluated on the consumer
 * engine's loop state (the loop-entry counts H_e of the consumer's engine:
 * the registers an implementation reads); the producer's semaphore counts
 * the producer engine's retirements, so a wait the producer engine never
 * reaches leaves the program deadlocked.  Count and per-loop modes only,
 * barrier-free simulation only (ORC_ERR_ARG otherwise).
 * Global iteration indices, instance and pair layouts are per engine: an
 * instruction has one instance per iteration of its loop on its engine. */

/* Sizes: pairs and instances in the layouts above. */
int orc_sizes(const orc_batch *b, int64_t *n_pairs, int64_t *n_instances);

/* Code-size proxy of the code-size comparison (Sec. 7, RQ2), in
 * instructions, summed over the programs.  The looped barrier-free program
 * (per-loop semaphores): every datapath instruction once; per dependency that
 * is waited on (not a barrier fallback) the 5 wait-value ops of Table 1 and
 * the wait instruction; per engine, every loop below the top level costs 4
 * control instructions (r-hat := 0, the branch, r++, r-hat++) and every loop
 * that ends its iterations with fallback barriers one barrier.  The unrolled
 * program: one instruction per datapath instance and one static wait per
 * (waited dependency, consumer instance) pair. */
int orc_code_size(const orc_batch *b, int64_t *looped, int64_t *unrolled);

/* Per dependency: innermost common loop S, producer parent loop P (program-
 * local ids), allocatable case (ORC_CASE_*), N and K of the per-loop
 * allocation.  Any output pointer may be NULL. */
int orc_classify(const orc_batch *b, int32_t *S, int32_t *P, int32_t *kase, int32_t *N,
                 int32_t *K);

/* Eq. (1) by definition: for each consumer instance, the number of producer
 * instances whose iteration vector restricted to the common loops is
 * lexicographically <= the target t = v - delta (0 on underflow). */
int orc_thresholds_bruteforce(const orc_batch *b, int mode, int32_t *out);
/* The same definition evaluated by counting producer instances per iteration
 * of the innermost common loop and prefix-summing. */
int orc_thresholds(const orc_batch *b, int mode, int32_t *out);
/* The paper's registers replayed literally per engine (Fig. 7/8): r-hat := 0
 * at each loop statement, r++ and r-hat++ at each iteration start, and the
 * masked wait value of Eq. (2)/(3)/(5) before each consumer.  Entries of
 * non-allocatable dependencies are set to -1, those of ORC_CASE_BARRIER
 * dependencies to 0 (the barrier fallback emits no wait).  Count and per-loop modes
 * only. */
int orc_register_replay(const orc_batch *b, int mode, int32_t *out);

/* Minimality check of a threshold array against Eq. (1): counts[0] = pairs
 * whose threshold is below the minimum (unsafe), counts[1] = above it
 * (over-synchronised); first_bad = first such pair index or -1.  An
 * ORC_CASE_BARRIER dependency is enforced by a barrier: its minimum is 0, so
 * any positive value over-synchronises. */
int orc_check(const orc_batch *b, int mode, const int32_t *thr, uint64_t counts[2],
              int64_t *first_bad);

/* Event-stepped semaphore machine (timing model stated in oracle.c).  `thr`
 * is a threshold array in `mode`'s encoding; the machine waits on the
 * per-producer semaphore (count), the per-(loop, engine) semaphore
 * (per-loop) or the producer's engine semaphore, which every retirement on
 * that engine increments (per-engine), until its value reaches the
 * threshold.  The unrolled variant needs per-engine thresholds.
 * ORC_CASE_BARRIER dependencies are not waited on and cost no wait ops; the
 * loop that carries one (unless it is the top level) ends every iteration
 * with an all-engine barrier, also barrier-free (the barrier scheme has
 * those barriers anyway); the static time bound counts one c_barrier per
 * such barrier.  Such programs take neither the unrolled variant nor
 * per-engine trips (ORC_ERR_ARG).
 * issue/retire may be NULL. */
int orc_simulate(const orc_batch *b, int mode, const int32_t *thr, const orc_sim_params *prm,
                 int variant, int32_t *makespan, uint64_t *checksum, int32_t *status,
                 int32_t *issue, int32_t *retire);

#ifdef __cplusplus
}
#endif
#endif
