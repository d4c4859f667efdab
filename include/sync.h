/*
 * sync.h -- C ABI of the GB300 barrier-free semaphore engine.
 *
 * The engine evaluates, checks and simulates the semaphore thresholds of
 * "A Barrier-Free Synchronization Algorithm for Multi-Engine AI Accelerators"
 * (arxiv 2608.13757) over batches of structured multi-engine programs, on one
 * GPU.  C99-compatible; no C++ types cross this boundary.
 *
 * Program model (Sec. 4.1): every construct is a loop (a conditional is a
 * loop of trip 0 or 1; the program itself is a top-level loop that runs
 * once).  Loops form a tree; a loop body is an ordered list of items --
 * datapath instructions, each bound to one engine, and child loops -- ordered
 * by a per-item position.  All engines walk this common tree, with the same
 * trip counts unless the batch gives per-engine trips (sync_batch_desc).  A
 * dependency (producer p, consumer c, offset k) is carried at
 * the innermost common loop S of p and c: consumer iteration v waits for the
 * producer through target t = v - k on S (Sec. 5.1).
 *
 * Conventions shared by every call:
 *  - Every call returns a sync_status; no C++ exception crosses the ABI.
 *    On a non-OK status, sync_last_error() describes it (thread-local).
 *  - Argument and structure errors are detected on the host before anything
 *    is launched.  Kernels run asynchronously on the caller's CUDA stream
 *    (`stream` is a cudaStream_t; NULL means the legacy default stream); a
 *    launch failure returns SYNC_ERR_CUDA.
 *  - "d_" arguments are caller-owned device buffers on the handle's device.
 *    The handle owns the device-resident program encoding and its scratch.
 *  - Results are integers and deterministic (sums and minima that do not
 *    depend on execution order).
 *
 * Pair layout (thresholds): one segment per dependency, in batch dependency
 * order; segment d starts at the offset reported by sync_pair_offsets and
 * holds one int32 per dynamic instance of the consumer, in the order of the
 * consumer loop's global iteration index g (0-based: iterations of a loop
 * numbered in program order across all iterations of its ancestors), padded
 * with zeros to a multiple of 4 entries.
 *
 * Instance layout (optional timelines): instruction-major in batch
 * instruction order; instruction x owns one int32 per global iteration of its
 * loop, starting at the sum of the instance counts of earlier instructions.
 *
 * Environment (read at each call; both only change how the work is split):
 *  - SYNCGB_LOAD_THREADS=n: host threads of sync_load_programs (default one
 *    per hardware thread, at most 32, at least 256 programs each).
 *  - SYNCGB_WIDE_INDEX=1: the threshold and check kernels index pairs with
 *    64-bit integers even when 32 bits suffice.
 *  - SYNCGB_SPLIT_MIN=n (read by sync_load_programs): the fewest instances a
 *    program needs to be simulated in pieces on several warps (default
 *    65536; see sync_simulate); SYNCGB_SPLIT_SPEC=1: such programs are
 *    always speculated, never probed, barrier-free.
 */
#ifndef SYNC_H
#define SYNC_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SYNC_OK = 0,
  SYNC_ERR_ARG = 1,              /* NULL pointer, bad enum, size mismatch      */
  SYNC_ERR_MALFORMED = 2,        /* the batch is not a valid program batch     */
  SYNC_ERR_NOT_ALLOCATABLE = 3,  /* a dependency outside Sec. 5.2's cases      */
  SYNC_ERR_OVERFLOW = 4,         /* a value stored as int32 would overflow     */
  SYNC_ERR_CUDA = 5,             /* a CUDA runtime call or launch failed       */
  SYNC_ERR_OOM = 6               /* host or device allocation failed           */
} sync_status;

/* Threshold encodings.  COUNT: the producer-completion count c of Eq. (3)
 * (per-instruction semaphores).  PERLOOP: the value T = N*c - (N-K), or 0
 * when c = 0, of the per-(loop, engine) semaphore of Eq. (5), where N is the
 * number of instructions directly in the producer's loop body on the
 * producer's engine and K the producer's 1-based rank among them.
 * PERENGINE: the per-engine allocation of Sec. 6.1 -- one semaphore per
 * engine counts every retirement on it, so the value is the 1-based position
 * of the producer's c-th instance in its engine's dynamic instruction stream
 * (program order), or 0 when c = 0. */
typedef enum { SYNC_THR_COUNT = 0, SYNC_THR_PERLOOP = 1, SYNC_THR_PERENGINE = 2 } sync_thr_mode;

/* Simulation variants.  BARRIER_FREE: the thresholds as semaphore waits
 * (Sec. 5).  BARRIER: all-engine barriers at loop statements and iteration
 * ends (Sec. 3.4).  UNROLLED: the straight-line program the loops would
 * unroll to (Sec. 3.3, the unrolled comparison of Sec. 7): per-engine
 * semaphores with static waits, so no loop-control and no wait-value
 * operations -- PERENGINE thresholds only.  Its code size is one
 * instruction per instance (sync_sizes.n_instances). */
typedef enum { SYNC_SIM_BARRIER_FREE = 0, SYNC_SIM_BARRIER = 1, SYNC_SIM_UNROLLED = 2 } sync_sim_variant;

/* Per-program simulation status (d_status). */
enum {
  SYNC_PROG_OK = 0,
  SYNC_PROG_OVERFLOW = 4,        /* static time bound exceeds INT32_MAX        */
  SYNC_PROG_DEADLOCK = 7,        /* no engine can progress before the end      */
  SYNC_PROG_ROUND_GUARD = 8,     /* internal round limit hit (a defect)        */
  SYNC_PROG_TIMEOUT = 10         /* the per-engine kernel gave up on a program
                                    after about 2 s of GPU time (a bound on a
                                    shared GPU, not a verdict on the program:
                                    rerun it); the sweep never reports it      */
};

/* Deepest supported nesting below the top-level loop. */
#define SYNC_MAX_DEPTH 15

/* A program batch in structure-of-arrays form.  Host pointers, borrowed for
 * the duration of sync_load_programs only (the data is copied).  Ids inside
 * a program are program-local (0-based).
 *   prog_loop_ptr, prog_instr_ptr, prog_dep_ptr [n_programs+1]: CSR row
 *     pointers into the loop / instruction / dependency arrays, starting at 0;
 *   prog_n_engines [n_programs]: 1..32;
 *   loop_parent, loop_pos [n_loops]: loop 0 of each program is the top-level
 *     loop (parent -1); every other loop's parent has a smaller id; loop_pos
 *     >= 0 is the loop's position among its parent's body items;
 *   instr_loop, instr_pos, instr_engine, instr_latency [n_instrs]: enclosing
 *     loop, position (>= 0, unique among the items of that loop body),
 *     engine (0..n_engines-1), latency in cycles (>= 1);
 *   dep_prod, dep_cons, dep_k [n_deps]: instruction ids and offset k >= 0;
 *   trip_ptr [n_loops+1] (starting at 0) and trips [trip_ptr[n_loops]]: loop
 *     l has one trip count (>= 0) per global iteration of its parent, in
 *     trips[trip_ptr[l] .. trip_ptr[l+1]); the top-level loop has exactly one
 *     entry, equal to 1;
 *   eng_trip_ptr, eng_trips (optional, both NULL for trips shared by all
 *     engines): per-engine trip counts (control-flow divergence, Sec. 7.5).
 *     One row per (program, loop, engine) -- programs in order, then loops,
 *     then engines, so program p's (loop l, engine e) is row R_p + l*ne + e
 *     with R_p the rows of the programs before p; eng_trip_ptr [rows+1]
 *     (starting at 0) and eng_trips [eng_trip_ptr[rows]]: a row holds the
 *     loop's trips on that engine during each global iteration of its parent
 *     on that engine (the top-level loop: one entry, 1).  When set, trip_ptr
 *     and trips are not read.  Every engine then walks the loop tree with its
 *     own trips; global iteration indices, instance and pair layouts are per
 *     engine (an instruction has one instance per iteration of its loop on
 *     its engine, a dependency one pair per instance of its consumer), and
 *     Eq. (1) is evaluated on the consumer engine's loop state (the loop-entry
 *     counts of the consumer's engine, the registers a consumer reads), while
 *     the producer's semaphore counts the producer engine's retirements: a
 *     wait that engine never reaches deadlocks the program.  Such handles
 *     take COUNT and PERLOOP thresholds and the barrier-free simulation only
 *     (SYNC_ERR_ARG otherwise): the barrier scheme needs every engine to meet
 *     the same barriers, and a per-engine wait value is a position in the
 *     producer engine's stream, which the consumer's loop state no longer
 *     determines;
 *   nonalloc_policy: what the loader does with a dependency outside the
 *     allocatable cases (see sync_load_programs): SYNC_NONALLOC_REJECT
 *     (0, the default) fails the load; SYNC_NONALLOC_BARRIER takes the
 *     paper's fallback to the barrier scheme for the ones a barrier can
 *     enforce (Sec. 5.2: a producer nested below S with a forward offset
 *     k >= 1 or a backward offset k >= 2, whose target lies in an earlier
 *     iteration of S): such a dependency gets no semaphore wait (its wait
 *     value is 0 in every threshold array, and the checker takes 0 as its
 *     minimum)
 *     and its carrying loop S, unless S is the top level, gets an all-engine
 *     barrier at the end of every iteration (drain-and-release, as in the
 *     barrier scheme) in the barrier-free simulation; the barrier scheme has
 *     those barriers already.  Such a batch takes the barrier-free and
 *     barrier simulations (SYNC_ERR_ARG for the unrolled variant) and shared
 *     trips (SYNC_ERR_ARG with per-engine trips). */
typedef enum { SYNC_NONALLOC_REJECT = 0, SYNC_NONALLOC_BARRIER = 1 } sync_nonalloc_policy;

typedef struct {
  int32_t n_programs;
  const int32_t *prog_loop_ptr, *prog_instr_ptr, *prog_dep_ptr;
  const int32_t *prog_n_engines;
  const int32_t *loop_parent, *loop_pos;
  const int32_t *instr_loop, *instr_pos, *instr_engine, *instr_latency;
  const int32_t *dep_prod, *dep_cons, *dep_k;
  const int64_t *trip_ptr;
  const int32_t *trips;
  const int64_t *eng_trip_ptr;
  const int32_t *eng_trips;
  int32_t nonalloc_policy;    /* sync_nonalloc_policy */
} sync_batch_desc;

typedef struct {
  int64_t n_pairs;          /* (dependency, consumer instance) pairs          */
  int64_t n_pairs_padded;   /* entries of a threshold array                   */
  int64_t n_instances;      /* dynamic datapath instruction instances         */
  int64_t n_loop_iters;     /* loop iterations, all loops of all programs     */
  int32_t n_programs, n_loops, n_instrs, n_deps;
  int64_t device_bytes;     /* device memory held by the handle               */
  int64_t h2d_bytes;        /* bytes sync_load_programs copied host -> device */
  int64_t struct_bytes;     /* encoding bytes the threshold and check kernels
                               read besides the thresholds (COUNT and PERLOOP),
                               each array once: per-iteration trip starts and
                               ancestors derived at load time, trip prefix
                               sums of nested producers' loops and their
                               offsets, dependency, segment and tile tables
                               (PERENGINE reads the engine-stream positions of
                               the waited producers' instances besides)       */
  int64_t code_bytes_looped;   /* code-size proxy of the barrier-free program
                                  (the code-size comparison of Sec. 7, RQ2), at
                                  SYNC_CODE_BYTES_PER_INSTR per instruction:
                                  every datapath instruction once; per waited
                                  dependency 5 wait-value ops (per-loop, Table
                                  1) and the wait; per loop below the top level
                                  and engine 4 control ops (r-hat := 0 at the
                                  statement, branch, r++, r-hat++); per engine
                                  one barrier per loop with fallback barriers */
  int64_t code_bytes_unrolled; /* the same for the unrolled program: one
                                  instruction per datapath instance and one
                                  static wait per waited pair                 */
  int32_t n_split_programs;    /* programs sync_simulate may simulate in pieces
                                  on several warps (see sync_simulate)        */
  int32_t n_pieces;            /* their pieces                                */
} sync_sizes;

/* Instruction size of the code-size proxy (a 128-bit instruction word). */
#define SYNC_CODE_BYTES_PER_INSTR 16

/* Timing-model constants in cycles, all >= 0 (see sync_simulate). */
typedef struct {
  int32_t ii;                 /* issue interval of a datapath instruction     */
  int32_t c_branch;           /* loop branch at each iteration start         */
  int32_t c_regop;            /* one register operation                       */
  int32_t c_wait_ops_count;   /* wait-value ops per dependency, COUNT (3, Table 1) */
  int32_t c_wait_ops_perloop; /* wait-value ops per dependency, PERLOOP (5, Table 1) */
  int32_t c_barrier;          /* all-engine barrier: handshake, reset, handshake */
  int32_t c_wait_ops_perengine_level; /* PERENGINE: extra ops per wait for every loop
                                 strictly between the top level and the
                                 producer's loop (3: the term N_l*(r_l - 1) of
                                 Sec. 6.1's path sum, O(D) in Table 1) */
  int32_t trip_register_elision; /* 1: omit r-hat of every loop at which only
                                 offset-0 dependencies are carried (Sec. 5.1:
                                 its no-wait check r-hat <= 0 never holds when
                                 a consumer issues), so its loop statement and
                                 iteration starts lose one register op each;
                                 0: every loop keeps r-hat (the default) */
  int32_t licm;               /* 1: loop-invariant code motion of the per-engine
                                 path sums (Sec. 6.2), barrier-free PERENGINE:
                                 the term of each loop l strictly between the
                                 top level and a producer's loop is kept in a
                                 cached partial sum that engine e updates at
                                 every iteration start of l (cost
                                 c_wait_ops_perengine_level, once per producer
                                 engine whose waits on e pass below l); a wait
                                 then costs c_wait_ops_perloop plus c_regop
                                 (the read of the cached sum; nothing when the
                                 producer's loop has depth <= 1).  0: off */
  int32_t cse;                /* 1: common-subexpression elimination of wait
                                 values (Sec. 6.2), barrier-free: on one engine,
                                 within one visit of a straight-line segment of
                                 a loop body (the items between two child loops,
                                 in one iteration), the waits in program order
                                 (an instruction's dependencies in dependency
                                 order) reuse an earlier wait's value when it
                                 has the same producer and offset (no cost),
                                 else its mask when it has the same carrying
                                 loop S and offset (min(c_regop, wait ops) less)
                                 and, PERENGINE, its outer partial sum when it
                                 has the same producer loop and producer engine
                                 (no levels term, or with licm no read).  0: off */
} sync_sim_params;

typedef struct sync_programs sync_programs;   /* opaque; owns device memory */

/* Validates a batch, classifies every dependency into the allocatable cases
 * of Sec. 5.2 (producer in S with any offset -- except offset 0 when the
 * consumer precedes the producer in S's body on the same engine, which can
 * never issue; producer nested below S and forward with offset 0; nested and
 * backward with offset 1), computes N and K of the per-loop allocation
 * (Sec. 5.5), and builds the device-resident encoding on `device`: loop
 * table, per-loop trip prefix sums (rowptr), dependency table, the derived
 * per-iteration arrays of the threshold kernels, per-(loop, engine)
 * instruction streams.
 * Returns SYNC_ERR_MALFORMED for structural errors (listed with sync.h's
 * batch description), SYNC_ERR_NOT_ALLOCATABLE for a dependency outside the
 * cases above (with SYNC_NONALLOC_BARRIER: one that no barrier at the end
 * of its carrying loop's iterations enforces either -- a nested backward
 * offset 0, or offset 0 to a later producer on the same engine),
 * SYNC_ERR_ARG for a policy value outside sync_nonalloc_policy or barrier
 * fallbacks in a batch with per-engine trips, SYNC_ERR_OVERFLOW when a loop's iteration total, a per-loop
 * threshold N*total, a pair count or an instance count exceeds INT32_MAX
 * (int64 totals are supported for pairs and instances across programs).
 * On SYNC_OK, *out receives a handle to free with sync_free_programs.
 * The call waits on `stream` for its validation pass (to report failures);
 * the rest of the load is left queued on `stream`, its completion recorded
 * in an event of the handle: every later call on the handle, on any stream,
 * makes that stream wait for the event first, and sync_free_programs waits
 * for the device.  The caller's arrays may be released when the call returns.
 * The host checks the batch's shape (the CSR offsets, trip offsets, NULL
 * arrays), then runs one routine per program in two passes on host threads
 * (SYNCGB_LOAD_THREADS=n sets their number): the first validates the
 * program and counts the entries it adds to each table, the second writes
 * the encoding at the programs' offsets (the prefix sums of the counts)
 * into pinned host memory, copied to the device in one transfer; the
 * per-iteration tables (derived arrays, per-mode semaphore records, tile
 * tables) are then built on the device.  The first failure
 * reported is the lowest-numbered failing program's first failure in check
 * order, the same as sync_validate_programs reports.  The device encoding
 * is one allocation owned by the handle.  The library keeps the passes'
 * host scratch and the pinned staging memory for reuse by later loads (one
 * set per load running at the same time, each grown to the largest batch
 * it has held) until the process ends. */
sync_status sync_load_programs(const sync_batch_desc *desc, int device, void *stream,
                               sync_programs **out);

/* The validation of sync_load_programs on the host alone (no device, no
 * CUDA call): the same shape checks and per-program checks, run on host
 * threads; returns the status and sets the message sync_load_programs would
 * for the same batch, or SYNC_OK when the batch would load (device memory
 * aside).  SYNCGB_LOAD_THREADS=n sets the number of host threads. */
sync_status sync_validate_programs(const sync_batch_desc *desc);

/* Sizes of a loaded batch (host struct). */
sync_status sync_query(const sync_programs *h, sync_sizes *out);

/* Host copies of the pair layout: offsets [n_deps + 1] int64 (segment starts;
 * entry n_deps is n_pairs_padded) and, unless NULL, counts [n_deps] int32
 * (consumer instances of each dependency, i.e. unpadded segment lengths).
 * The first call on a handle reads them back from the device (synchronous
 * copies on the handle's device); later calls copy the kept host copy. */
sync_status sync_pair_offsets(const sync_programs *h, int64_t *offsets, int32_t *counts);

/* Threshold kernel: for every pair (dependency d, consumer instance g) the
 * wait value of Sec. 5.3, Eq. (2), with the trip register r-hat_S (position
 * of the consumer's S-iteration in its trip, 1-based), the monotone registers
 * (iteration counts including the current one, Sec. 5.1) and expr of
 * Sec. 5.2 (r_S - k for a producer in S, r_P for a nested producer, r_P
 * counted through the current / previous S-iteration when forward /
 * backward), in `mode`'s encoding (Eq. 3, Eq. 5 or Sec. 6.1).
 * d_thr: [n_pairs_padded] int32, caller-owned device memory, fully written
 * (padding entries 0, and the pairs of a dependency taken by the barrier
 * fallback of SYNC_NONALLOC_BARRIER: 0, no wait).
 * The first PERENGINE call (thresholds or check) on a handle derives the
 * engine-stream positions of the waited producers' instances on the GPU: it
 * allocates device memory held by the handle (sync_sizes.device_bytes grows)
 * and synchronizes `stream`; later calls reuse them.  It returns
 * SYNC_ERR_OVERFLOW if an engine of a program has more than INT32_MAX
 * instances. */
sync_status sync_eval_thresholds(const sync_programs *h, sync_thr_mode mode, int32_t *d_thr,
                                 void *stream);

/* Minimality checker: recomputes the dependency-satisfaction condition of
 * Eq. (1) for every pair (the target t = v - k on S, underflow when its
 * S-component is <= 0, otherwise the producer instances lexicographically
 * <= t) and compares the value stored in d_thr (read in `mode`'s encoding)
 * with the required minimum: below it is unsafe (the consumer could issue
 * before its producer, Sec. 4), above it over-synchronises.
 * d_counts: [2] uint64 device -- unsafe, over-synchronised pair counts;
 * d_first_bad: [1] int64 device -- smallest offending index into d_thr, or
 * -1.  Both are overwritten (no accumulation across calls); padding entries
 * of d_thr are ignored.  A barrier-fallback dependency (SYNC_NONALLOC_BARRIER)
 * is enforced by barriers, not by its wait value: its minimum is 0, so a
 * positive stored value counts as over-synchronised. */
sync_status sync_check_minimal(const sync_programs *h, sync_thr_mode mode, const int32_t *d_thr,
                               unsigned long long *d_counts, long long *d_first_bad,
                               void *stream);

/* Schedule simulator.  Runs every program under a timing model of the
 * paper's execution model: per-engine in-order issue and in-order
 * retirement, waits `semaphore >= threshold` at issue, increments at
 * retirement (Sec. 3.2-3.3, Appendix A.5), counters starting at 0
 * (Appendix A.6).  Semaphores are per producer instruction (COUNT), per
 * (loop, engine) (PERLOOP) or per engine (PERENGINE, incremented by every
 * retirement on the engine); d_thr holds the thresholds in that encoding
 * (normally the output of sync_eval_thresholds).  Costs in cycles, per
 * engine cursor t:
 *   loop statement: barrier-free t += c_regop (r-hat := 0); barrier: barrier
 *   iteration start: barrier-free t += c_branch + 2*c_regop; barrier: t += c_branch
 *   (with trip_register_elision, a loop that carries only offset-0
 *   dependencies, or none, costs 0 at its statement and c_branch + c_regop
 *   at each iteration start, barrier-free)
 *   iteration end: barrier: barrier; barrier-free: a barrier at the end of
 *     each iteration of a loop that carries a barrier-fallback dependency
 *     (SYNC_NONALLOC_BARRIER), none otherwise
 *   datapath x (barrier-fallback dependencies are not waited on and cost
 *     nothing here): barrier-free t += sum over its dependencies of the wait
 *     ops: c_wait_ops_count (COUNT), c_wait_ops_perloop (PERLOOP), or
 *     c_wait_ops_perloop + c_wait_ops_perengine_level * (depth of the
 *     producer's loop - 1, at least 0; the top level has depth 0)
 *     (PERENGINE);
 *     issue = max(t, times at which the waited semaphores reached their
 *     thresholds); retire = max(issue + latency, previous retire on the
 *     engine); t = issue + ii
 *   barrier: release = max over engines of max(t, last retire) + c_barrier;
 *     every engine continues at release
 *   the top-level loop costs nothing; makespan = max over engines of
 *   max(t, last retire).
 * The ALU reductions licm and cse (sync_sim_params) change the wait-op and
 * iteration-start costs above as described there; with licm the static time
 * bound (SYNC_PROG_OVERFLOW) adds c_wait_ops_perengine_level per cached-sum
 * update and c_regop per pair of a wait with a cached-sum read.
 * Large programs (sync_sizes.n_split_programs) whose top-level body is one
 * loop L are simulated in pieces -- runs of L's iterations -- on separate
 * warps when every wait of a piece targets an increment of the same piece
 * (checked on the thresholds of each call; otherwise, and whenever a piece
 * deadlocks or waits forward, the program is simulated whole): the barrier
 * scheme from the barrier before each piece, the barrier-free scheme by
 * composing the pieces' max-plus maps of the engines' cursors and last
 * retires (read off by one probe run per cursor and last retire), or, for
 * a batch of many such programs, by speculation: a piece runs from a guessed
 * start and is accepted when its true start differs from the guess by one
 * constant in every cursor and last retire (a few rounds of guesses at
 * most).  The results are identical either way.
 * UNROLLED: as barrier-free with c_branch, c_regop and every wait-op cost
 * taken as 0 (ii and latencies unchanged); it requires PERENGINE and a batch
 * without barrier-fallback dependencies, and returns SYNC_ERR_ARG otherwise.
 * Outputs per program (device, [n_programs]): d_makespan (int32, -1 unless
 * status OK), d_checksum (uint64, 0 unless OK: the sum mod 2^64 over
 * datapath instances of (a << 32) | b in 32-bit arithmetic, a = (issue ^
 * (n*0x9E3779B9 + e)) * 0x85EBCA6B, a ^= a >> 13, b = (retire ^
 * (n*0xC2B2AE35 + e)) * 0x27D4EB2F, b ^= b >> 15, e the engine and n the
 * instance's 1-based ordinal in engine e's stream), d_status (SYNC_PROG_*).  d_issue / d_retire:
 * [n_instances] int32 in instance layout, both NULL or both set (entries of
 * programs whose status is not OK are unspecified).  The handle's history
 * scratch is shared: calls on one handle must not overlap on the GPU. */
sync_status sync_simulate(const sync_programs *h, sync_thr_mode mode, const int32_t *d_thr,
                          const sync_sim_params *params, sync_sim_variant variant,
                          int32_t *d_makespan, unsigned long long *d_checksum, int32_t *d_status,
                          int32_t *d_issue, int32_t *d_retire, void *stream);

/* Fused threshold -> check -> simulate: sync_simulate without a threshold
 * array.  Every wait value is computed where the simulators reach the
 * consumer, from the loop state of the walk (the register form of Sec. 5.1:
 * the masked r_S - k or r_P, encoded as the mode says), so the 4 bytes per
 * pair are neither written nor read.  Outputs, statuses and argument rules
 * as sync_simulate (identical results).  d_counts ([2] uint64 device) and
 * d_first_bad ([1] int64 device), both NULL or both set: each wait value is
 * also recomputed by Eq. (1) as sync_check_minimal does, and mismatches are
 * counted (unsafe, over-synchronised) with the smallest offending pair index
 * (in sync_eval_thresholds' layout), or -1; only programs whose status is
 * OK contribute.  Both are overwritten.  PERENGINE derives the engine-stream
 * positions on first use, as sync_eval_thresholds does. */
sync_status sync_simulate_fused(const sync_programs *h, sync_thr_mode mode, const sync_sim_params *params,
                                sync_sim_variant variant, int32_t *d_makespan, unsigned long long *d_checksum,
                                int32_t *d_status, int32_t *d_issue, int32_t *d_retire,
                                unsigned long long *d_counts, long long *d_first_bad, void *stream);

/* Size of the device scratch used by sync_simulate_noalloc (see below). */
#define SYNC_NOALLOC_SCRATCH_BYTES (64u << 20)

/* sync_simulate without any device allocation during the call.
 *
 * The paper has no counterpart; this entry point exists for callers of this
 * library that cannot call cudaMalloc or cudaFree around a simulation: for
 * example a host thread that must not trigger the implicit device-wide
 * synchronisation an allocation may cause, or a process whose device memory
 * is fully reserved up front by its own allocator.  The handle must already
 * be loaded; the outputs are caller-owned as for sync_simulate, and the
 * results are identical to sync_simulate's.
 *
 * Instead of the handle's scratch, the call uses one scratch array of
 * SYNC_NOALLOC_SCRATCH_BYTES that the library declares statically in device
 * memory: every GPU that loads the library holds it until the process exits.
 * It must hold the semaphore history of the batch (one int32 per increment
 * of every waited semaphore), a program list and two counters; a batch that
 * does not fit returns SYNC_ERR_ARG with the required size in
 * sync_last_error(), before anything is launched.  The call zeroes the
 * counters it needs on `stream`; the history is written before it is read.
 *
 * Every call looks up the array's device address with the handle's device
 * current.  With CUDA's lazy module loading (the default) the array is only
 * reserved when the library's module is first loaded on a device, which is
 * this lookup in the first call there: that call needs
 * SYNC_NOALLOC_SCRATCH_BYTES of free device memory and fails with
 * SYNC_ERR_CUDA without it.  A caller whose allocator reserves device memory
 * up front should therefore make one warm-up call (on a small batch) at
 * set-up, before the reservation and before any stream capture.  All
 * calls share the one array and it keeps the last call's contents, so calls
 * whose work overlaps on the GPU (other streams, other threads) race with
 * each other: serialise them, e.g. on one stream. */
sync_status sync_simulate_noalloc(const sync_programs *h, sync_thr_mode mode, const int32_t *d_thr,
                                  const sync_sim_params *params, sync_sim_variant variant,
                                  int32_t *d_makespan, unsigned long long *d_checksum,
                                  int32_t *d_status, int32_t *d_issue, int32_t *d_retire,
                                  void *stream);

/* Releases a handle (NULL is ignored).  Waits for the device to finish work
 * that may still use the handle's memory. */
void sync_free_programs(sync_programs *h);

/* Message for the last non-OK status returned on this thread ("" if none). */
const char *sync_last_error(void);

/* Number of kernels this library has launched in this process, over every
 * handle, stream and thread: the loader's kernels, and per call of the
 * entry points above the kernels it enqueued (sync_simulate: one sweep and
 * one per-engine launch per call, plus the piece-parallel kernels when
 * programs are cut into pieces).  A launch counts once the CUDA runtime has
 * accepted it.  Monotonic; reading it has no other effect and cannot fail. */
int64_t sync_kernel_launches(void);

#ifdef __cplusplus
}
#endif
#endif /* SYNC_H */
