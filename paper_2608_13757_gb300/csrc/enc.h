// Device-resident program encoding shared by the host loader and the kernels.
//
// All ids are global across the batch.  Loops are numbered as in the input
// (program by program), so a program's loops are contiguous and parents
// precede children.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/sync.h"

namespace syncgb {

enum : int32_t { CASE_PS = 0, CASE_NEST_FWD = 1, CASE_NEST_BWD = 2, CASE_BARRIER = 3 };

// Pairs are processed in chunks of 4 consecutive entries (one int4).  The
// threshold kernels find a chunk's dependency through a table of the first
// dependency of every tile of kTilePairs pairs: tiles much shorter than a
// typical segment leave most chunks with a one-dependency range, no search
// (128 against 1024: threshold kernel 0.490 -> 0.442 ms on the chain batch).
constexpr int kChunk = 4;
constexpr int kTilePairs = 128;

// Per loop.  rowptr_l[j], j in [0, total(parent)], is the number of l's
// iterations that start before the parent's global iteration j (exclusive
// prefix sum of the trips).  The top-level loop has rowptr [0, 1].
struct alignas(16) LoopInfo {
  int64_t rowptr_off;
  int32_t parent;     // -1 for a top-level loop
  int32_t total;      // global iterations
  int32_t n_parent;   // total(parent), 1 for a top-level loop
  int32_t depth;
};

// Per dependency.  `path` points into the int64 path pool:
//   [0, up)            rowptr offsets of the loops from the consumer's loop
//                      up to (excluding) S, innermost first (read at load
//                      time, for the consumer iterations' S-ancestors);
//   [up, up+clen)      rowptr offsets of the loops from S's child down to P
//                      (nested cases; clen = 0 when P = S).
struct alignas(16) DepInfo {
  // read for every chunk: the first 48 bytes (three 16-byte loads)
  int64_t seg_off;    // pair-layout offset of this dependency's segment
  int64_t src;        // derived pool, per consumer iteration: its trip start of S
                      // (consumer directly in S) or its enclosing S-iteration (below
                      // S); -1 when S runs once (S-iteration 0, trip start 0)
  int64_t tstart;     // derived pool: first iteration of the trip, per iteration of S
  int32_t total;      // consumer instances (= total of the consumer's loop)
  int32_t k, N, K;
  int32_t up;         // consumer depth below S
  int32_t clen;       // producer depth below S
  // read for nested producers and per-engine values only
  int64_t path;
  int64_t ordp;       // ordinal pool: engine-stream position per producer instance
  int32_t kase, pad_;
};
// Per program, for the simulator.
constexpr int kModes = 3;   // threshold encodings: COUNT, PERLOOP, PERENGINE

struct alignas(16) ProgInfo {
  int64_t agg_lat;    // sum over instructions of instances * latency (saturated)
  int64_t n_inst;     // datapath instances
  int64_t n_pairs;    // (dependency, consumer instance) pairs
  int64_t n_stmt;     // loop statements one engine reaches (sum over non-top loops of
                      // total(parent); per-engine trips: the largest over the engines)
  int64_t n_iter;     // loop iterations of one engine (likewise)
  int64_t eng_stmt;   // loop statements summed over the engines
  int64_t eng_iter;   // loop iterations summed over the engines
  int64_t el_stmt;    // of these, those of loops that carry no offset > 0 (whose trip
  int64_t el_iter;    // register can be elided)
  int64_t pair_levels;  // sum over pairs of the per-engine wait's extra levels
  int64_t fb_iters;   // iterations ended by a barrier-fallback barrier (barrier-free);
                      // > 0: simulated by the per-engine kernel
  int64_t licm_upd;   // LICM (per-engine waits): cached-sum updates, summed over the
                      // (loop, engine) rows of their counts times the loop's iterations
  int64_t lv_pairs;   // pairs of per-engine waits whose producer loop has depth > 1
  int32_t ne;
  int32_t le_base;    // row of (top-level loop, engine 0); row of (program-local
                      // loop l, engine e) = le_base + l*ne + e
  int32_t nsem[kModes];    // waited semaphores, per threshold mode
  int32_t semhb_off[kModes];  // first entry of the program's history bases, per mode
  int32_t loop_base;  // global id of the program's top-level loop
  int32_t divergent;  // 1: engines run their own trip counts (per-engine kernel only)
};

// Program-order sweep tables.  Per loop, a plan: its body cut at child loops
// into straight-line segments; items [plan_ptr[l], plan_ptr[l+1]):
//   {ITEM_SEG, first chunk, chunks, w}
//   {ITEM_LOOP, child loop (global id), child's elidable-trip-register flag, 0}
// with w >= 0 a multi-iteration chunk, w <= -2 (the body's last segment) a
// chunk of that segment and the next iteration's first (chunk -2 - w), -1
// neither.  A chunk holds up to 32 datapath records of one segment (all
// engines), in lanes ordered engine-major (then iteration copy, then body
// position):
//   chunk {first lane record, lanes, iteration copies, engines with lanes in
//          the last copy}
// A multi-iteration chunk repeats a short innermost segment for `copies`
// consecutive iterations; a joined chunk holds a body's closing segment
// (copy 0) and its opening one (copy 1) -- both for the barrier-free sweep
// only, whose iteration start between the copies is inside the chunk.  Per lane:
//   lrec {x (global instruction), latency, dependencies, first dependency}
//   lmeta {engine, copy, first lane of the engine's run, flags}
//     flags bit 0: first record of its engine in a copy >= 1 (an iteration
//     start precedes it); bit 1: last lane of its engine's run
//   lsem per mode {semaphore, stride, koff, levels} as the simulator's records.
enum : int32_t { ITEM_SEG = 0, ITEM_LOOP = 1 };
constexpr int32_t LANE_ITER_START = 1;
constexpr int32_t LANE_RUN_LAST = 2;

// Simulator op records, one list ("row") per (loop, engine): the engine's own
// instructions and every child loop of the loop's body, in body order, then
// an END record.  16 bytes each:
//   datapath  {x >= 0 (global instruction), latency, dependencies consumed,
//              first entry in the consumer-grouped dependency list}
//   loop      {OP_LOOP, row of (child, engine 0), rowptr offset lo, hi}
//   end       {OP_END, 0, 0, 0}
// Per record: opstop = index of the first LOOP or END record at or after it
// in its row.  Per row: op_ptr = first record, rowinfo = {END record index,
// bit 0: the row holds a LOOP record, bit 1: the row's loop carries no
// offset > 0 (its trip register can be elided), bit 2: the row's loop ends
// every iteration with a barrier-fallback barrier}.
// Per-mode semaphore records parallel to the op records (mode 0 = one
// semaphore per producer instruction, mode 1 = one per (loop, engine),
// mode 2 = one per engine):
//   {semaphore (program-local, -1 if nothing waits on it), increments per
//    iteration (1 or N), koff (1 or K), levels}: the increment of iteration g
//    brings the semaphore to stride*g + koff and its retire time lives at
//    history slot semhb[semaphore] + stride*g + koff - 1.  Per-engine
//    semaphores have stride -1: every instance of the engine increments, and
//    the increment is the instance's ordinal n in the engine's stream (slot
//    n - 1).  levels (mode 2): sum over the record's dependencies of the
//    loops strictly between the top level and the producer's loop, the
//    extra terms of a per-engine wait.
// Consumer-grouped dependencies: segment offset (int64) and, per mode, the
// waited semaphore (program-local).  semhb: per program and mode, the
// history base of each waited semaphore.
constexpr int32_t OP_LOOP = -1;
constexpr int32_t OP_END = -2;

// Derived per-iteration arrays of the threshold and check kernels, built at
// load time from the trip prefix sums alone (one job each).  Both are
// constant on runs of consecutive entries, one run per row:
//   DERIVE_TSTART  per iteration gs of S, the first iteration of its trip.
//                  Rows: S's parent iterations j; row j covers
//                  [rowptr_S[j], rowptr_S[j+1]) with the value rowptr_S[j]
//                  (path = rowptr offset of S).
//   DERIVE_ANC     per iteration g of a loop `up` levels below S, its
//                  enclosing S-iteration.  Rows: S's iterations j; row j
//                  covers the first iterations below j, [R(j), R(j+1)), R
//                  the trip prefix sums composed from S's child down to the
//                  consumer's loop (path = path pool offset of their rowptr
//                  offsets, innermost first), with the value j.
// After its nrows rows a job has one more, [n, len) with the value 0: the
// padding to a multiple of 4 entries (or, for a barrier-fallback
// dependency, its whole zero-filled array).  Every array starts at a
// multiple of 4 entries, so a 4-pair chunk reads its four entries with one
// int4 load.
enum : int32_t { DERIVE_TSTART = 0, DERIVE_ANC = 1 };
constexpr int kJobTileRows = 32;   // rows per derive tile (one warp's rows)
struct alignas(16) DeriveJob {
  int64_t out;        // derived pool offset of the array
  int64_t row0;       // the job's first row among the rows of all jobs
  int64_t path;
  int64_t len;        // entries reserved (n padded)
  int32_t nrows;
  int32_t n;          // entries of the array proper
  int32_t kind;
  int32_t up;
};

struct ThrArgs {
  const DepInfo* dep;
  const int32_t* derived;
  const int32_t* ord;        // per-engine mode: engine-stream positions (ordinal pool)
  const int64_t* seg;        // [n_deps + 1] segment offsets
  const int32_t* tile_first; // [n_tiles + 1]
  const int64_t* path;
  const int32_t* rowptr;
  int64_t n_chunks;
  int32_t mode;
};

struct CheckArgs {
  ThrArgs t;
  const int32_t* thr;
  unsigned long long* counts;
  unsigned long long* first_bad;
};

// Sec. 6.2's ALU reductions (sync_sim_params.licm / cse), per instruction x:
//   xcse[x] = {waits computed, of those with a reused mask, of those with a
//              cached-sum read (producer loop depth > 1, outer sum not
//              reused), their levels} with CSE;
//   xlvr[x] = waits whose producer loop has depth > 1 (cached-sum reads
//             without CSE);
// per (loop, engine) row: hoist[row] = producer engines whose cached path
// sums the engine updates at each iteration start of the loop (LICM).
struct CostTables {
  const int4* xcse;
  const int32_t* xlvr;
  const int32_t* hoist;
};

// Piece-parallel simulation of a large program whose top-level body is one
// loop L: the program is cut into pieces of consecutive iterations of L,
// simulated on separate warps.  Per piece (built at load time): the
// instances of every instruction before it, and from those the engines'
// instance counts and each waited semaphore's published increments at its
// start.  Per call: a validation that every wait of a piece targets an
// increment the piece itself produces (else the program is simulated whole),
// then barrier scheme: one run per piece from a barrier release at 0 and a
// prefix sum of the piece durations; barrier-free: the piece's end state
// (engine cursors and last retires) is a max-plus linear map of its start
// state, read off by one probe run per state variable (the variable raised
// by kProbe, the others 0), composed piece by piece.  The runs store every
// instance's times, from which a last pass forms the true ones.
constexpr int32_t kProbe = 1 << 30;         // probe offset; split programs' time bound < kProbe

struct alignas(16) PieceInfo {
  int64_t hdelta[kModes];   // probe runs: history entry = semhb + hdelta + probe * probe_hist_len[mode]
  int64_t tl[2];            // compact scratch index of instance o = o + tl[0] (barrier scheme: every
                            // split program) or o + tl[1] (barrier-free: the ones split barrier-free)
  int32_t prog, split;      // program id, its index among the split programs
  int32_t loop, g0, g1;     // iterations [g0, g1) of L (global loop id and iteration indices)
  int32_t pub_off[kModes];  // published increments at the start, per waited semaphore (pool pub)
  int32_t nbase_off;        // engines' instances before the piece (pool pub)
  int32_t pad_;
};

struct alignas(16) SplitProg {
  int64_t cnt_base;         // instances of instruction x before piece j: cnt[cnt_base + j*nx + x]
                            // (j = n_pieces: all of them)
  int32_t prog, first_piece, n_pieces, nx;
  int32_t vdep0, vdep1;     // its waited dependencies in vdep
  int32_t ne, loop;         // engines, L (global id)
  int32_t x0, pad_[3];      // its first instruction (global id)
};

// A waited dependency of a split program, for the validation.
struct alignas(16) VDep {
  int64_t seg;              // its segment in the threshold layout
  int32_t cons;             // consumer (program-local instruction)
  int32_t sem[kModes];      // waited semaphore (program-local), per mode
  int32_t pad_[2];
};

// What the piece kernels (and the ordinary sweep, to skip the programs they
// simulated) read.
struct PieceArgs {
  const PieceInfo* piece;   // [n_pieces]
  const SplitProg* split;   // [n_split]
  const int32_t* prog_split;  // [n_programs]: index among the split programs, -1 if none (NULL: none)
  const int32_t* pub;       // published increments / engine instance counts at piece starts
  int32_t* fail;            // [n_split]: 0 = simulated by pieces in this call
  int32_t* out;             // [n_pieces * out_probes * 64]: end states of the runs (run q of a piece
                            // at 64 * (out_probes * piece + q))
  int32_t* x;               // [n_pieces * 64]: true start states (cursors, then last retires)
  int32_t* phist;           // probe runs' private semaphore history
  int64_t phist_len;        // entries per probe
  int32_t* ptimes;          // stored times of the piece runs (tl_write in sweep.cuh)
  int64_t plen;             // instances of the compact scratch
  const int32_t* xeng;      // engine of every instruction (global id)
  int32_t n_pieces, probes; // this launch: items = n_pieces * probes
  int32_t nx_max;           // most instructions of a split program
  int32_t out_probes;       // end states per piece in out (its stride: 64 * out_probes per piece)
  // barrier-free speculation (split programs with cls 1, too many to probe):
  // a piece runs from a guessed start state xhat; it is accepted when its
  // true start equals xhat plus one shift for every state variable (the
  // times are then the stored ones plus that shift); a rejected piece runs
  // again from its true start, the later ones from guesses of the last round
  int32_t spec;             // 1: this launch runs the speculative pieces
  const int32_t* cls;       // [n_split]: 0 = probed, 1 = speculated (barrier-free)
  int32_t* need;            // [n_pieces]: run in the next round
  int32_t* has;             // [n_pieces]: has run at least once
  int32_t* xhat;            // [n_pieces * 64]: start state of its last run
  int32_t* shift;           // [n_pieces]: accepted pieces: true times - stored times
  int32_t* vp;              // [n_split]: pieces accepted so far
};

struct SimArgs {
  const ProgInfo* prog;
  const int32_t* order;      // program ids in descending-work order
  const int32_t* rowptr;
  const int32_t* op_ptr;     // [rows] first record of each row
  const int2* rowinfo;       // [rows]
  const int4* ops;
  const int32_t* opstop;
  const int4* opsem;         // per-mode records, parallel to ops
  const int64_t* dseg;
  const int32_t* dsem;       // per-mode waited semaphore, parallel to dseg
  const int64_t* semhb;
  const int64_t* inst_off;   // per instruction, instance-layout offset
  const int32_t* thr;
  int32_t* hist;             // scratch: retire time of each semaphore increment
  int32_t* next_slot;        // scratch: next program slot to fetch (zeroed per launch)
  int32_t* makespan;
  unsigned long long* checksum;
  int32_t* status;
  int32_t* issue;
  int32_t* retire;
  sync_sim_params prm;
  int32_t n_programs;
  int32_t mode;
  int32_t warps;             // warps per CTA (largest engine count of the batch)
  int32_t sem_cap;           // semaphore slots in shared memory
  int32_t frame_depth;       // frames per warp
  const int32_t* only;       // if set: [0] count, [1..] the program ids to simulate
  // fused simulation (thresholds from the walk's loop state, no threshold
  // array): dep is set (NULL otherwise) and thr is unused
  const DepInfo* dep;
  const int32_t* ddep;       // per consumer-grouped dependency: its dependency id
  const int64_t* path;
  const int32_t* ord;        // per-engine mode: engine-stream positions
  unsigned long long* chk_counts;  // optional: [2] unsafe / over-synchronised wait values
  unsigned long long* chk_first;   // optional: [1] smallest offending pair index
  CostTables cost;
};

struct SweepArgs {
  const ProgInfo* prog;
  const int32_t* order;
  const LoopInfo* loop;
  const int32_t* rowptr;
  const int32_t* plan_ptr;   // [n_loops + 1]
  const int4* plan;
  const int4* chunk;
  const int4* lrec;
  const int4* lmeta;
  const int4* lsem;          // per-mode records, parallel to lrec
  const int64_t* dseg;
  const int32_t* dsem;       // per-mode, parallel to dseg
  const int64_t* semhb;
  const int64_t* inst_off;
  const int32_t* thr;
  int32_t* hist;
  int32_t* next_slot;        // scratch: program slot counter (zeroed per launch)
  int32_t* fallback;         // scratch: [0] count, [1..] programs for the fallback kernel
  int32_t* makespan;
  unsigned long long* checksum;
  int32_t* status;
  int32_t* issue;
  int32_t* retire;
  sync_sim_params prm;
  int32_t n_programs;
  int32_t mode;
  int32_t sem_cap;
  int32_t frame_depth;
  int32_t ring;              // latest increments kept per semaphore (power of two)
  const int32_t* lflag;      // per loop: 1 if it carries no offset > 0 (trip register elidable)
  const int4* paux;          // per plan item: loop statement {child rowptr offset lo, hi,
                             // chunk of its whole body barrier-free, barrier} (-1: none);
                             // segment: its first chunk's record
  // fused simulation (thresholds from the walk's loop state, no threshold
  // array): dep is set (NULL otherwise) and thr is unused
  const DepInfo* dep;
  const int32_t* ddep;       // per consumer-grouped dependency: its dependency id
  const int64_t* path;
  const int32_t* ord;        // per-engine mode: engine-stream positions
  unsigned long long* chk_counts;  // optional: [2] unsafe / over-synchronised wait values
  unsigned long long* chk_first;   // optional: [1] smallest offending pair index
  CostTables cost;
  PieceArgs pcs;             // piece-parallel simulation (prog_split NULL: none)
};

// Launchers (return the launch error, if any).
// Semaphore records of the op rows and sweep lanes, per threshold mode,
// gathered from the per-instruction table xsem[m * n_instrs + x] by the
// record's global instruction x (LOOP and END op records: {-1, 0, 0, 0}):
// opsem[m * n_ops + r], lsem[m * n_lanes + i].
cudaError_t launch_sem_records(const int4* xsem, int64_t n_instrs, const int4* ops, int64_t n_ops,
                               const int4* lrec, int64_t n_lanes, int4* opsem, int4* lsem, int num_sms,
                               cudaStream_t s);
// tile_job[t] = job holding row t*kJobTileRows (largest i with jobs[i].row0
// <= t*kJobTileRows), with one extra entry n_jobs-1; n_rows = rows of all
// jobs, n = derived pool entries.
cudaError_t launch_derive(const DeriveJob* jobs, const int32_t* tile_job, int64_t n_rows, const int32_t* rowptr,
                          const int64_t* path, int32_t* derived, int64_t n, int num_sms, cudaStream_t s);
// Per-engine allocation (Sec. 6.1): ord[ord_off[x] + g] = 1-based position of
// instruction x's instance at global iteration g of its loop in its engine's
// dynamic stream, for every x with ord_off[x] >= 0; one thread per (program,
// engine) walks that engine's op rows in program order.
cudaError_t launch_ordinals(const ProgInfo* prog, const int32_t* order, int32_t n_programs, int32_t ne_max,
                            const int32_t* op_ptr, const int4* ops, const int32_t* rowptr,
                            const int64_t* ord_off, int32_t* ord, int num_sms, cudaStream_t s);
cudaError_t launch_thresholds(const ThrArgs& a, int32_t* thr, int num_sms, cudaStream_t s);
cudaError_t launch_check(const CheckArgs& a, int num_sms, cudaStream_t s);
cudaError_t launch_simulate(const SimArgs& a, bool barrier, int num_sms, cudaStream_t s);
// The sweep simulates every program it can; programs whose waits reach
// forward in program order are listed in a.fallback and then simulated by
// the per-engine kernel (launch_simulate with SimArgs::only set).
cudaError_t launch_sweep(const SweepArgs& a, bool barrier, int num_sms, cudaStream_t s);
size_t sweep_smem_bytes(int sem_cap, int frame_depth, int ring);
// Piece-parallel simulation of the split programs (a.pcs): validation, the
// probe (barrier-free) or relative (barrier) runs, the composition of the
// pieces, and the pass that forms the instances' true times (checksums,
// timelines); the programs it completes are marked in a.pcs.fail (0) for
// launch_sweep to skip.
struct PieceLaunch {
  const VDep* vdep;
  const int32_t* cnt;
  int32_t* one;              // stored times of single runs (barrier scheme, speculation)
  int64_t one_len;           // instances of all split programs
  int32_t n_split, n_probed, n_spec;   // split programs; of these barrier-free probed / speculated
};
cudaError_t launch_pieces(const SweepArgs& a, bool barrier, const PieceLaunch& L, int num_sms, cudaStream_t s);
// Largest ring (32, 16, ..., 1) whose sweep shared memory fits in `limit`
// bytes, or 0 if none does.
int sweep_ring_for(int sem_cap, int frame_depth, size_t limit);
size_t simulate_smem_bytes(int warps, int sem_cap, int frame_depth);

// Kernels this library has launched in this process (every handle and
// stream), counted by launched() after each launch the runtime accepted.
void count_launch();
inline cudaError_t launched() {
  const cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) count_launch();
  return e;
}

}  // namespace syncgb
