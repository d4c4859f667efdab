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

enum : int32_t { CASE_PS = 0, CASE_NEST_FWD = 1, CASE_NEST_BWD = 2 };

// Pairs are processed in chunks of 4 consecutive entries (one int4).  A tile
// is the span one 256-thread CTA covers in one pass.
constexpr int kChunk = 4;
constexpr int kTilePairs = 1024;

// Per loop.  rowptr_l[j], j in [0, total(parent)], is the number of l's
// iterations that start before the parent's global iteration j (exclusive
// prefix sum of the trips); pidx_l[g] is the parent's global iteration during
// l's global iteration g.  The top-level loop has rowptr [0, 1], pidx [0].
struct alignas(16) LoopInfo {
  int64_t rowptr_off;
  int64_t pidx_off;
  int32_t parent;     // -1 for a top-level loop
  int32_t total;      // global iterations
  int32_t n_parent;   // total(parent), 1 for a top-level loop
  int32_t depth;
};

// Per dependency.  `path` points into the int64 path pool:
//   [0, up)            pidx offsets of the loops from the consumer's loop up
//                      to (excluding) S, innermost first;
//   up, up+1           pidx offset and rowptr offset of S;
//   [up+2, up+2+clen)  rowptr offsets of the loops from S's child down to P
//                      (nested cases; clen = 0 when P = S).
struct alignas(16) DepInfo {
  int64_t seg_off;    // pair-layout offset of this dependency's segment
  int64_t path;
  int32_t total;      // consumer instances (= total of the consumer's loop)
  int32_t up;
  int32_t clen;
  int32_t kase;
  int32_t k, N, K, pad_;
};

// Per program, for the simulator.
struct alignas(16) ProgInfo {
  int64_t agg_lat;    // sum over instructions of instances * latency (saturated)
  int64_t n_inst;     // datapath instances
  int64_t n_pairs;    // (dependency, consumer instance) pairs
  int64_t n_stmt;     // loop statements reached (sum over non-top loops of total(parent))
  int64_t n_iter;     // loop iterations (sum over non-top loops of total)
  int32_t loop_base;  // global id of the program's top-level loop
  int32_t ne;
  int32_t le_base;    // index of (top-level loop, engine 0) in op_ptr
  int32_t nsem[2];    // waited semaphores, per threshold mode
  int32_t depth;      // deepest nesting level
};

// Per instruction, for the simulator.  Semaphore fields per threshold mode
// (0 = per instruction, 1 = per (loop, engine)); own_sem -1 when nothing
// waits on that semaphore (no history kept).
struct alignas(16) InstrSim {
  int64_t hbase[2];   // history slot of this instruction's increment in g = 0
  int64_t inst_off;   // instance-layout offset
  int32_t own_sem[2];
  int32_t hstride[2]; // history slots between consecutive iterations
  int32_t lat;
  int32_t ndeps;      // dependencies consumed
  int32_t dep_begin;  // first entry in the consumer-grouped dependency list
  int32_t pad_;
};

// Per (consumer, dependency), grouped by consumer.
struct alignas(16) ConsDep {
  int64_t seg_off;    // pair-layout offset of the dependency's segment
  int64_t thist[2];   // history base of the waited semaphore
  int32_t tsem[2];    // local id of the waited semaphore
};

struct ThrArgs {
  const DepInfo* dep;
  const int64_t* seg;        // [n_deps + 1] segment offsets
  const int32_t* tile_first; // [n_tiles + 1]
  const int64_t* path;
  const int32_t* rowptr;
  const int32_t* pidx;
  int64_t n_chunks;
  int32_t mode;
};

struct CheckArgs {
  ThrArgs t;
  const int32_t* thr;
  unsigned long long* counts;
  unsigned long long* first_bad;
};

struct SimArgs {
  const ProgInfo* prog;
  const int32_t* order;      // program slots in descending-work order
  const LoopInfo* loop;
  const int32_t* rowptr;
  const int32_t* op_ptr;
  const int32_t* ops;        // x >= 0 own instruction, -(m+1) child loop m
  const InstrSim* instr;
  const ConsDep* cdep;
  const int32_t* thr;
  int32_t* hist;
  int32_t* makespan;
  unsigned long long* checksum;
  int32_t* status;
  int32_t* issue;
  int32_t* retire;
  sync_sim_params prm;
  int32_t n_programs;
  int32_t mode;
  int32_t sem_ints;          // shared-memory ints for semaphore values per warp
  int32_t frame_depth;       // frames per lane
  int32_t ne_max;
};

// Launchers (return the launch error, if any).
// tile_loop[t] = loop whose pidx segment holds entry t*kTilePairs (largest l
// with pidx_off[l] <= t*kTilePairs), with one extra entry n_loops-1.
cudaError_t launch_expand(const LoopInfo* loop, const int32_t* tile_loop, const int32_t* rowptr,
                          int32_t* pidx, int64_t n_iters, int num_sms, cudaStream_t s);
cudaError_t launch_thresholds(const ThrArgs& a, int32_t* thr, int num_sms, cudaStream_t s);
cudaError_t launch_check(const CheckArgs& a, int num_sms, cudaStream_t s);
cudaError_t launch_simulate(const SimArgs& a, bool barrier, int num_sms, cudaStream_t s);
size_t simulate_smem_per_warp(int sem_ints, int frame_depth, int ne_max);

}  // namespace syncgb
