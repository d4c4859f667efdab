// sync_simulate_noalloc: the schedule simulation without device allocation.
//
// For callers that cannot call cudaMalloc / cudaFree around a simulation,
// the scratch the simulator needs (semaphore history, program-slot counter,
// fallback list) comes from one array declared statically in device memory
// here instead of from the handle.  A GPU holds the array from the moment the
// library's module is loaded on it until the process exits; with CUDA's lazy
// module loading that is the first call on that device (the address lookup
// below loads it).  The array's device address is looked up on every call,
// with the call's device current, so a re-created context (after
// cudaDeviceReset) never sees a stale address.  All calls share the array
// and it keeps the last call's contents: the counters the kernels start from
// are zeroed on the caller's stream by every call, the history is written
// before it is read, and calls whose work overlaps on the GPU race with each
// other.
#include <algorithm>
#include <cstring>
#include <string>

#include "handle.h"

namespace {

constexpr size_t kScratchInts = SYNC_NOALLOC_SCRATCH_BYTES / sizeof(int32_t);

// [0] program-slot counter, [1] fallback count, [2 .. 2+P) fallback list,
// then (at a 256-byte boundary) the semaphore history.
static __device__ __align__(256) int32_t g_scratch[kScratchInts];

// Device address of g_scratch in the current context (looked up each call:
// cheap once the module is loaded, and never stale after a context reset).
cudaError_t scratch_address(int32_t** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
  if (e != cudaSuccess) return e;
  *out = static_cast<int32_t*>(p);
  return cudaSuccess;
}

sync_status cuda_error(cudaError_t e, const char* what) {
  if (e == cudaSuccess) return SYNC_OK;
  return syncgb::set_error(SYNC_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

}  // namespace

extern "C" sync_status sync_simulate_noalloc(const sync_programs* h, sync_thr_mode mode, const int32_t* d_thr,
                                             const sync_sim_params* params, sync_sim_variant variant,
                                             int32_t* d_makespan, unsigned long long* d_checksum,
                                             int32_t* d_status, int32_t* d_issue, int32_t* d_retire,
                                             void* stream) {
  using namespace syncgb;
  if (!h || !params) return set_error(SYNC_ERR_ARG, "handle and params must not be NULL");
  if (mode != SYNC_THR_COUNT && mode != SYNC_THR_PERLOOP && mode != SYNC_THR_PERENGINE)
    return set_error(SYNC_ERR_ARG, "unknown threshold mode");
  if (variant != SYNC_SIM_BARRIER_FREE && variant != SYNC_SIM_BARRIER && variant != SYNC_SIM_UNROLLED)
    return set_error(SYNC_ERR_ARG, "unknown variant");
  if (variant == SYNC_SIM_UNROLLED && mode != SYNC_THR_PERENGINE)
    return set_error(SYNC_ERR_ARG, "the unrolled variant takes per-engine thresholds");
  if (variant == SYNC_SIM_UNROLLED && h->n_bar_deps > 0)
    return set_error(SYNC_ERR_ARG, "the unrolled variant takes no barrier-fallback dependencies");
  if (h->divergent && (mode == SYNC_THR_PERENGINE || variant != SYNC_SIM_BARRIER_FREE))
    return set_error(SYNC_ERR_ARG, "per-engine trip counts: barrier-free count or per-loop simulation only");
  if (h->sz.n_programs > 0 && (!d_makespan || !d_checksum || !d_status))
    return set_error(SYNC_ERR_ARG, "per-program outputs must not be NULL");
  if (h->sz.n_pairs_padded > 0 && !d_thr) return set_error(SYNC_ERR_ARG, "d_thr must not be NULL");
  if ((d_issue == nullptr) != (d_retire == nullptr))
    return set_error(SYNC_ERR_ARG, "d_issue and d_retire: both or neither");
  sync_sim_params q;
  if (!sim_params_for(*params, variant, q)) return set_error(SYNC_ERR_ARG, "timing constants must be >= 0");
  // the scratch must hold two counters, the fallback list and the history
  const int64_t list_ints = ((2 + (int64_t)h->sz.n_programs) + 63) & ~int64_t(63);
  const int64_t need = list_ints + h->hist_len[mode];
  if (need > (int64_t)kScratchInts)
    return set_error(SYNC_ERR_ARG, "batch needs " + std::to_string(need * 4) + " bytes of simulator scratch; "
                                   "sync_simulate_noalloc has " + std::to_string(kScratchInts * 4) +
                                   " (use sync_simulate)");
  const int32_t sem_cap = std::max(4, (h->nsem_max[mode] + 3) & ~3);
  const int32_t frame_depth = std::max(1, h->depth_max);
  const int ring = sweep_ring_for(sem_cap, frame_depth, 200 * 1024);
  if (simulate_smem_bytes(h->ne_max, sem_cap, frame_depth) > 200 * 1024 || ring == 0)
    return set_error(SYNC_ERR_ARG, "a program has too many waited semaphores for the simulator's shared memory");
  sync_status st = cuda_error(cudaSetDevice(h->device), "cudaSetDevice");
  if (st != SYNC_OK) return st;
  st = cuda_error(h->wait_ready(static_cast<cudaStream_t>(stream)), "load completion");
  if (st != SYNC_OK) return st;
  int32_t* base = nullptr;
  st = cuda_error(scratch_address(&base), "cudaGetSymbolAddress");
  if (st != SYNC_OK) return st;

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const bool barrier = variant == SYNC_SIM_BARRIER;
  SweepArgs w;
  std::memset(&w, 0, sizeof w);
  w.prog = h->prog; w.order = h->order; w.loop = h->loop; w.rowptr = h->rowptr;
  w.plan_ptr = h->plan_ptr; w.plan = h->plan; w.chunk = h->chunk;
  w.lrec = h->lrec; w.lmeta = h->lmeta; w.lsem = h->lsem + (size_t)mode * h->n_lanes;
  w.dseg = h->dseg; w.dsem = h->dsem + (size_t)mode * h->sz.n_deps; w.semhb = h->semhb;
  w.inst_off = h->inst_off; w.thr = d_thr;
  w.hist = base + list_ints; w.next_slot = base; w.fallback = base + 1;
  w.makespan = d_makespan; w.checksum = d_checksum; w.status = d_status;
  w.issue = d_issue; w.retire = d_retire;
  w.prm = q; w.n_programs = h->sz.n_programs; w.mode = mode;
  w.sem_cap = sem_cap; w.frame_depth = frame_depth; w.ring = ring; w.lflag = h->lflag; w.paux = h->paux;
  w.cost = h->cost;
  st = cuda_error(launch_sweep(w, barrier, h->num_sms, s), "sweep simulator kernel");
  if (st != SYNC_OK) return st;
  SimArgs a;
  std::memset(&a, 0, sizeof a);
  a.prog = h->prog; a.order = h->order; a.rowptr = h->rowptr;
  a.op_ptr = h->op_ptr; a.rowinfo = h->rowinfo; a.ops = h->ops; a.opstop = h->opstop;
  a.opsem = h->opsem + (size_t)mode * h->n_ops;
  a.dseg = h->dseg; a.dsem = h->dsem + (size_t)mode * h->sz.n_deps;
  a.semhb = h->semhb; a.inst_off = h->inst_off;
  a.thr = d_thr; a.hist = base + list_ints; a.next_slot = base; a.only = base + 1;
  a.makespan = d_makespan; a.checksum = d_checksum; a.status = d_status;
  a.issue = d_issue; a.retire = d_retire;
  a.prm = q; a.n_programs = h->sz.n_programs; a.mode = mode;
  a.sem_cap = sem_cap; a.frame_depth = frame_depth; a.warps = h->ne_max;
  a.cost = h->cost;
  return cuda_error(launch_simulate(a, barrier, h->num_sms, s), "per-engine simulator kernel");
}
