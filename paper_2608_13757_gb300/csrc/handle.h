// The handle behind sync_programs (internal to the library).
#pragma once

#include <mutex>
#include <string>
#include <vector>

#include "enc.h"

namespace syncgb {
// Host arrays that are filled right after allocation: default-initialised,
// so allocating one does not write it first.
template <class T>
struct NoInit : std::allocator<T> {
  template <class U>
  struct rebind { using other = NoInit<U>; };
  NoInit() = default;
  template <class U>
  NoInit(const NoInit<U>&) {}
  template <class U>
  void construct(U* p) { ::new (static_cast<void*>(p)) U; }
  template <class U, class... A>
  void construct(U* p, A&&... a) { ::new (static_cast<void*>(p)) U(std::forward<A>(a)...); }
};
template <class T>
using HostVec = std::vector<T, NoInit<T>>;

// Throws the loader's failure for a CUDA error (caught at the C ABI).
void cuda_or_raise(cudaError_t e, const char* what);
// Sets the message sync_last_error() returns on this thread; returns status.
sync_status set_error(sync_status status, const std::string& msg);
// The timing constants the simulation kernels take: false if any is
// negative; for the unrolled variant (the straight-line program) the
// loop-control and wait-value costs are 0.
bool sim_params_for(const sync_sim_params& p, sync_sim_variant variant, sync_sim_params& q);
}  // namespace syncgb

struct sync_programs {
  int device = 0;
  int num_sms = 0;
  sync_sizes sz{};
  // pair layout for sync_pair_offsets, read back on first use
  mutable std::mutex pair_mu;
  mutable bool pairs_ready = false;
  mutable syncgb::HostVec<int64_t> seg_host;
  mutable syncgb::HostVec<int32_t> count_host;
  int32_t* dep_count = nullptr;     // pairs per dependency
  std::vector<void*> blocks;
  // threshold / checker encoding
  syncgb::LoopInfo* loop = nullptr;
  int32_t* rowptr = nullptr;
  syncgb::DepInfo* dep = nullptr;
  int32_t* ddep = nullptr;          // per consumer-grouped dependency: dependency id
  int32_t* lflag = nullptr;         // per loop: trip register elidable
  int4* paux = nullptr;             // per sweep plan item: loop-statement side record
  int64_t* seg = nullptr;
  int32_t* tile_first = nullptr;
  int64_t* path = nullptr;
  int32_t* derived = nullptr;       // per-iteration trip starts and S-ancestors
  // per-engine mode, derived on first use: engine-stream positions of the
  // waited producers' instances
  mutable std::mutex ord_mu;
  mutable int32_t* ord = nullptr;
  mutable bool ord_ready = false;
  bool divergent = false;           // some program runs per-engine trip counts
  int64_t n_bar_deps = 0;           // barrier-fallback dependencies (no unrolled variant)
  int64_t n_ord = 0;
  bool ord_overflow = false;        // an engine of a program has > INT32_MAX instances
  int64_t* ord_off = nullptr;       // per instruction: ordinal pool offset of a waited producer, or -1
  int64_t n_chunks = 0;
  // simulator encoding
  syncgb::ProgInfo* prog = nullptr;
  int32_t* order = nullptr;
  int32_t* op_ptr = nullptr;
  int2* rowinfo = nullptr;
  syncgb::CostTables cost{};        // Sec. 6.2 reductions: per-instruction and per-row counts
  int4* ops = nullptr;
  int32_t* opstop = nullptr;
  int4* opsem = nullptr;            // [kModes][n_ops]
  int64_t* dseg = nullptr;
  int32_t* dsem = nullptr;          // [kModes][n_deps]
  int64_t* semhb = nullptr;
  int64_t* inst_off = nullptr;
  int64_t n_ops = 0;
  int32_t* hist = nullptr;          // scratch: retire time of each semaphore increment
  int32_t* next_slot = nullptr;     // scratch: simulator's program-slot counter
  int32_t* fallback = nullptr;      // scratch: programs handed to the per-engine kernel
  // program-order sweep
  int32_t* plan_ptr = nullptr;
  int4* plan = nullptr;
  int4* chunk = nullptr;
  int4* lrec = nullptr;
  int4* lmeta = nullptr;
  int4* lsem = nullptr;             // [kModes][n_lanes]
  int64_t n_lanes = 0;
  int64_t hist_len[syncgb::kModes] = {0, 0, 0};  // history entries needed per threshold mode
  // piece-parallel simulation of large programs (PieceArgs in enc.h)
  int32_t n_split = 0, n_pieces = 0, probes_bf = 0;
  syncgb::PieceInfo* pieces = nullptr;
  syncgb::SplitProg* splits = nullptr;
  int32_t* prog_split = nullptr;        // per program: its index among the split programs, or -1
  int32_t* piece_pub = nullptr;         // published increments / engine instance counts at piece starts
  int32_t* piece_cnt = nullptr;         // instances of each instruction before each piece
  syncgb::VDep* vdep = nullptr;
  int32_t* piece_fail = nullptr;        // scratch [n_split]
  int32_t* piece_cls = nullptr;         // [n_split]: barrier-free, 0 = probed, 1 = speculated
  int32_t n_probed = 0, n_spec = 0;     // split programs of each class
  int32_t* spec_need = nullptr;         // speculation scratch (PieceArgs)
  int32_t* spec_has = nullptr;
  int32_t* spec_xhat = nullptr;
  int32_t* spec_vp = nullptr;
  int32_t* piece_shift = nullptr;
  int32_t* piece_out = nullptr;         // scratch: probe end states
  int32_t* piece_x = nullptr;           // scratch: start states
  int64_t phist_len[syncgb::kModes] = {0, 0, 0};   // probe history entries per probe, per mode
  mutable std::mutex phist_mu;
  mutable int32_t* phist[syncgb::kModes] = {nullptr, nullptr, nullptr};   // allocated on first use
  int64_t pinst[2] = {0, 0};            // instances of the split programs (barrier scheme, barrier-free)
  mutable int32_t* ptimes[2] = {nullptr, nullptr};   // their stored times, allocated on first use
  int32_t* xeng = nullptr;              // engine per instruction (split batches)
  int32_t nx_max_split = 1;             // most instructions of a split program
  int32_t nsem_max[syncgb::kModes] = {0, 0, 0};
  int32_t ne_max = 1;
  int32_t depth_max = 0;
  // recorded on the load's stream after its last operation; every call on
  // the handle makes its own stream wait for it
  cudaEvent_t ready = nullptr;

  cudaError_t wait_ready(cudaStream_t s) const { return ready ? cudaStreamWaitEvent(s, ready, 0) : cudaSuccess; }

  ~sync_programs() {
    if (blocks.empty()) return;
    int prev = 0;
    cudaGetDevice(&prev);
    cudaSetDevice(device);
    cudaDeviceSynchronize();
    if (ready) cudaEventDestroy(ready);
    for (void* p : blocks) cudaFree(p);
    cudaSetDevice(prev);
  }

  template <class V, class T = typename V::value_type>
  T* upload(const V& v, cudaStream_t s, const char* what) {
    const size_t bytes = std::max<size_t>(v.size(), 1) * sizeof(T);
    void* p = nullptr;
    syncgb::cuda_or_raise(cudaMalloc(&p, bytes), what);
    blocks.push_back(p);
    sz.device_bytes += (int64_t)bytes;
    if (!v.empty()) syncgb::cuda_or_raise(cudaMemcpyAsync(p, v.data(), v.size() * sizeof(T), cudaMemcpyHostToDevice, s), what);
    sz.h2d_bytes += (int64_t)(v.size() * sizeof(T));
    return static_cast<T*>(p);
  }
  // device memory the handle frees (mutable: lazily derived tables)
  template <class T>
  T* alloc_lazy(int64_t n, const char* what) const {
    return const_cast<sync_programs*>(this)->alloc<T>(n, what);
  }
  template <class T>
  T* alloc(int64_t n, const char* what) {
    const size_t bytes = (size_t)std::max<int64_t>(n, 1) * sizeof(T);
    void* p = nullptr;
    syncgb::cuda_or_raise(cudaMalloc(&p, bytes), what);
    blocks.push_back(p);
    sz.device_bytes += (int64_t)bytes;
    return static_cast<T*>(p);
  }
};

