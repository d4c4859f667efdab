// C ABI of the engine: host loader (validation, dependency classification,
// device encoding) and the launch wrappers.  Declarations and contracts are
// in include/sync.h.
#include <algorithm>
#include <array>
#include <atomic>
#include <cstdlib>
#include <cstring>
#include <exception>
#include <memory>
#include <mutex>
#include <new>
#include <string>
#include <thread>
#include <unordered_map>
#include <utility>
#include <vector>

#include "enc.h"
#include "handle.h"
#include "progbuild.cuh"

using namespace syncgb;

namespace {

thread_local std::string g_err;

struct Failure {
  sync_status status;
  std::string msg;
};

[[noreturn]] void raise(sync_status s, std::string msg) { throw Failure{s, std::move(msg)}; }

void cuda_check(cudaError_t e, const char* what) {
  if (e == cudaSuccess) return;
  if (e == cudaErrorMemoryAllocation) {
    cudaGetLastError();
    raise(SYNC_ERR_OOM, std::string(what) + ": " + cudaGetErrorString(e));
  }
  raise(SYNC_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

sync_status report(const Failure& f) {
  g_err = f.msg;
  return f.status;
}

}  // namespace

namespace syncgb {
sync_status set_error(sync_status status, const std::string& msg) {
  g_err = msg;
  return status;
}
void cuda_or_raise(cudaError_t e, const char* what) { cuda_check(e, what); }

std::atomic<int64_t> g_launches{0};
void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

// Timing constants a variant runs with: the unrolled variant has no loop
// control and static waits, so it costs neither.
bool sim_params_for(const sync_sim_params& p, sync_sim_variant variant, sync_sim_params& q) {
  if (p.ii < 0 || p.c_branch < 0 || p.c_regop < 0 || p.c_wait_ops_count < 0 || p.c_wait_ops_perloop < 0 ||
      p.c_barrier < 0 || p.c_wait_ops_perengine_level < 0)
    return false;
  q = p;
  if (variant == SYNC_SIM_UNROLLED) {
    q.c_branch = q.c_regop = 0;
    q.c_wait_ops_count = q.c_wait_ops_perloop = q.c_wait_ops_perengine_level = 0;
    q.licm = q.cse = 0;
  }
  return true;
}
}  // namespace syncgb

namespace {

// Threads of the host validation pass: one per hardware thread (at most 32)
// while each gets at least 256 programs.  SYNCGB_LOAD_THREADS=n sets the count.
int load_threads(int32_t P) {
  int n = 0;
  if (const char* v = std::getenv("SYNCGB_LOAD_THREADS")) n = std::atoi(v);
  if (n <= 0) {
    n = std::min(32, (int)std::max(1u, std::thread::hardware_concurrency()));
    n = (int)std::min<int64_t>(n, std::max<int64_t>(1, P / 256));
  }
  return std::max(1, std::min(n, std::max(1, (int)P)));
}

void check_csr(const int32_t* ptr, int32_t P, const char* name) {
  if (ptr[0] != 0) raise(SYNC_ERR_MALFORMED, std::string(name) + "[0] must be 0");
  for (int32_t p = 0; p < P; ++p)
    if (ptr[p + 1] < ptr[p]) raise(SYNC_ERR_MALFORMED, std::string(name) + " is not nondecreasing");
}

std::string where(int32_t p, const char* what, int64_t i) {
  return "program " + std::to_string(p) + ", " + what + " " + std::to_string(i);
}

// Status and text of each failure of the per-program pass (progbuild.cuh).
struct BuildErrorText {
  sync_status status;
  const char* what;
  bool located;              // reported as "program p, <what> <index>"
};
const BuildErrorText kBuildErrorText[kBuildErrors] = {
    {SYNC_OK, "", false},
    {SYNC_ERR_MALFORMED, "has no top-level loop", true},
    {SYNC_ERR_MALFORMED, "n_engines", true},
    {SYNC_ERR_MALFORMED, "loop 0 must have parent -1, loop", true},
    {SYNC_ERR_MALFORMED, "parent must precede the loop, loop", true},
    {SYNC_ERR_MALFORMED, "negative position, loop", true},
    {SYNC_ERR_MALFORMED, "nesting deeper than SYNC_MAX_DEPTH, loop", true},
    {SYNC_ERR_MALFORMED, "negative trip count, loop", true},
    {SYNC_ERR_MALFORMED, "top-level loop must run once, loop", true},
    {SYNC_ERR_OVERFLOW, "iterations exceed INT32_MAX, loop", true},
    {SYNC_ERR_MALFORMED, "trip count array length != parent's iterations, loop", true},
    {SYNC_ERR_MALFORMED, "per-engine trip row length != parent's iterations on the engine, loop", true},
    {SYNC_ERR_ARG, "eng_trips must not be NULL", false},
    {SYNC_ERR_MALFORMED, "loop out of range, instruction", true},
    {SYNC_ERR_MALFORMED, "negative position, instruction", true},
    {SYNC_ERR_MALFORMED, "engine out of range, instruction", true},
    {SYNC_ERR_MALFORMED, "latency < 1, instruction", true},
    {SYNC_ERR_MALFORMED, "two items share a position in the body of loop", true},
    {SYNC_ERR_MALFORMED, "instruction out of range, dependency", true},
    {SYNC_ERR_MALFORMED, "negative offset, dependency", true},
    {SYNC_ERR_NOT_ALLOCATABLE, "offset 0 to a later producer on the same engine, dependency", true},
    {SYNC_ERR_NOT_ALLOCATABLE, "nested forward producer needs offset 0, dependency", true},
    {SYNC_ERR_NOT_ALLOCATABLE, "nested backward producer needs offset 1, dependency", true},
    {SYNC_ERR_ARG, "barrier fallback with per-engine trip counts, dependency", true},
    {SYNC_ERR_OVERFLOW, "per-loop semaphore value N*iterations exceeds INT32_MAX, dependency", true},
};

[[noreturn]] void raise_build_error(int32_t p, int32_t kind, int64_t index) {
  if (kind <= BE_NONE || kind >= kBuildErrors) raise(SYNC_ERR_ARG, "unexpected loader failure");
  const BuildErrorText& t = kBuildErrorText[kind];
  raise(t.status, t.located ? where(p, t.what, index) : std::string(t.what));
}

// The batch's shape (everything the per-program pass relies on to stay in
// bounds) and its (loop, engine) rows.  With per-engine trips the rows index
// the caller's eng_trip_ptr, so the passes stop before the first program
// whose engine count is out of range (`covered`); that program's own failure
// is reported if none before it fails.
struct Shape {
  int32_t P = 0, covered = 0;
  int64_t NL = 0, NX = 0, ND = 0, rows = 0;
  bool div = false;
  std::vector<int64_t> row_base;
};

Shape shape_checks(const sync_batch_desc& d) {
  Shape s;
  if (d.n_programs < 0) raise(SYNC_ERR_ARG, "n_programs < 0");
  if (d.nonalloc_policy != SYNC_NONALLOC_REJECT && d.nonalloc_policy != SYNC_NONALLOC_BARRIER)
    raise(SYNC_ERR_ARG, "nonalloc_policy is not a sync_nonalloc_policy");
  const int32_t P = s.P = d.n_programs;
  if (!d.prog_loop_ptr || !d.prog_instr_ptr || !d.prog_dep_ptr || (P > 0 && !d.prog_n_engines))
    raise(SYNC_ERR_ARG, "program CSR arrays must not be NULL");
  check_csr(d.prog_loop_ptr, P, "prog_loop_ptr");
  check_csr(d.prog_instr_ptr, P, "prog_instr_ptr");
  check_csr(d.prog_dep_ptr, P, "prog_dep_ptr");
  s.NL = d.prog_loop_ptr[P];
  s.NX = d.prog_instr_ptr[P];
  s.ND = d.prog_dep_ptr[P];
  s.div = d.eng_trip_ptr != nullptr;
  if (s.NL > 0 && (!d.loop_parent || !d.loop_pos || (!s.div && !d.trip_ptr)))
    raise(SYNC_ERR_ARG, "loop arrays must not be NULL");
  if (s.NX > 0 && (!d.instr_loop || !d.instr_pos || !d.instr_engine || !d.instr_latency))
    raise(SYNC_ERR_ARG, "instruction arrays must not be NULL");
  if (s.ND > 0 && (!d.dep_prod || !d.dep_cons || !d.dep_k))
    raise(SYNC_ERR_ARG, "dependency arrays must not be NULL");
  if (s.div && d.eng_trip_ptr[0] != 0) raise(SYNC_ERR_MALFORMED, "eng_trip_ptr[0] must be 0");
  if (s.NL > 0 && !s.div) {
    if (d.trip_ptr[0] != 0) raise(SYNC_ERR_MALFORMED, "trip_ptr[0] must be 0");
    for (int64_t l = 0; l < s.NL; ++l)
      if (d.trip_ptr[l + 1] < d.trip_ptr[l]) raise(SYNC_ERR_MALFORMED, "trip_ptr is not nondecreasing");
    if (d.trip_ptr[s.NL] > 0 && !d.trips) raise(SYNC_ERR_ARG, "trips must not be NULL");
  }
  s.row_base.assign(P + 1, 0);
  s.covered = P;
  for (int32_t p = 0; p < P; ++p) {
    const int64_t nl = d.prog_loop_ptr[p + 1] - d.prog_loop_ptr[p];
    const int32_t ne = d.prog_n_engines[p];
    const bool ok = ne >= 1 && ne <= 32;
    if (!ok && s.div && s.covered == P) s.covered = p;
    s.row_base[p + 1] = s.row_base[p] + (ok ? nl * ne : 0);
  }
  s.rows = s.row_base[P];
  if (s.div) {
    const int64_t R = s.row_base[s.covered];
    for (int64_t r = 0; r < R; ++r)
      if (d.eng_trip_ptr[r + 1] < d.eng_trip_ptr[r]) raise(SYNC_ERR_MALFORMED, "eng_trip_ptr is not nondecreasing");
  }
  return s;
}

// Programs past the covered ones: the first uncovered program's failure.
void check_uncovered(const sync_batch_desc& d, const Shape& s) {
  if (s.covered == s.P) return;
  const int32_t p = s.covered;
  if (d.prog_loop_ptr[p + 1] - d.prog_loop_ptr[p] < 1) raise_build_error(p, BE_NO_TOP, 0);
  raise_build_error(p, BE_ENGINES, d.prog_n_engines[p]);
}

// Totals that index 32-bit fields of the encoding.
void check_totals(const int64_t* count) {
  if (count[BC_OPS] > kI32Max) raise(SYNC_ERR_OVERFLOW, "op records exceed INT32_MAX entries");
  if (count[BC_PLAN] > kI32Max || count[BC_CHUNKS] > kI32Max || count[BC_LANES] > kI32Max)
    raise(SYNC_ERR_OVERFLOW, "sweep tables exceed INT32_MAX entries");
}

}  // namespace

// Fewest instances of a program cut into pieces: 65536 (SYNCGB_SPLIT_MIN=n
// sets another floor; tests lower it).
static int64_t split_floor() {
  int64_t min_inst = 65536;
  if (const char* e = std::getenv("SYNCGB_SPLIT_MIN")) min_inst = std::max<int64_t>(1, std::atoll(e));
  return min_inst;
}

// Piece-parallel simulation (PieceArgs in enc.h): which programs are split,
// into which pieces, and what each piece starts from.  A program qualifies
// when its top-level body is one loop L (no instruction of its own), its
// engines share their trips and it has no fallback barriers, L runs at least
// twice, and it is large against the batch: at least 65536 instances (the
// environment variable SYNCGB_SPLIT_MIN sets another floor) and
// more than 8 times the instances per resident sweep warp (152 SMs x 24
// warps on a GB300) of the whole batch, so that its serial walk, not the
// batch's throughput, bounds the simulation (the barrier scheme runs each
// piece twice).  Barrier-free, a program is probed (2*ne runs per piece)
// when it stays above 4 * (2*ne + 1) times that share, and speculated
// otherwise (SYNCGB_SPLIT_SPEC=1 speculates always).
static void build_pieces(const sync_batch_desc& d, const LoopInfo* loop, const int32_t* rowptr, const int4* xsem,
                         const DepInfo* dep, const int64_t* seg, const int64_t* semhb, const ProgInfo* prog,
                         const int64_t* inst_off, int64_t n_inst, cudaStream_t stream, sync_programs& h) {
  const int32_t P = d.n_programs;
  const int64_t NX = d.prog_instr_ptr[P];
  const double share = (double)n_inst / ((double)h.num_sms * 24.0);
  const int64_t min_inst = split_floor();
  const char* spec_env = std::getenv("SYNCGB_SPLIT_SPEC");   // 1: speculate, never probe (tests)
  const bool force_spec = spec_env && spec_env[0] == '1';
  std::vector<int32_t> split_of(P, -1);
  std::vector<SplitProg> splits;
  std::vector<PieceInfo> pieces;
  std::vector<VDep> vdep;
  std::vector<int32_t> pub, cnt, bf_init;
  int64_t hist_split[kModes] = {0, 0, 0};
  int64_t inst_bb = 0, inst_bf = 0;               // compact instance spaces (barrier scheme, barrier-free)
  int32_t ne_max = 0;
  std::vector<int32_t> path, row;
  for (int32_t p = 0; p < P; ++p) {
    const ProgInfo& pi = prog[p];
    if (pi.divergent || pi.fb_iters > 0 || pi.n_inst < min_inst || (double)pi.n_inst <= 8.0 * share) continue;
    const int32_t l0 = d.prog_loop_ptr[p], nl = d.prog_loop_ptr[p + 1] - l0;
    const int32_t x0 = d.prog_instr_ptr[p], nx = d.prog_instr_ptr[p + 1] - x0;
    int32_t L = -1, children = 0;
    bool own = false;
    for (int32_t l = 1; l < nl; ++l)
      if (d.loop_parent[l0 + l] == 0) { ++children; L = l; }
    for (int32_t x = 0; x < nx; ++x) own = own || d.instr_loop[x0 + x] == 0;
    if (children != 1 || own) continue;
    const int32_t T = loop[l0 + L].total;
    if (T < 2) continue;
    // instances of instruction x before iteration g of L: L's iterations
    // 0..g-1 hold, for a loop m below L, the iterations of m that start
    // before them -- the trip prefix sums composed from L's child down to m
    auto count = [&](int32_t x, int32_t g) {
      int32_t m = d.instr_loop[x0 + x];
      path.clear();
      for (; m != L; m = d.loop_parent[l0 + m]) path.push_back(m);
      int64_t c = g;
      for (size_t i = path.size(); i-- > 0;) c = rowptr[loop[l0 + path[i]].rowptr_off + c];
      return (int32_t)c;
    };
    // pieces: at most 64 runs of L's iterations, of about equal instances
    const int32_t np = std::min<int32_t>(T, 64);
    std::vector<int32_t> bnd(np + 1, 0);
    bnd[np] = T;
    if ((int64_t)T * nx <= (4 << 20)) {
      std::vector<int64_t> before(T + 1, 0);         // instances before each iteration of L
      for (int32_t g = 0; g <= T; ++g)
        for (int32_t x = 0; x < nx; ++x) before[g] += count(x, g);
      for (int32_t j = 1; j < np; ++j) {
        const int64_t target = before[T] * j / np;
        int32_t g = (int32_t)(std::lower_bound(before.begin(), before.end(), target) - before.begin());
        bnd[j] = std::min(std::max(g, bnd[j - 1] + 1), T - (np - j));
      }
    } else {
      for (int32_t j = 1; j < np; ++j) bnd[j] = (int32_t)((int64_t)T * j / np);
    }
    SplitProg S{};
    S.prog = p; S.first_piece = (int32_t)pieces.size(); S.n_pieces = np; S.nx = nx;
    S.ne = pi.ne; S.loop = l0 + L; S.x0 = x0;
    S.cnt_base = (int64_t)cnt.size();
    for (int32_t j = 0; j <= np; ++j)
      for (int32_t x = 0; x < nx; ++x) cnt.push_back(count(x, bnd[j]));
    S.vdep0 = (int32_t)vdep.size();
    for (int32_t k = d.prog_dep_ptr[p]; k < d.prog_dep_ptr[p + 1]; ++k) {
      if (dep[k].kase == CASE_BARRIER) continue;
      VDep v{};
      v.seg = seg[k];
      v.cons = d.dep_cons[k];
      for (int m = 0; m < kModes; ++m) v.sem[m] = xsem[(size_t)m * NX + x0 + d.dep_prod[k]].x;
      vdep.push_back(v);
    }
    S.vdep1 = (int32_t)vdep.size();
    // a semaphore's increments before a point: the instances before it of the
    // instructions that increment it (each instance increments once)
    int64_t span[kModes] = {0, 0, 0};
    for (int32_t j = 0; j < np; ++j) {
      PieceInfo pc{};
      pc.prog = p; pc.split = (int32_t)splits.size(); pc.loop = l0 + L; pc.g0 = bnd[j]; pc.g1 = bnd[j + 1];
      const int32_t* c = cnt.data() + S.cnt_base + (int64_t)j * nx;
      for (int m = 0; m < kModes; ++m) {
        pc.pub_off[m] = (int32_t)pub.size();
        pub.resize(pub.size() + pi.nsem[m], 0);
        for (int32_t x = 0; x < nx; ++x) {
          const int32_t sm = xsem[(size_t)m * NX + x0 + x].x;
          if (sm >= 0) pub[pc.pub_off[m] + sm] += c[x];
        }
      }
      pc.nbase_off = (int32_t)pub.size();
      pub.resize(pub.size() + pi.ne, 0);
      for (int32_t x = 0; x < nx; ++x) pub[pc.nbase_off + d.instr_engine[x0 + x]] += c[x];
      pieces.push_back(pc);
    }
    // probe histories: the program's history entries, per probe, at the
    // split programs' running offset (its entries are contiguous per mode)
    const int32_t* tot = cnt.data() + S.cnt_base + (int64_t)np * nx;
    for (int m = 0; m < kModes; ++m) {
      for (int32_t x = 0; x < nx; ++x)
        if (xsem[(size_t)m * NX + x0 + x].x >= 0) span[m] += tot[x];
      const int64_t first = pi.nsem[m] > 0 ? semhb[pi.semhb_off[m]] : 0;
      for (int32_t j = 0; j < np; ++j) pieces[S.first_piece + j].hdelta[m] = hist_split[m] - first;
      hist_split[m] += span[m];
    }
    // barrier-free: probed when the 2*ne runs per piece still leave the
    // program far above the batch's share per warp, speculated otherwise
    const bool bf = !force_spec && (double)pi.n_inst > 4.0 * (2.0 * pi.ne + 1.0) * share;
    bf_init.push_back(bf ? 0 : 1);
    if (bf) ne_max = std::max(ne_max, pi.ne);
    // the program's instances in the compact scratch of the stored times
    const int64_t first = nx > 0 ? inst_off[x0] : 0;
    for (int32_t j = 0; j < np; ++j) {
      pieces[S.first_piece + j].tl[0] = inst_bb - first;
      pieces[S.first_piece + j].tl[1] = bf ? inst_bf - first : 0;
    }
    inst_bb += pi.n_inst;
    if (bf) inst_bf += pi.n_inst;
    split_of[p] = (int32_t)splits.size();
    splits.push_back(S);
  }
  if (splits.empty()) return;
  h.n_split = (int32_t)splits.size();
  h.n_pieces = (int32_t)pieces.size();
  for (int32_t c : bf_init) (c ? h.n_spec : h.n_probed) += 1;
  h.sz.n_split_programs = h.n_split;
  h.sz.n_pieces = h.n_pieces;
  h.probes_bf = std::max(1, 2 * ne_max);
  for (int m = 0; m < kModes; ++m) h.phist_len[m] = hist_split[m];
  for (const SplitProg& S : splits) h.nx_max_split = std::max(h.nx_max_split, S.nx);
  h.pinst[0] = inst_bb;
  h.pinst[1] = inst_bf;
  {
    std::vector<int32_t> xe(d.instr_engine, d.instr_engine + NX);
    h.xeng = h.upload(xe, stream, "instruction engines");
  }
  h.pieces = h.upload(pieces, stream, "pieces");
  h.splits = h.upload(splits, stream, "split programs");
  h.prog_split = h.upload(split_of, stream, "program split index");
  h.piece_pub = h.upload(pub, stream, "piece start counts");
  h.piece_cnt = h.upload(cnt, stream, "piece instance counts");
  h.vdep = h.upload(vdep, stream, "split programs' dependencies");
  h.piece_cls = h.upload(bf_init, stream, "barrier-free split classes");
  h.spec_need = h.alloc<int32_t>(h.n_pieces, "speculation: runs due");
  h.spec_has = h.alloc<int32_t>(h.n_pieces, "speculation: runs done");
  h.spec_xhat = h.alloc<int32_t>((int64_t)h.n_pieces * 64, "speculation: guessed starts");
  h.piece_shift = h.alloc<int32_t>(h.n_pieces, "piece shifts");
  h.spec_vp = h.alloc<int32_t>(h.n_split, "speculation: accepted pieces");
  h.piece_fail = h.alloc<int32_t>(h.n_split, "piece validation flags");
  h.piece_out = h.alloc<int32_t>((int64_t)h.n_pieces * h.probes_bf * 64, "piece probe states");
  h.piece_x = h.alloc<int32_t>((int64_t)h.n_pieces * 64, "piece start states");
}

namespace {

// Host memory the loader reuses across loads (no page faults or zeroing of
// fresh pages after the first load of a size): the passes' scratch, and the
// pinned arena the tables are written into and copied from with one DMA.
// Each load takes one of each from a pool and gives it back; a pinned arena
// is reused only after the copy out of it has completed (its event).
struct HostScratch {
  HostVec<int32_t> i32_nl[2], body_ptr, body, i32_nx[6], i32_rows[2], anc, i32_nd[3];
  HostVec<uint8_t> u8_nl[2], rpflag, dep_bar;
  HostVec<int64_t> keys, i64_rows[3], ord_off, count, base;
  HostVec<uint32_t> pe_of;
  HostVec<Seen> seen;
  HostVec<ProgSummary> sum;
};
struct PinnedArena {
  char* p = nullptr;
  size_t cap = 0;
  int device = -1;
  cudaEvent_t done = nullptr;     // the last copy out of the arena
};
std::mutex g_pool_mu;
std::vector<HostScratch*> g_scratch_pool;
std::vector<PinnedArena*> g_arena_pool;

struct ScratchLease {
  HostScratch* s;
  ScratchLease() {
    std::lock_guard<std::mutex> g(g_pool_mu);
    if (g_scratch_pool.empty()) {
      s = new HostScratch();
    } else {
      s = g_scratch_pool.back();
      g_scratch_pool.pop_back();
    }
  }
  ~ScratchLease() {
    std::lock_guard<std::mutex> g(g_pool_mu);
    g_scratch_pool.push_back(s);
  }
};

struct ArenaLease {
  PinnedArena* a = nullptr;
  ArenaLease(size_t bytes, int device) {
    {
      std::lock_guard<std::mutex> g(g_pool_mu);
      // one of this device large enough, else any to grow
      size_t pick = g_arena_pool.size();
      for (size_t i = 0; i < g_arena_pool.size() && pick == g_arena_pool.size(); ++i)
        if (g_arena_pool[i]->device == device && g_arena_pool[i]->cap >= bytes) pick = i;
      if (pick == g_arena_pool.size() && !g_arena_pool.empty()) pick = 0;
      if (pick < g_arena_pool.size()) {
        a = g_arena_pool[pick];
        g_arena_pool.erase(g_arena_pool.begin() + (std::ptrdiff_t)pick);
      }
    }
    if (!a) a = new PinnedArena();
    if (a->done) cuda_check(cudaEventSynchronize(a->done), "host arena");
    if (a->cap < bytes || a->device != device) {
      if (a->p) cuda_check(cudaFreeHost(a->p), "host arena");
      a->p = nullptr;
      a->cap = 0;
      if (a->done) cudaEventDestroy(a->done);
      a->done = nullptr;
      a->device = device;
      const size_t cap = bytes + bytes / 8 + ((size_t)1 << 20);  // room to grow
      void* p = nullptr;
      cuda_check(cudaHostAlloc(&p, cap, cudaHostAllocDefault), "host arena");
      a->p = static_cast<char*>(p);
      a->cap = cap;
      cuda_check(cudaEventCreateWithFlags(&a->done, cudaEventDisableTiming), "host arena");
    }
  }
  ~ArenaLease() {
    std::lock_guard<std::mutex> g(g_pool_mu);
    g_arena_pool.push_back(a);
  }
};

template <class T>
T* sized(HostVec<T>& v, int64_t n) {
  if ((int64_t)v.size() < std::max<int64_t>(n, 1)) v.resize((size_t)std::max<int64_t>(n, 1));
  return v.data();
}

// Runs f(p) for programs [0, P) on host threads, in contiguous blocks.
template <class F>
void for_programs(int32_t P, F f) {
  const int n_threads = load_threads(P);
  std::vector<std::thread> pool;
  std::vector<std::exception_ptr> err(n_threads);
  for (int t = 0; t < n_threads; ++t) {
    const int32_t b = (int32_t)((int64_t)P * t / n_threads), e = (int32_t)((int64_t)P * (t + 1) / n_threads);
    auto job = [&f, &err, t, b, e] {
      try {
        for (int32_t p = b; p < e; ++p) f(p);
      } catch (...) {
        err[t] = std::current_exception();
      }
    };
    if (t + 1 < n_threads) pool.emplace_back(job); else job();
  }
  for (auto& th : pool) th.join();
  for (auto& x : err)
    if (x) std::rethrow_exception(x);
}

// COUNT over the covered programs on host threads (validation, counts and
// summaries), the first failure reported as the loader reports it, then the
// exclusive prefix sums of the counts; returns the totals.
void count_pass(const sync_batch_desc& d, const Shape& sh, HostScratch& H, BuildArgs& a,
                int64_t tot[kBuildCounts]) {
  const int32_t P = sh.P, Pq = sh.covered;
  const int64_t NL = sh.NL, NX = sh.NX, ND = sh.ND, rows = sh.rows;
  RawBatch& r = a.d;
  r.prog_loop_ptr = d.prog_loop_ptr; r.prog_instr_ptr = d.prog_instr_ptr; r.prog_dep_ptr = d.prog_dep_ptr;
  r.prog_n_engines = d.prog_n_engines; r.loop_parent = d.loop_parent; r.loop_pos = d.loop_pos;
  r.instr_loop = d.instr_loop; r.instr_pos = d.instr_pos; r.instr_engine = d.instr_engine;
  r.instr_latency = d.instr_latency; r.dep_prod = d.dep_prod; r.dep_cons = d.dep_cons; r.dep_k = d.dep_k;
  r.trip_ptr = d.trip_ptr; r.trips = d.trips; r.eng_trip_ptr = d.eng_trip_ptr; r.eng_trips = d.eng_trips;
  r.row_base = sh.row_base.data();
  r.P = Pq;
  r.div = sh.div ? 1 : 0;
  r.fallback = d.nonalloc_policy == SYNC_NONALLOC_BARRIER ? 1 : 0;
  r.NX = NX;
  r.ND = ND;
  BuildScratch& S = a.s;
  S.depth = sized(H.i32_nl[0], NL);
  S.lfill = sized(H.i32_nl[1], NL);
  S.needs_rhat = sized(H.u8_nl[0], NL);
  S.fbar = sized(H.u8_nl[1], NL);
  S.body_ptr = sized(H.body_ptr, NL + P);
  S.keys = sized(H.keys, NX + NL);
  S.body = sized(H.body, NX + NL);
  int32_t** nx_arrays[6] = {&S.rank, &S.x_ndeps, &S.x_dep_begin, &S.x_levels, &S.cons_next, &S.sem_x};
  for (int i = 0; i < 6; ++i) *nx_arrays[i] = sized(H.i32_nx[i], NX);
  S.nloop_eng = sized(H.i32_rows[0], rows);
  S.sem_row = sized(H.i32_rows[1], rows);
  int64_t** row_arrays[3] = {&S.stot, &S.srp, &S.tstart};
  for (int i = 0; i < 3; ++i) *row_arrays[i] = sized(H.i64_rows[i], rows);
  S.pe_of = sized(H.pe_of, rows);
  S.rpflag = sized(H.rpflag, rows);
  S.anc = sized(H.anc, rows * SYNC_MAX_DEPTH);
  S.dep_bar = sized(H.dep_bar, ND);
  S.dep_S = sized(H.i32_nd[0], ND);
  S.dep_N = sized(H.i32_nd[1], ND);
  S.by_cons = sized(H.i32_nd[2], ND);
  S.seen = sized(H.seen, ND);
  a.o.ord_off = sized(H.ord_off, NX);          // COUNT's dedup marks
  a.count = sized(H.count, (int64_t)Pq * kBuildCounts);
  a.sum = sized(H.sum, Pq);
  for_programs(Pq, [&a](int32_t p) {
    ProgBuilder<false> b(a, p);
    b.run();
  });
  for (int32_t p = 0; p < Pq; ++p)
    if (a.sum[p].err) raise_build_error(p, a.sum[p].err, a.sum[p].err_index);
  check_uncovered(d, sh);
  int64_t* base = sized(H.base, (int64_t)Pq * kBuildCounts);
  for (int i = 0; i < kBuildCounts; ++i) tot[i] = 0;
  for (int32_t p = 0; p < Pq; ++p)
    for (int i = 0; i < kBuildCounts; ++i) {
      base[(int64_t)p * kBuildCounts + i] = tot[i];
      tot[i] += a.count[(int64_t)p * kBuildCounts + i];
    }
  a.base = base;
  check_totals(tot);
}

// One allocation holding tables one after the other (each 256-byte aligned).
struct Layout {
  size_t bytes = 0;
  template <class T>
  size_t add(int64_t n) {
    const size_t off = bytes;
    bytes += ((size_t)std::max<int64_t>(n, 1) * sizeof(T) + 255) & ~(size_t)255;
    return off;
  }
};

// Programs in descending order of simulated work, equal work in program
// order: a stable least-significant-digit radix sort (11-bit digits) of the
// works' complements.
void work_order(const ProgSummary* sum, int32_t P, int32_t* order) {
  std::vector<uint64_t> key(P);
  uint64_t all_bits = 0;
  for (int32_t p = 0; p < P; ++p) {
    key[p] = ~(uint64_t)sum[p].work;             // work >= 0: larger work, smaller key
    order[p] = p;
  }
  for (int32_t p = 0; p < P; ++p) all_bits |= key[p] ^ key[0];   // the digits that differ somewhere
  std::vector<int32_t> tmp(P);
  for (int shift = 0; shift < 64; shift += 11) {
    if (((all_bits >> shift) & 0x7ff) == 0) continue;
    int32_t cnt[2049] = {0};
    for (int32_t i = 0; i < P; ++i) ++cnt[((key[order[i]] >> shift) & 0x7ff) + 1];
    for (int b = 0; b < 2048; ++b) cnt[b + 1] += cnt[b];
    for (int32_t i = 0; i < P; ++i) tmp[cnt[(key[order[i]] >> shift) & 0x7ff]++] = order[i];
    std::copy(tmp.begin(), tmp.end(), order);
  }
}

}  // namespace

// The loader.  On the host: the shape checks, then COUNT (validation and
// per-program counts) and FILL (every table at the program's offsets) of
// progbuild.cuh, one program at a time on host threads, FILL writing into a
// pinned arena; the tables go to the device in one copy.  On the device,
// from those tables: the tile tables, the per-mode semaphore records and
// the derived per-iteration arrays.  The
// per-program passes are scalar, branchy code over small tables (a few
// hundred entries per program); the per-iteration and per-pair arrays are
// built by the GPU.
static void build(const sync_batch_desc& d, int device, cudaStream_t stream, sync_programs& h) {
  const Shape sh = shape_checks(d);
  const int32_t P = sh.P;
  const int64_t NL = sh.NL, NX = sh.NX, ND = sh.ND, rows = sh.rows;
  const bool div = sh.div;
  ScratchLease SL;
  BuildArgs a{};
  int64_t cnt[kBuildCounts];
  count_pass(d, sh, *SL.s, a, cnt);
  cuda_check(cudaSetDevice(device), "cudaSetDevice");
  h.device = device;
  cuda_check(cudaDeviceGetAttribute(&h.num_sms, cudaDevAttrMultiProcessorCount, device), "device attributes");

  // ----------------------------------------------------------- layout
  const int64_t n_ops = cnt[BC_OPS], n_plan = cnt[BC_PLAN], n_lanes = cnt[BC_LANES];
  const int64_t n_iters = cnt[BC_ITERS], n_derived = cnt[BC_DERIVED], n_jobs = cnt[BC_JOBS];
  const int64_t n_pairs_padded = cnt[BC_PADDED];
  const int64_t n_xloops = div ? rows : NL;
  int64_t hist_max = 0;
  for (int m = 0; m < kModes; ++m) hist_max = std::max(hist_max, h.hist_len[m] = cnt[BC_HIST + m]);
  const int64_t n_first_tiles = (n_pairs_padded + kTilePairs - 1) / kTilePairs;
  const int64_t n_drows = cnt[BC_DROWS];
  const int64_t n_job_tiles = (n_drows + kJobTileRows - 1) / kJobTileRows;
  Layout L;   // the tables the host writes, then the device's own
  const size_t o_loop = L.add<LoopInfo>(NL), o_dep = L.add<DepInfo>(ND), o_prog = L.add<ProgInfo>(P);
  const size_t o_inst = L.add<int64_t>(NX), o_ord = L.add<int64_t>(NX), o_xsem = L.add<int4>(kModes * NX);
  const size_t o_xcse = L.add<int4>(NX), o_xlvr = L.add<int32_t>(NX), o_seg = L.add<int64_t>(ND + 1);
  const size_t o_count = L.add<int32_t>(ND), o_dseg = L.add<int64_t>(ND), o_ddep = L.add<int32_t>(ND);
  const size_t o_dsem = L.add<int32_t>(kModes * ND), o_lflag = L.add<int32_t>(NL);
  const size_t o_plan_ptr = L.add<int32_t>(NL + 1), o_op_ptr = L.add<int32_t>(rows + 1);
  const size_t o_rowinfo = L.add<int2>(rows), o_hoist = L.add<int32_t>(rows);
  const size_t o_xloops = L.add<LoopInfo>(n_xloops), o_reads = L.add<uint8_t>(n_xloops);
  const size_t o_rowptr = L.add<int32_t>(cnt[BC_ROWPTR]), o_path = L.add<int64_t>(cnt[BC_PATH]);
  const size_t o_jobs = L.add<DeriveJob>(n_jobs), o_ops = L.add<int4>(n_ops), o_opstop = L.add<int32_t>(n_ops);
  const size_t o_semhb = L.add<int64_t>(cnt[BC_SEMHB]), o_plan = L.add<int4>(n_plan), o_paux = L.add<int4>(n_plan);
  const size_t o_chunks = L.add<int4>(cnt[BC_CHUNKS]), o_lrec = L.add<int4>(n_lanes), o_lmeta = L.add<int4>(n_lanes);
  const size_t o_order = L.add<int32_t>(P);
  const size_t host_bytes = L.bytes;
  const size_t o_derived = L.add<int32_t>(n_derived);
  const size_t o_opsem = L.add<int4>(kModes * n_ops), o_lsem = L.add<int4>(kModes * n_lanes);
  const size_t o_hist = L.add<int32_t>(hist_max), o_slot = L.add<int32_t>(1), o_fallback = L.add<int32_t>((int64_t)P + 1);
  const size_t o_tile_first = L.add<int32_t>(n_first_tiles + 1), o_tile_job = L.add<int32_t>(n_job_tiles + 1);
  char* dev = h.alloc<char>((int64_t)L.bytes, "encoding");

  // ------------------------------------------------------------- FILL
  ArenaLease AL(host_bytes, device);
  char* host = AL.a->p;
  BuildOut& O = a.o;
  O.loop = reinterpret_cast<LoopInfo*>(host + o_loop);
  O.dep = reinterpret_cast<DepInfo*>(host + o_dep);
  O.prog = reinterpret_cast<ProgInfo*>(host + o_prog);
  O.inst_off = reinterpret_cast<int64_t*>(host + o_inst);
  O.ord_off = reinterpret_cast<int64_t*>(host + o_ord);
  O.xsem = reinterpret_cast<int4*>(host + o_xsem);
  O.xcse = reinterpret_cast<int4*>(host + o_xcse);
  O.xlvr = reinterpret_cast<int32_t*>(host + o_xlvr);
  O.seg = reinterpret_cast<int64_t*>(host + o_seg);
  O.dep_count = reinterpret_cast<int32_t*>(host + o_count);
  O.dseg = reinterpret_cast<int64_t*>(host + o_dseg);
  O.ddep = reinterpret_cast<int32_t*>(host + o_ddep);
  O.dsem = reinterpret_cast<int32_t*>(host + o_dsem);
  O.lflag = reinterpret_cast<int32_t*>(host + o_lflag);
  O.plan_ptr = reinterpret_cast<int32_t*>(host + o_plan_ptr);
  O.op_ptr = reinterpret_cast<int32_t*>(host + o_op_ptr);
  O.rowinfo = reinterpret_cast<int2*>(host + o_rowinfo);
  O.hoist = reinterpret_cast<int32_t*>(host + o_hoist);
  O.xloops = reinterpret_cast<LoopInfo*>(host + o_xloops);
  O.reads_rowptr = reinterpret_cast<uint8_t*>(host + o_reads);
  O.rowptr = reinterpret_cast<int32_t*>(host + o_rowptr);
  O.path = reinterpret_cast<int64_t*>(host + o_path);
  O.jobs = reinterpret_cast<DeriveJob*>(host + o_jobs);
  O.ops = reinterpret_cast<int4*>(host + o_ops);
  O.opstop = reinterpret_cast<int32_t*>(host + o_opstop);
  O.semhb = reinterpret_cast<int64_t*>(host + o_semhb);
  O.plan = reinterpret_cast<int4*>(host + o_plan);
  O.paux = reinterpret_cast<int4*>(host + o_paux);
  O.chunks = reinterpret_cast<int4*>(host + o_chunks);
  O.lrec = reinterpret_cast<int4*>(host + o_lrec);
  O.lmeta = reinterpret_cast<int4*>(host + o_lmeta);
  // the closing entries of the offset tables: 0 without programs, else the
  // last program's FILL writes them
  O.seg[ND] = 0;
  O.op_ptr[rows] = 0;
  O.plan_ptr[NL] = 0;
  for_programs(P, [&a](int32_t p) {
    ProgBuilder<true> b(a, p);
    b.run();
  });
  work_order(a.sum, P, reinterpret_cast<int32_t*>(host + o_order));
  cuda_check(cudaMemcpyAsync(dev, host, host_bytes, cudaMemcpyHostToDevice, stream), "encoding");
  cuda_check(cudaEventRecord(AL.a->done, stream), "encoding");
  h.sz.h2d_bytes += (int64_t)host_bytes;

  // ----------------------------------------------------------- handle
  auto D = [dev](size_t off) { return dev + off; };
  h.loop = reinterpret_cast<LoopInfo*>(D(o_loop));
  h.dep = reinterpret_cast<DepInfo*>(D(o_dep));
  h.prog = reinterpret_cast<ProgInfo*>(D(o_prog));
  h.inst_off = reinterpret_cast<int64_t*>(D(o_inst));
  h.ord_off = reinterpret_cast<int64_t*>(D(o_ord));
  h.cost.xcse = reinterpret_cast<int4*>(D(o_xcse));
  h.cost.xlvr = reinterpret_cast<int32_t*>(D(o_xlvr));
  h.cost.hoist = reinterpret_cast<int32_t*>(D(o_hoist));
  h.seg = reinterpret_cast<int64_t*>(D(o_seg));
  h.dep_count = reinterpret_cast<int32_t*>(D(o_count));
  h.dseg = reinterpret_cast<int64_t*>(D(o_dseg));
  h.ddep = reinterpret_cast<int32_t*>(D(o_ddep));
  h.dsem = reinterpret_cast<int32_t*>(D(o_dsem));
  h.lflag = reinterpret_cast<int32_t*>(D(o_lflag));
  h.plan_ptr = reinterpret_cast<int32_t*>(D(o_plan_ptr));
  h.op_ptr = reinterpret_cast<int32_t*>(D(o_op_ptr));
  h.rowinfo = reinterpret_cast<int2*>(D(o_rowinfo));
  h.rowptr = reinterpret_cast<int32_t*>(D(o_rowptr));
  h.path = reinterpret_cast<int64_t*>(D(o_path));
  h.ops = reinterpret_cast<int4*>(D(o_ops));
  h.opstop = reinterpret_cast<int32_t*>(D(o_opstop));
  h.semhb = reinterpret_cast<int64_t*>(D(o_semhb));
  h.plan = reinterpret_cast<int4*>(D(o_plan));
  h.paux = reinterpret_cast<int4*>(D(o_paux));
  h.chunk = reinterpret_cast<int4*>(D(o_chunks));
  h.lrec = reinterpret_cast<int4*>(D(o_lrec));
  h.lmeta = reinterpret_cast<int4*>(D(o_lmeta));
  h.order = reinterpret_cast<int32_t*>(D(o_order));
  h.derived = reinterpret_cast<int32_t*>(D(o_derived));
  h.opsem = reinterpret_cast<int4*>(D(o_opsem));
  h.lsem = reinterpret_cast<int4*>(D(o_lsem));
  h.hist = reinterpret_cast<int32_t*>(D(o_hist));
  h.next_slot = reinterpret_cast<int32_t*>(D(o_slot));
  h.fallback = reinterpret_cast<int32_t*>(D(o_fallback));
  h.tile_first = reinterpret_cast<int32_t*>(D(o_tile_first));
  const DeriveJob* d_jobs = reinterpret_cast<const DeriveJob*>(D(o_jobs));
  int32_t* tile_job = reinterpret_cast<int32_t*>(D(o_tile_job));

  // ------------------------------------------------------------ sizes
  int64_t struct_extra = 0, code_looped = 0, code_unrolled = 0, n_bar_deps = 0;
  int32_t ne_max = 1, depth_max = 0, ord_overflow = 0;
  for (int32_t p = 0; p < P; ++p) {
    const ProgSummary& s = a.sum[p];
    struct_extra += s.struct_bytes;
    code_looped += s.code_looped;
    code_unrolled += s.code_unrolled;
    n_bar_deps += s.n_bar_deps;
    ne_max = std::max(ne_max, s.ne);
    depth_max = std::max(depth_max, s.depth_max);
    ord_overflow |= s.ord_overflow;
    for (int m = 0; m < kModes; ++m) h.nsem_max[m] = std::max(h.nsem_max[m], s.nsem[m]);
  }
  h.sz.n_pairs = cnt[BC_PAIRS];
  h.sz.n_pairs_padded = n_pairs_padded;
  h.sz.n_instances = cnt[BC_INST];
  h.sz.n_loop_iters = n_iters;
  h.sz.n_programs = P;
  h.sz.n_loops = (int32_t)NL;
  h.sz.n_instrs = (int32_t)NX;
  h.sz.n_deps = (int32_t)ND;
  // of the path pool the kernels read only the rowptr offsets from S's
  // child down to a nested producer's loop; the consumer side's are read at
  // load time only
  h.sz.struct_bytes = ND * (int64_t)sizeof(DepInfo) + 8 * (ND + 1) + struct_extra + 4 * (n_first_tiles + 1) +
                      4 * n_derived;
  h.sz.code_bytes_looped = SYNC_CODE_BYTES_PER_INSTR * code_looped;
  h.sz.code_bytes_unrolled = SYNC_CODE_BYTES_PER_INSTR * code_unrolled;
  h.ne_max = ne_max;
  h.depth_max = depth_max;
  h.n_bar_deps = n_bar_deps;
  h.n_ord = cnt[BC_ORD];
  h.ord_overflow = ord_overflow != 0;
  h.n_chunks = n_pairs_padded / kChunk;
  h.n_ops = n_ops;
  h.n_lanes = n_lanes;
  h.divergent = div;

  // ------------------------------------------- piece-parallel candidates
  // (build_pieces reads the host tables: the arena stays leased until the
  // end of the load)
  {
    const double share = (double)cnt[BC_INST] / ((double)h.num_sms * 24.0);
    const int64_t min_inst = split_floor();
    bool any = false;
    for (int32_t p = 0; p < P && !any; ++p)
      any = a.sum[p].splittable && a.sum[p].n_inst >= min_inst && (double)a.sum[p].n_inst > 8.0 * share;
    if (any)
      build_pieces(d, O.loop, O.rowptr, O.xsem, O.dep, O.seg, O.semhb, O.prog, O.inst_off, cnt[BC_INST], stream, h);
  }

  // ----------------------------------------------------------- device
  cuda_check(launch_tile_tables(h.seg, ND, h.tile_first, n_first_tiles, d_jobs, n_jobs, tile_job, n_job_tiles,
                                h.num_sms, stream),
             "tile tables");
  cuda_check(launch_sem_records(reinterpret_cast<const int4*>(D(o_xsem)), NX, h.ops, n_ops, h.lrec, n_lanes, h.opsem,
                                h.lsem, h.num_sms, stream),
             "semaphore records");
  cuda_check(launch_derive(d_jobs, tile_job, n_drows, h.rowptr, h.path, h.derived, n_derived, h.num_sms, stream),
             "derive");
  cuda_check(cudaEventCreateWithFlags(&h.ready, cudaEventDisableTiming), "load event");
  cuda_check(cudaEventRecord(h.ready, stream), "load event");
}

// Host validation (sync_validate_programs): the shape checks and COUNT.
static void validate(const sync_batch_desc& d) {
  const Shape sh = shape_checks(d);
  ScratchLease SL;
  BuildArgs a{};
  int64_t tot[kBuildCounts];
  count_pass(d, sh, *SL.s, a, tot);
}


extern "C" {

sync_status sync_load_programs(const sync_batch_desc* desc, int device, void* stream,
                               sync_programs** out) {
  try {
    if (!desc || !out) raise(SYNC_ERR_ARG, "desc and out must not be NULL");
    *out = nullptr;
    std::unique_ptr<sync_programs> h(new sync_programs());
    build(*desc, device, static_cast<cudaStream_t>(stream), *h);
    *out = h.release();
    g_err.clear();
    return SYNC_OK;
  } catch (const Failure& f) {
    return report(f);
  } catch (const std::bad_alloc&) {
    return report(Failure{SYNC_ERR_OOM, "host allocation failed"});
  } catch (...) {
    return report(Failure{SYNC_ERR_ARG, "unexpected error"});
  }
}

sync_status sync_query(const sync_programs* h, sync_sizes* out) {
  if (!h || !out) return report(Failure{SYNC_ERR_ARG, "handle and out must not be NULL"});
  *out = h->sz;
  return SYNC_OK;
}

sync_status sync_pair_offsets(const sync_programs* h, int64_t* offsets, int32_t* counts) {
  if (!h || !offsets) return report(Failure{SYNC_ERR_ARG, "handle and offsets must not be NULL"});
  try {
    std::lock_guard<std::mutex> lock(h->pair_mu);
    if (!h->pairs_ready) {                         // read back on first use
      const int64_t nd = h->sz.n_deps;
      h->seg_host.resize((size_t)nd + 1);
      h->count_host.resize((size_t)nd);
      cuda_check(cudaSetDevice(h->device), "cudaSetDevice");
      // a stream of its own, blocking nothing else: the copies wait for the
      // load only, not for work queued on other streams
      cudaStream_t s = nullptr;
      cuda_check(cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking), "pair layout stream");
      cudaError_t e = h->wait_ready(s);
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(h->seg_host.data(), h->seg, (size_t)(nd + 1) * sizeof(int64_t), cudaMemcpyDeviceToHost, s);
      if (e == cudaSuccess && nd > 0)
        e = cudaMemcpyAsync(h->count_host.data(), h->dep_count, (size_t)nd * sizeof(int32_t), cudaMemcpyDeviceToHost, s);
      if (e == cudaSuccess) e = cudaStreamSynchronize(s);
      cudaStreamDestroy(s);
      cuda_check(e, "pair layout");
      h->pairs_ready = true;
    }
  } catch (const Failure& f) {
    return report(f);
  }
  std::memcpy(offsets, h->seg_host.data(), h->seg_host.size() * sizeof(int64_t));
  if (counts) std::memcpy(counts, h->count_host.data(), h->count_host.size() * sizeof(int32_t));
  return SYNC_OK;
}

static ThrArgs thr_args(const sync_programs* h, sync_thr_mode mode) {
  ThrArgs a;
  a.dep = h->dep; a.derived = h->derived; a.ord = h->ord; a.seg = h->seg; a.tile_first = h->tile_first;
  a.path = h->path; a.rowptr = h->rowptr; a.n_chunks = h->n_chunks; a.mode = mode;
  return a;
}

// thresholds and check: all three encodings
// Per-engine trip counts: per-engine wait values are not defined (a position
// in the producer engine's stream that the consumer's loop state no longer
// determines), and the barrier scheme has no common barrier sequence.
static void check_divergent(const sync_programs* h, sync_thr_mode mode, bool sim, sync_sim_variant variant) {
  if (!h->divergent) return;
  if (mode == SYNC_THR_PERENGINE)
    raise(SYNC_ERR_ARG, "per-engine trip counts: per-engine thresholds are not defined");
  if (sim && variant != SYNC_SIM_BARRIER_FREE)
    raise(SYNC_ERR_ARG, "per-engine trip counts: only the barrier-free schedule is defined");
}

static void check_thr_mode(sync_thr_mode mode) {
  if (mode != SYNC_THR_COUNT && mode != SYNC_THR_PERLOOP && mode != SYNC_THR_PERENGINE)
    raise(SYNC_ERR_ARG, "unknown threshold mode");
}

// Per-engine mode: derive the engine-stream positions of the waited
// producers' instances on first use (kept by the handle).
static void ensure_ordinals(const sync_programs* h, cudaStream_t s) {
  std::lock_guard<std::mutex> lock(h->ord_mu);
  if (h->ord_ready) return;
  if (h->ord_overflow)
    raise(SYNC_ERR_OVERFLOW, "an engine of a program has more than INT32_MAX instances: its stream positions do not fit int32");
  sync_programs* m = const_cast<sync_programs*>(h);
  int32_t* ord = m->alloc<int32_t>(h->n_ord, "engine-stream positions");
  cuda_check(launch_ordinals(h->prog, h->order, h->sz.n_programs, h->ne_max, h->op_ptr, h->ops, h->rowptr, h->ord_off, ord,
                             h->num_sms, s), "engine-stream positions");
  cuda_check(cudaStreamSynchronize(s), "engine-stream positions");
  h->ord = ord;
  h->ord_ready = true;
}

sync_status sync_eval_thresholds(const sync_programs* h, sync_thr_mode mode, int32_t* d_thr,
                                 void* stream) {
  try {
    if (!h) raise(SYNC_ERR_ARG, "handle must not be NULL");
    check_thr_mode(mode);
    check_divergent(h, mode, false, SYNC_SIM_BARRIER_FREE);
    if (h->sz.n_pairs_padded > 0 && !d_thr) raise(SYNC_ERR_ARG, "d_thr must not be NULL");
    if (reinterpret_cast<uintptr_t>(d_thr) % 16) raise(SYNC_ERR_ARG, "d_thr must be 16-byte aligned");
    cuda_check(cudaSetDevice(h->device), "cudaSetDevice");
    cuda_check(h->wait_ready(static_cast<cudaStream_t>(stream)), "load completion");
    if (mode == SYNC_THR_PERENGINE) ensure_ordinals(h, static_cast<cudaStream_t>(stream));
    cuda_check(launch_thresholds(thr_args(h, mode), d_thr, h->num_sms, static_cast<cudaStream_t>(stream)),
               "threshold kernel");
    return SYNC_OK;
  } catch (const Failure& f) {
    return report(f);
  }
}

sync_status sync_check_minimal(const sync_programs* h, sync_thr_mode mode, const int32_t* d_thr,
                               unsigned long long* d_counts, long long* d_first_bad, void* stream) {
  try {
    if (!h || !d_counts || !d_first_bad) raise(SYNC_ERR_ARG, "handle and outputs must not be NULL");
    check_thr_mode(mode);
    check_divergent(h, mode, false, SYNC_SIM_BARRIER_FREE);
    if (h->sz.n_pairs_padded > 0 && !d_thr) raise(SYNC_ERR_ARG, "d_thr must not be NULL");
    if (reinterpret_cast<uintptr_t>(d_thr) % 16) raise(SYNC_ERR_ARG, "d_thr must be 16-byte aligned");
    cuda_check(cudaSetDevice(h->device), "cudaSetDevice");
    cuda_check(h->wait_ready(static_cast<cudaStream_t>(stream)), "load completion");
    if (mode == SYNC_THR_PERENGINE) ensure_ordinals(h, static_cast<cudaStream_t>(stream));
    CheckArgs a;
    a.t = thr_args(h, mode);
    a.thr = d_thr;
    a.counts = d_counts;
    a.first_bad = reinterpret_cast<unsigned long long*>(d_first_bad);
    cuda_check(launch_check(a, h->num_sms, static_cast<cudaStream_t>(stream)), "checker kernel");
    return SYNC_OK;
  } catch (const Failure& f) {
    return report(f);
  }
}

// The probe runs' private semaphore histories of a mode (barrier-free piece
// simulation), allocated on first use and kept by the handle.
static int32_t* probe_history(const sync_programs* h, sync_thr_mode mode) {
  std::lock_guard<std::mutex> lock(h->phist_mu);
  if (!h->phist[mode])
    h->phist[mode] = h->alloc_lazy<int32_t>((int64_t)h->probes_bf * std::max<int64_t>(h->phist_len[mode], 1),
                                            "probe histories");
  return h->phist[mode];
}

// The stored times of the piece runs: per instance of the split programs
// (barrier-free: of the ones split barrier-free) issue and retire per run
// and the position in its engine's stream; allocated on first use.
static int32_t* stored_times(const sync_programs* h, bool barrier) {
  std::lock_guard<std::mutex> lock(h->phist_mu);
  const int k = barrier ? 0 : 1;
  if (!h->ptimes[k]) {
    const int64_t runs = barrier ? 1 : h->probes_bf;
    h->ptimes[k] = h->alloc_lazy<int32_t>((2 * runs + 1) * std::max<int64_t>(h->pinst[k], 1), "piece times");
  }
  return h->ptimes[k];
}

// Both simulation entry points: thresholds from d_thr, or (fused) from the
// simulators' loop state, optionally checked.
static void simulate(const sync_programs* h, sync_thr_mode mode, bool fused, const int32_t* d_thr,
                     const sync_sim_params* params,
                     sync_sim_variant variant, int32_t* d_makespan, unsigned long long* d_checksum,
                     int32_t* d_status, int32_t* d_issue, int32_t* d_retire, unsigned long long* d_counts,
                     long long* d_first_bad, void* stream) {
  if (!h || !params) raise(SYNC_ERR_ARG, "handle and params must not be NULL");
  check_thr_mode(mode);
  if (variant != SYNC_SIM_BARRIER_FREE && variant != SYNC_SIM_BARRIER && variant != SYNC_SIM_UNROLLED)
    raise(SYNC_ERR_ARG, "unknown variant");
  if (variant == SYNC_SIM_UNROLLED && mode != SYNC_THR_PERENGINE)
    raise(SYNC_ERR_ARG, "the unrolled variant takes per-engine thresholds");
  if (variant == SYNC_SIM_UNROLLED && h->n_bar_deps > 0)
    raise(SYNC_ERR_ARG, "the unrolled variant takes no barrier-fallback dependencies");
  check_divergent(h, mode, true, variant);
  if (h->sz.n_programs > 0 && (!d_makespan || !d_checksum || !d_status))
    raise(SYNC_ERR_ARG, "per-program outputs must not be NULL");
  if ((d_issue == nullptr) != (d_retire == nullptr)) raise(SYNC_ERR_ARG, "d_issue and d_retire: both or neither");
  if ((d_counts == nullptr) != (d_first_bad == nullptr))
    raise(SYNC_ERR_ARG, "d_counts and d_first_bad: both or neither");
  sync_sim_params q;
  if (!syncgb::sim_params_for(*params, variant, q)) raise(SYNC_ERR_ARG, "timing constants must be >= 0");
  cuda_check(cudaSetDevice(h->device), "cudaSetDevice");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cuda_check(h->wait_ready(st), "load completion");
  if (fused && mode == SYNC_THR_PERENGINE) ensure_ordinals(h, st);
  if (d_counts) {
    cuda_check(cudaMemsetAsync(d_counts, 0, 2 * sizeof(unsigned long long), st), "cudaMemsetAsync");
    cuda_check(cudaMemsetAsync(d_first_bad, 0xff, sizeof(long long), st), "cudaMemsetAsync");
  }
  SimArgs a;
  std::memset(&a, 0, sizeof a);
  a.prog = h->prog; a.order = h->order; a.rowptr = h->rowptr;
  a.op_ptr = h->op_ptr; a.rowinfo = h->rowinfo; a.ops = h->ops; a.opstop = h->opstop;
  a.opsem = h->opsem + (size_t)mode * h->n_ops;
  a.dseg = h->dseg; a.dsem = h->dsem + (size_t)mode * h->sz.n_deps;
  a.semhb = h->semhb;
  a.inst_off = h->inst_off;
  a.thr = d_thr; a.hist = h->hist; a.next_slot = h->next_slot;
  a.makespan = d_makespan; a.checksum = d_checksum; a.status = d_status;
  a.issue = d_issue; a.retire = d_retire;
  a.prm = q;
  a.n_programs = h->sz.n_programs;
  a.mode = mode;
  a.sem_cap = std::max(4, (h->nsem_max[mode] + 3) & ~3);
  a.frame_depth = std::max(1, h->depth_max);
  a.warps = h->ne_max;
  a.cost = h->cost;
  if (fused) {
    a.dep = h->dep; a.ddep = h->ddep; a.path = h->path; a.ord = h->ord;
    a.chk_counts = d_counts; a.chk_first = reinterpret_cast<unsigned long long*>(d_first_bad);
  }
  const int ring = sweep_ring_for(a.sem_cap, a.frame_depth, 200 * 1024);
  if (simulate_smem_bytes(a.warps, a.sem_cap, a.frame_depth) > 200 * 1024 || ring == 0)
    raise(SYNC_ERR_ARG, "a program has too many waited semaphores for the simulator's shared memory");
  SweepArgs w;
  std::memset(&w, 0, sizeof w);
  w.prog = h->prog; w.order = h->order; w.loop = h->loop; w.rowptr = h->rowptr;
  w.plan_ptr = h->plan_ptr; w.plan = h->plan; w.chunk = h->chunk;
  w.lrec = h->lrec; w.lmeta = h->lmeta; w.lsem = h->lsem + (size_t)mode * h->n_lanes;
  w.dseg = h->dseg; w.dsem = a.dsem; w.semhb = h->semhb; w.inst_off = h->inst_off;
  w.thr = d_thr; w.hist = h->hist; w.next_slot = h->next_slot; w.fallback = h->fallback;
  w.makespan = d_makespan; w.checksum = d_checksum; w.status = d_status;
  w.issue = d_issue; w.retire = d_retire;
  w.prm = q; w.n_programs = a.n_programs; w.mode = mode;
  w.sem_cap = a.sem_cap; w.frame_depth = a.frame_depth; w.ring = ring; w.lflag = h->lflag; w.paux = h->paux;
  w.cost = h->cost;
  w.dep = a.dep; w.ddep = a.ddep; w.path = a.path; w.ord = a.ord;
  w.chk_counts = a.chk_counts; w.chk_first = a.chk_first;
  const bool barrier = variant == SYNC_SIM_BARRIER;
  // split programs (array thresholds): simulated piece by piece on many warps
  // first; the sweep skips the ones the pieces completed
  if (!fused && h->n_split > 0) {
    cuda_check(cudaMemsetAsync(h->piece_fail, 0, sizeof(int32_t) * (size_t)h->n_split, st), "cudaMemsetAsync");
    w.pcs.piece = h->pieces; w.pcs.split = h->splits; w.pcs.prog_split = h->prog_split;
    w.pcs.pub = h->piece_pub; w.pcs.fail = h->piece_fail; w.pcs.out = h->piece_out; w.pcs.x = h->piece_x;
    w.pcs.n_pieces = h->n_pieces;
    w.pcs.out_probes = h->probes_bf;
    w.pcs.xeng = h->xeng;
    w.pcs.nx_max = h->nx_max_split;
    w.pcs.cls = h->piece_cls; w.pcs.need = h->spec_need; w.pcs.has = h->spec_has; w.pcs.xhat = h->spec_xhat;
    w.pcs.shift = h->piece_shift; w.pcs.vp = h->spec_vp;
    SweepArgs wp = w;
    PieceLaunch L{h->vdep, h->piece_cnt, stored_times(h, true), h->pinst[0], h->n_split, 0, 0};
    if (barrier) {
      wp.pcs.probes = 1;
    } else {
      L.n_probed = h->n_probed;
      L.n_spec = h->n_spec;
      wp.pcs.probes = h->probes_bf;
      if (h->n_probed > 0) {                       // the probes' histories and stored times
        wp.pcs.phist = probe_history(h, mode);
        wp.pcs.phist_len = h->phist_len[mode];
        wp.pcs.ptimes = stored_times(h, false);
        wp.pcs.plen = h->pinst[1];
      }
    }
    cuda_check(launch_pieces(wp, barrier, L, h->num_sms, st), "piece simulation");
  }
  cuda_check(launch_sweep(w, barrier, h->num_sms, st), "sweep simulator kernel");
  a.only = h->fallback;
  cuda_check(launch_simulate(a, barrier, h->num_sms, st), "per-engine simulator kernel");
}

sync_status sync_simulate(const sync_programs* h, sync_thr_mode mode, const int32_t* d_thr,
                          const sync_sim_params* params, sync_sim_variant variant,
                          int32_t* d_makespan, unsigned long long* d_checksum, int32_t* d_status,
                          int32_t* d_issue, int32_t* d_retire, void* stream) {
  try {
    if (h && h->sz.n_pairs_padded > 0 && !d_thr) raise(SYNC_ERR_ARG, "d_thr must not be NULL");
    simulate(h, mode, false, d_thr, params, variant, d_makespan, d_checksum, d_status, d_issue, d_retire, nullptr,
             nullptr, stream);
    return SYNC_OK;
  } catch (const Failure& f) {
    return report(f);
  }
}

sync_status sync_simulate_fused(const sync_programs* h, sync_thr_mode mode, const sync_sim_params* params,
                                sync_sim_variant variant, int32_t* d_makespan, unsigned long long* d_checksum,
                                int32_t* d_status, int32_t* d_issue, int32_t* d_retire,
                                unsigned long long* d_counts, long long* d_first_bad, void* stream) {
  try {
    simulate(h, mode, true, nullptr, params, variant, d_makespan, d_checksum, d_status, d_issue, d_retire, d_counts,
             d_first_bad, stream);
    return SYNC_OK;
  } catch (const Failure& f) {
    return report(f);
  }
}

void sync_free_programs(sync_programs* h) { delete h; }

sync_status sync_validate_programs(const sync_batch_desc* desc) {
  try {
    if (!desc) raise(SYNC_ERR_ARG, "desc must not be NULL");
    validate(*desc);
    g_err.clear();
    return SYNC_OK;
  } catch (const Failure& f) {
    return report(f);
  } catch (const std::bad_alloc&) {
    return report(Failure{SYNC_ERR_OOM, "host allocation failed"});
  } catch (...) {
    return report(Failure{SYNC_ERR_ARG, "unexpected error"});
  }
}

const char* sync_last_error(void) { return g_err.c_str(); }

int64_t sync_kernel_launches(void) { return g_launches.load(std::memory_order_relaxed); }

}  // extern "C"
