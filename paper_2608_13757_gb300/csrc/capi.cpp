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

constexpr int64_t kI32Max = 2147483647;

int64_t pad4(int64_t n) { return (n + 3) & ~int64_t(3); }

// Code-size proxy: wait-value ops of a per-loop wait (Table 1) and control
// ops of a loop on one engine (r-hat := 0, branch, r++, r-hat++).
constexpr int64_t kCodeWaitOps = 5;
constexpr int64_t kCodeLoopOps = 4;

// Threads of the loader's per-program pass: one per hardware thread (at most
// 32) while each gets at least 256 programs.  SYNCGB_LOAD_THREADS=n sets the
// count (tests use it to run the block join on small batches).
int load_threads(int32_t P) {
  int n = 0;
  if (const char* v = std::getenv("SYNCGB_LOAD_THREADS")) n = std::atoi(v);
  if (n <= 0) {
    n = std::min(32, (int)std::max(1u, std::thread::hardware_concurrency()));
    n = (int)std::min<int64_t>(n, std::max<int64_t>(1, P / 256));
  }
  return std::max(1, std::min(n, std::max(1, (int)P)));
}

}  // namespace

namespace {

struct Batch {
  const sync_batch_desc& d;
  int32_t P;
  int64_t NL, NX, ND, NT;
};

void check_csr(const int32_t* ptr, int32_t P, const char* name) {
  if (ptr[0] != 0) raise(SYNC_ERR_MALFORMED, std::string(name) + "[0] must be 0");
  for (int32_t p = 0; p < P; ++p)
    if (ptr[p + 1] < ptr[p]) raise(SYNC_ERR_MALFORMED, std::string(name) + " is not nondecreasing");
}

// Per-program scratch of the loader (reused across programs).
struct ProgScratch {
  std::vector<int32_t> depth, body_ptr, body, rank, nloop_eng, x_ndeps, x_dep_begin;
  std::vector<int32_t> x_own[kModes], x_hstride[kModes], x_koff[kModes], x_levels;
  std::vector<int64_t> total, keys;
  std::vector<int64_t> etot;                      // per-engine trips: iterations per (loop, engine)
  std::vector<LoopInfo> el;                       // per-engine trips: loop table per (loop, engine)
  std::vector<int32_t> xid;                       // per-engine trips: expansion-table entry per (loop, engine)
  std::vector<int64_t> tstart_of;                 // derived trip-start array per loop (and engine), -1 if none
  std::vector<uint8_t> needs_rhat;                // per loop: carries a dependency with offset > 0
  std::vector<uint8_t> fbar;                      // per loop: ends its iterations with a fallback barrier
  std::vector<uint8_t> dep_bar;                   // per dependency: barrier fallback (not waited on)
  std::vector<int32_t> dep_S;                     // per dependency: innermost common loop
  std::vector<std::array<int32_t, 6>> cse_seen;   // waits of the current straight-line segment
  std::vector<uint32_t> pe_of;                    // per (loop, engine): producer engines of cached sums
  std::unordered_map<int64_t, int64_t> anc_of;    // derived ancestor array per (consumer loop, S)
  std::vector<int32_t> by_cons, cons_next, sem_of;  // dependencies by consumer; semaphore per key
  std::vector<int64_t> inst_eng, sem_hist;        // instances per engine; history bases of one mode
};


// What the per-program pass appends, for one block of consecutive programs.
// Offsets recorded in it (into the rowptr, parent-index, pair, derived,
// path, op, plan, chunk, lane, semaphore-base, history and ordinal spaces)
// are relative to the block's start; joining the blocks shifts them.
struct Part {
  std::vector<int32_t> rowptr_host;
  std::vector<int64_t> path;
  std::vector<uint8_t> path_kind;          // per path entry: 0 parent-index offset, 1 rowptr offset
  std::vector<int32_t> op_ptr, opstop;
  std::vector<int2> rowinfo;
  std::vector<int4> ops;
  std::vector<int64_t> semhb;
  std::vector<uint8_t> semhb_mode;         // per semaphore base: its mode (history space)
  std::vector<int32_t> plan_ptr;
  std::vector<int4> plan, paux, chunks, lrec, lmeta;
  std::vector<LoopInfo> xloops;
  std::vector<uint8_t> reads_rowptr;
  std::vector<DeriveJob> jobs;
  int64_t n_ord = 0, n_derived = 0, n_pairs = 0, n_pairs_padded = 0, n_inst = 0, n_iters = 0, rowptr_len = 0;
  int64_t hist_len[kModes] = {0, 0, 0};
  bool ord_overflow = false;
  int32_t nsem_max[kModes] = {0, 0, 0}, ne_max = 0, depth_max = 0;
  int64_t n_bar_deps = 0;                  // barrier-fallback dependencies
  int64_t code_looped = 0, code_unrolled = 0;   // static instructions (code-size proxy)
  std::vector<int32_t> hoist;              // per (loop, engine) row: LICM's cached sums
  std::exception_ptr error;
};

// Appends one sweep chunk: n <= 32 lanes `recs` (program-local
// instructions, already engine-major) with their iteration copies (nullptr:
// all copy 0).
void add_chunk(const sync_batch_desc& d, int32_t x0, const ProgScratch& S, const int32_t* recs,
               const int32_t* copies, int32_t n, int32_t ncopies, std::vector<int4>& chunks,
               std::vector<int4>& lrec, std::vector<int4>& lmeta) {
  const int32_t base = (int32_t)lrec.size();
  int32_t eng[32];
  for (int32_t i = 0; i < n; ++i) eng[i] = d.instr_engine[x0 + recs[i]];
  int32_t emask = 0, head = 0;
  for (int32_t i = 0; i < n; ++i) {
    const int32_t x = recs[i], e = eng[i];
    const int32_t c = copies ? copies[i] : 0;
    emask |= 1 << e;
    if (i > 0 && eng[i - 1] != e) head = i;          // first lane of the engine's run
    const bool last = i + 1 == n || eng[i + 1] != e;
    const bool first_in_copy = c > 0 && (i == head || copies[i - 1] != c);
    lrec.push_back(make_int4(x0 + x, d.instr_latency[x0 + x], S.x_ndeps[x], S.x_dep_begin[x]));
    lmeta.push_back(make_int4(e, c, head, (first_in_copy ? LANE_ITER_START : 0) | (last ? LANE_RUN_LAST : 0)));
  }
  chunks.push_back(make_int4(base, n, ncopies, emask));
}

std::string where(int32_t p, const char* what, int64_t i) {
  return "program " + std::to_string(p) + ", " + what + " " + std::to_string(i);
}

}  // namespace

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
static void build_pieces(const sync_batch_desc& d, const HostVec<LoopInfo>& loop, const HostVec<int32_t>& rowptr,
                         const HostVec<int4>& xsem, const HostVec<DepInfo>& dep, const HostVec<int64_t>& seg,
                         const HostVec<int64_t>& semhb, const HostVec<ProgInfo>& prog, const HostVec<int64_t>& inst_off,
                         int64_t n_inst, cudaStream_t stream, sync_programs& h) {
  const int32_t P = d.n_programs;
  const int64_t NX = d.prog_instr_ptr[P];
  const double share = (double)n_inst / ((double)h.num_sms * 24.0);
  int64_t min_inst = 65536;                       // SYNCGB_SPLIT_MIN=n lowers it (tests)
  if (const char* e = std::getenv("SYNCGB_SPLIT_MIN")) min_inst = std::max<int64_t>(1, std::atoll(e));
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

static void build(const sync_batch_desc& d, int device, cudaStream_t stream, sync_programs& h) {
  // ---------------------------------------------------------- shape checks
  if (d.n_programs < 0) raise(SYNC_ERR_ARG, "n_programs < 0");
  if (d.nonalloc_policy != SYNC_NONALLOC_REJECT && d.nonalloc_policy != SYNC_NONALLOC_BARRIER)
    raise(SYNC_ERR_ARG, "nonalloc_policy is not a sync_nonalloc_policy");
  const int32_t P = d.n_programs;
  if (!d.prog_loop_ptr || !d.prog_instr_ptr || !d.prog_dep_ptr || (P > 0 && !d.prog_n_engines))
    raise(SYNC_ERR_ARG, "program CSR arrays must not be NULL");
  check_csr(d.prog_loop_ptr, P, "prog_loop_ptr");
  check_csr(d.prog_instr_ptr, P, "prog_instr_ptr");
  check_csr(d.prog_dep_ptr, P, "prog_dep_ptr");
  const int64_t NL = d.prog_loop_ptr[P], NX = d.prog_instr_ptr[P], ND = d.prog_dep_ptr[P];
  const bool div = d.eng_trip_ptr != nullptr;     // per-engine trip counts
  if (NL > 0 && (!d.loop_parent || !d.loop_pos || (!div && !d.trip_ptr)))
    raise(SYNC_ERR_ARG, "loop arrays must not be NULL");
  if (NX > 0 && (!d.instr_loop || !d.instr_pos || !d.instr_engine || !d.instr_latency))
    raise(SYNC_ERR_ARG, "instruction arrays must not be NULL");
  if (ND > 0 && (!d.dep_prod || !d.dep_cons || !d.dep_k))
    raise(SYNC_ERR_ARG, "dependency arrays must not be NULL");
  if (div && d.eng_trip_ptr[0] != 0) raise(SYNC_ERR_MALFORMED, "eng_trip_ptr[0] must be 0");
  if (NL > 0 && !div) {
    if (d.trip_ptr[0] != 0) raise(SYNC_ERR_MALFORMED, "trip_ptr[0] must be 0");
    for (int64_t l = 0; l < NL; ++l)
      if (d.trip_ptr[l + 1] < d.trip_ptr[l]) raise(SYNC_ERR_MALFORMED, "trip_ptr is not nondecreasing");
    if (d.trip_ptr[NL] > 0 && !d.trips) raise(SYNC_ERR_ARG, "trips must not be NULL");
  }

  // ------------------------------------ per-program validation and tables
  // Indexed by global loop / dependency / program / instruction id: written
  // by the block that owns the id (offsets block-relative until the join).
  HostVec<LoopInfo> loop(NL);
  HostVec<DepInfo> dep(ND);
  HostVec<ProgInfo> prog(P);
  HostVec<int64_t> inst_off(NX), dseg(ND);
  HostVec<int32_t> ddep(ND);
  HostVec<int32_t> dsem((size_t)kModes * ND);   // [kModes][n_deps]
  HostVec<int64_t> seg(ND + 1);
  HostVec<int64_t> ord_off(NX);   // per instruction: ordinal pool offset (waited producers) or -1
  // per dependency, for the simulator's semaphore numbering
  HostVec<int32_t> dep_N(ND), dep_K(ND);
  HostVec<int32_t> dep_count(ND);          // consumer instances per dependency (host copy)
  HostVec<int32_t> lflag(NL);              // per loop: carries no offset > 0 (trip register elidable)
  // per mode and instruction: {own semaphore or -1, history stride, offset,
  // per-engine wait levels}, gathered on the device into the op and lane
  // records that name the instruction
  HostVec<int4> xsem((size_t)kModes * NX);
  HostVec<int4> xcse(NX);                  // Sec. 6.2 reductions: per-instruction wait counts
  HostVec<int32_t> xlvr(NX);

  // Programs [p_begin, p_end) into `part`; erow0: their first per-engine row.
  auto run_block = [&d, div, &loop, &dep, &prog, &inst_off, &dseg, &ddep, &dsem, &seg, &ord_off, &dep_N,
                    &dep_K, &lflag, &xsem, &xcse, &xlvr, &dep_count, NX, ND](Part& part, int32_t p_begin,
                                                                            int32_t p_end, int64_t erow0) {
  auto& rowptr_host = part.rowptr_host;
  auto& path = part.path;
  auto& op_ptr = part.op_ptr;
  auto& opstop = part.opstop;
  auto& rowinfo = part.rowinfo;
  auto& ops = part.ops;
  auto& semhb = part.semhb;
  auto& plan_ptr = part.plan_ptr;
  auto& plan = part.plan;
  auto& paux = part.paux;
  auto& chunks = part.chunks;
  auto& lrec = part.lrec;
  auto& lmeta = part.lmeta;
  auto& xloops = part.xloops;
  auto& reads_rowptr = part.reads_rowptr;
  auto& jobs = part.jobs;
  auto& n_ord = part.n_ord;
  auto& n_derived = part.n_derived;
  auto& n_pairs = part.n_pairs;
  auto& n_pairs_padded = part.n_pairs_padded;
  auto& n_inst = part.n_inst;
  auto& n_iters = part.n_iters;
  auto& rowptr_len = part.rowptr_len;
  auto& hist_len = part.hist_len;
  auto push_path = [&](int64_t v, uint8_t kind) { path.push_back(v); part.path_kind.push_back(kind); };
  int64_t erow = erow0;                     // per-engine trips: first row of the program
  const bool fallback = d.nonalloc_policy == SYNC_NONALLOC_BARRIER;
  ProgScratch S;

  for (int32_t p = p_begin; p < p_end; ++p) {
    const int32_t l0 = d.prog_loop_ptr[p], x0 = d.prog_instr_ptr[p], d0 = d.prog_dep_ptr[p];
    const int32_t nl = d.prog_loop_ptr[p + 1] - l0, nx = d.prog_instr_ptr[p + 1] - x0,
                  nd = d.prog_dep_ptr[p + 1] - d0;
    const int32_t ne = d.prog_n_engines[p];
    std::fill(ord_off.begin() + x0, ord_off.begin() + x0 + nx, (int64_t)-1);
    if (nl < 1) raise(SYNC_ERR_MALFORMED, where(p, "has no top-level loop", 0));
    if (ne < 1 || ne > 32) raise(SYNC_ERR_MALFORMED, where(p, "n_engines", ne));
    const int32_t* par = d.loop_parent + l0;
    const int32_t* lpos = d.loop_pos + l0;
    S.depth.assign(nl, 0);
    S.total.assign(nl, 0);
    S.tstart_of.assign((size_t)nl * (div ? ne : 1), -1);
    S.anc_of.clear();
    S.needs_rhat.assign(nl, 0);
    S.fbar.assign(nl, 0);
    S.dep_bar.assign(nd, 0);
    S.dep_S.assign(nd, 0);
    if (par[0] != -1) raise(SYNC_ERR_MALFORMED, where(p, "loop 0 must have parent -1, loop", 0));
    int32_t depth_max = 0;
    for (int32_t l = 1; l < nl; ++l) {
      if (par[l] < 0 || par[l] >= l) raise(SYNC_ERR_MALFORMED, where(p, "parent must precede the loop, loop", l));
      if (lpos[l] < 0) raise(SYNC_ERR_MALFORMED, where(p, "negative position, loop", l));
      S.depth[l] = S.depth[par[l]] + 1;
      if (S.depth[l] > SYNC_MAX_DEPTH) raise(SYNC_ERR_MALFORMED, where(p, "nesting deeper than SYNC_MAX_DEPTH, loop", l));
      depth_max = std::max(depth_max, S.depth[l]);
    }
    // trips and iteration totals: one iteration space per loop, or per
    // (loop, engine) with per-engine trips; trip prefix sums (rowptr) appended
    auto add_space = [&](int32_t l, const int32_t* trips, int64_t want) -> LoopInfo {
      int64_t tot = 0;
      for (int64_t j = 0; j < want; ++j) {
        if (trips[j] < 0) raise(SYNC_ERR_MALFORMED, where(p, "negative trip count, loop", l));
        tot += trips[j];
      }
      if (l == 0 && tot != 1) raise(SYNC_ERR_MALFORMED, where(p, "top-level loop must run once, loop", 0));
      if (tot > kI32Max) raise(SYNC_ERR_OVERFLOW, where(p, "iterations exceed INT32_MAX, loop", l));
      LoopInfo L;
      std::memset(&L, 0, sizeof L);
      L.parent = l == 0 ? -1 : l0 + par[l];
      L.total = (int32_t)tot;
      L.n_parent = (int32_t)want;
      L.depth = S.depth[l];
      L.rowptr_off = rowptr_len;
      L.pidx_off = n_iters;
      rowptr_host.push_back(0);
      for (int64_t j = 0; j < want; ++j) rowptr_host.push_back(rowptr_host.back() + trips[j]);
      rowptr_len += want + 1;
      n_iters += tot;
      xloops.push_back(L);
      reads_rowptr.push_back(0);
      return L;
    };
    if (!div) {
      for (int32_t l = 0; l < nl; ++l) {
        const int64_t gl = l0 + l;
        const int64_t t0 = d.trip_ptr[gl], t1 = d.trip_ptr[gl + 1];
        const int64_t want = l == 0 ? 1 : S.total[par[l]];
        if (t1 - t0 != want) raise(SYNC_ERR_MALFORMED, where(p, "trip count array length != parent's iterations, loop", l));
        loop[gl] = add_space(l, d.trips + t0, want);
        S.total[l] = loop[gl].total;
      }
      S.xid.assign((size_t)nl * ne, 0);
      for (int32_t l = 0; l < nl; ++l)
        for (int32_t e = 0; e < ne; ++e) S.xid[(size_t)l * ne + e] = (int32_t)xloops.size() - nl + l;
    } else {
      S.etot.assign((size_t)nl * ne, 0);
      S.el.assign((size_t)nl * ne, LoopInfo{});
      S.xid.assign((size_t)nl * ne, 0);
      for (int32_t l = 0; l < nl; ++l)
        for (int32_t e = 0; e < ne; ++e) {
          const int64_t r = erow + (int64_t)l * ne + e;
          const int64_t t0 = d.eng_trip_ptr[r], t1 = d.eng_trip_ptr[r + 1];
          const int64_t want = l == 0 ? 1 : S.etot[(size_t)par[l] * ne + e];
          if (t1 - t0 != want)
            raise(SYNC_ERR_MALFORMED, where(p, "per-engine trip row length != parent's iterations on the engine, loop", l));
          if (want > 0 && !d.eng_trips) raise(SYNC_ERR_ARG, "eng_trips must not be NULL");
          S.xid[(size_t)l * ne + e] = (int32_t)xloops.size();
          S.el[(size_t)l * ne + e] = add_space(l, d.eng_trips + t0, want);
          S.etot[(size_t)l * ne + e] = S.el[(size_t)l * ne + e].total;
        }
      for (int32_t l = 0; l < nl; ++l) {            // engine 0's spaces stand for the loops
        loop[l0 + l] = S.el[(size_t)l * ne];
        S.total[l] = S.etot[(size_t)l * ne];
      }
      erow += (int64_t)nl * ne;
    }
    // iterations of loop l on engine e, and that iteration space
    auto tot = [&](int32_t l, int32_t e) -> int64_t { return div ? S.etot[(size_t)l * ne + e] : S.total[l]; };
    auto space = [&](int32_t l, int32_t e) -> const LoopInfo& { return div ? S.el[(size_t)l * ne + e] : loop[l0 + l]; };
    // instructions
    for (int32_t x = 0; x < nx; ++x) {
      const int64_t gx = x0 + x;
      if (d.instr_loop[gx] < 0 || d.instr_loop[gx] >= nl) raise(SYNC_ERR_MALFORMED, where(p, "loop out of range, instruction", x));
      if (d.instr_pos[gx] < 0) raise(SYNC_ERR_MALFORMED, where(p, "negative position, instruction", x));
      if (d.instr_engine[gx] < 0 || d.instr_engine[gx] >= ne) raise(SYNC_ERR_MALFORMED, where(p, "engine out of range, instruction", x));
      if (d.instr_latency[gx] < 1) raise(SYNC_ERR_MALFORMED, where(p, "latency < 1, instruction", x));
    }
    // bodies sorted by position; positions unique within a body
    S.body_ptr.assign(nl + 1, 0);
    for (int32_t x = 0; x < nx; ++x) S.body_ptr[d.instr_loop[x0 + x] + 1]++;
    for (int32_t l = 1; l < nl; ++l) S.body_ptr[par[l] + 1]++;
    for (int32_t l = 0; l < nl; ++l) S.body_ptr[l + 1] += S.body_ptr[l];
    S.keys.resize(S.body_ptr[nl]);
    {
      auto& fill = S.cons_next;                  // scratch: next free slot per body
      fill.assign(S.body_ptr.begin(), S.body_ptr.end() - 1);
      for (int32_t x = 0; x < nx; ++x)
        S.keys[fill[d.instr_loop[x0 + x]]++] = ((int64_t)d.instr_pos[x0 + x] << 32) | (uint32_t)x;
      for (int32_t l = 1; l < nl; ++l)
        S.keys[fill[par[l]]++] = ((int64_t)lpos[l] << 32) | (uint32_t)(-(l + 1));
    }
    S.body.resize(S.keys.size());
    for (int32_t l = 0; l < nl; ++l) {
      auto b = S.keys.begin() + S.body_ptr[l], e = S.keys.begin() + S.body_ptr[l + 1];
      std::sort(b, e);
      for (auto it = b; it != e; ++it) {
        if (it != b && (*it >> 32) == (*(it - 1) >> 32))
          raise(SYNC_ERR_MALFORMED, where(p, "two items share a position in the body of loop", l));
        S.body[it - S.keys.begin()] = (int32_t)(uint32_t)(*it & 0xffffffffu);
      }
    }
    // N (instructions directly in a loop body on one engine) and K (rank)
    S.rank.assign(nx, 0);
    S.nloop_eng.assign((size_t)nl * ne, 0);
    for (int32_t l = 0; l < nl; ++l)
      for (int32_t i = S.body_ptr[l]; i < S.body_ptr[l + 1]; ++i) {
        const int32_t it = S.body[i];
        if (it >= 0) S.rank[it] = ++S.nloop_eng[(size_t)l * ne + d.instr_engine[x0 + it]];
      }
    // per-program aggregates
    ProgInfo& pi = prog[p];
    std::memset(&pi, 0, sizeof pi);
    pi.ne = ne;
    pi.loop_base = l0;
    pi.le_base = (int32_t)op_ptr.size();
    __int128 agg = 0;
    for (int32_t x = 0; x < nx; ++x) {
      const int64_t n = tot(d.instr_loop[x0 + x], d.instr_engine[x0 + x]);
      agg += (__int128)n * d.instr_latency[x0 + x];
      inst_off[x0 + x] = n_inst;
      n_inst += n;
      pi.n_inst += n;
    }
    pi.agg_lat = agg > (__int128)INT64_MAX ? INT64_MAX : (int64_t)agg;
    {
      auto& per_engine = S.inst_eng;            // scratch: instances per engine
      per_engine.assign(ne, 0);
      for (int32_t x = 0; x < nx; ++x)
        per_engine[d.instr_engine[x0 + x]] += tot(d.instr_loop[x0 + x], d.instr_engine[x0 + x]);
      for (int64_t c : per_engine) if (c > kI32Max) part.ord_overflow = true;
    }
    for (int32_t e = 0; e < ne; ++e) {
      int64_t st = 0, it = 0;
      for (int32_t l = 1; l < nl; ++l) { st += tot(par[l], e); it += tot(l, e); }
      pi.eng_stmt += st;
      pi.eng_iter += it;
      pi.n_stmt = std::max(pi.n_stmt, st);
      pi.n_iter = std::max(pi.n_iter, it);
    }
    pi.divergent = div ? 1 : 0;
    S.x_ndeps.assign(nx, 0);
    S.x_dep_begin.assign(nx, d0);
    for (int m = 0; m < kModes; ++m) { S.x_own[m].assign(nx, -1); S.x_hstride[m].assign(nx, 0); S.x_koff[m].assign(nx, 0); }
    S.x_levels.assign(nx, 0);
    // dependencies: innermost common loop S, cases of Sec. 5.2, N and K
    for (int32_t k = 0; k < nd; ++k) {
      const int64_t gd = d0 + k;
      const int32_t px = d.dep_prod[gd], cx = d.dep_cons[gd], off = d.dep_k[gd];
      if (px < 0 || px >= nx || cx < 0 || cx >= nx) raise(SYNC_ERR_MALFORMED, where(p, "instruction out of range, dependency", k));
      if (off < 0) raise(SYNC_ERR_MALFORMED, where(p, "negative offset, dependency", k));
      const int32_t Pl = d.instr_loop[x0 + px], Cl = d.instr_loop[x0 + cx];
      // climb to the innermost common loop; remember the child of it on each side
      int32_t a = Pl, b = Cl, ca = -1, cb = -1;
      while (S.depth[a] > S.depth[b]) { ca = a; a = par[a]; }
      while (S.depth[b] > S.depth[a]) { cb = b; b = par[b]; }
      while (a != b) { ca = a; a = par[a]; cb = b; b = par[b]; }
      const int32_t Sl = a;
      S.dep_S[k] = Sl;
      const int32_t ppos = ca < 0 ? d.instr_pos[x0 + px] : lpos[ca];
      const int32_t cpos = cb < 0 ? d.instr_pos[x0 + cx] : lpos[cb];
      const bool forward = cpos > ppos;
      const bool same_engine = d.instr_engine[x0 + px] == d.instr_engine[x0 + cx];
      int32_t kase;
      if (ca < 0) {
        // producer directly in S: any offset; offset 0 with the consumer not
        // after the producer on the same engine can never issue (in-order)
        if (off == 0 && !forward && same_engine)
          raise(SYNC_ERR_NOT_ALLOCATABLE, where(p, "offset 0 to a later producer on the same engine, dependency", k));
        kase = CASE_PS;
      } else if (forward) {
        // a larger offset targets an earlier iteration of S: with the
        // fallback, barriers at the ends of S's iterations enforce it
        if (off != 0 && !fallback)
          raise(SYNC_ERR_NOT_ALLOCATABLE, where(p, "nested forward producer needs offset 0, dependency", k));
        kase = off == 0 ? CASE_NEST_FWD : CASE_BARRIER;
      } else {
        if (off != 1 && (!fallback || off == 0))
          raise(SYNC_ERR_NOT_ALLOCATABLE, where(p, "nested backward producer needs offset 1, dependency", k));
        kase = off == 1 ? CASE_NEST_BWD : CASE_BARRIER;
      }
      const int32_t ep = d.instr_engine[x0 + px], ec = d.instr_engine[x0 + cx];
      S.dep_bar[k] = kase == CASE_BARRIER;
      if (kase == CASE_BARRIER) {
        // no wait value, semaphore, register or derived array: its pairs stay
        // in the threshold layout (wait value 0) and S ends its iterations
        // with all-engine barriers (none at the top level, which runs once)
        if (div) raise(SYNC_ERR_ARG, where(p, "barrier fallback with per-engine trip counts, dependency", k));
        if (Sl != 0) S.fbar[Sl] = 1;
        // for the threshold and check kernels: a producer in S with an offset
        // no trip reaches, over a zero trip-start array (a derive job of
        // length 0 fills its region with zeros), so the masked wait value
        // (Eq. 2) and the required minimum are 0 on every pair
        DepInfo& D = dep[gd];
        std::memset(&D, 0, sizeof D);
        D.total = (int32_t)tot(Cl, ec);
        dep_count[gd] = D.total;
        D.kase = CASE_PS;
        D.k = (int32_t)kI32Max;
        DeriveJob J{};
        J.out = n_derived; J.n = 0; J.kind = DERIVE_TSTART;
        jobs.push_back(J);
        D.tstart = D.src = n_derived;
        n_derived += pad4(tot(Cl, ec));
        D.path = (int64_t)path.size();
        D.seg_off = n_pairs_padded;
        seg[gd] = n_pairs_padded;
        n_pairs += tot(Cl, ec);
        n_pairs_padded += pad4(tot(Cl, ec));
        dep_N[gd] = 0;
        dep_K[gd] = 0;
        continue;
      }
      if (off > 0) S.needs_rhat[Sl] = 1;           // r-hat_S's no-wait check matters
      const int32_t N = S.nloop_eng[(size_t)Pl * ne + ep];
      const int32_t K = S.rank[px];
      if ((int64_t)N * tot(Pl, ep) > kI32Max)
        raise(SYNC_ERR_OVERFLOW, where(p, "per-loop semaphore value N*iterations exceeds INT32_MAX, dependency", k));
      DepInfo& D = dep[gd];
      std::memset(&D, 0, sizeof D);
      D.total = (int32_t)tot(Cl, ec);            // consumer instances, on its engine
      dep_count[gd] = D.total;
      D.up = S.depth[Cl] - S.depth[Sl];
      D.clen = S.depth[Pl] - S.depth[Sl];
      D.kase = kase;
      D.k = off; D.N = N; D.K = K;
      D.path = (int64_t)path.size();
      // everything below is read on the consumer engine's iteration spaces
      // (Eq. (1) with that engine's loop-entry counts)
      for (int32_t l = Cl; l != Sl; l = par[l]) push_path(space(l, ec).pidx_off, 0);
      for (int32_t l = Pl; l != Sl; l = par[l]) reads_rowptr[S.xid[(size_t)l * ne + ec]] = 1;
      // derived arrays: trip starts of S, and the S-ancestors of the consumer loop
      const size_t skey = div ? (size_t)Sl * ne + ec : (size_t)Sl;
      if (S.tstart_of[skey] < 0) {
        S.tstart_of[skey] = n_derived;
        DeriveJob J{};
        J.out = n_derived; J.a = space(Sl, ec).pidx_off; J.b = space(Sl, ec).rowptr_off;
        J.n = (int32_t)tot(Sl, ec); J.kind = DERIVE_TSTART;
        jobs.push_back(J);
        n_derived += pad4(tot(Sl, ec));
      }
      D.tstart = S.tstart_of[skey];
      if (ord_off[x0 + px] < 0) {
        ord_off[x0 + px] = n_ord;
        n_ord += tot(Pl, ep);
      }
      D.ordp = ord_off[x0 + px];
      D.src = D.tstart;
      if (D.up > 0) {
        const int64_t key = ((int64_t)Cl * nl + Sl) * (div ? ne : 1) + (div ? ec : 0);
        auto f = S.anc_of.find(key);
        if (f == S.anc_of.end()) {
          DeriveJob J{};
          J.out = n_derived; J.a = D.path; J.b = 0;
          J.n = (int32_t)tot(Cl, ec); J.kind = DERIVE_ANC; J.up = D.up;
          jobs.push_back(J);
          f = S.anc_of.emplace(key, n_derived).first;
          n_derived += pad4(tot(Cl, ec));
        }
        D.src = f->second;
      }
      push_path(space(Sl, ec).pidx_off, 0);
      push_path(space(Sl, ec).rowptr_off, 1);
      {
        const size_t at = path.size();
        for (int32_t l = Pl; l != Sl; l = par[l]) push_path(space(l, ec).rowptr_off, 1);
        std::reverse(path.begin() + at, path.end());
      }
      D.seg_off = n_pairs_padded;
      seg[gd] = n_pairs_padded;
      n_pairs += tot(Cl, ec);
      n_pairs_padded += pad4(tot(Cl, ec));
      pi.n_pairs += tot(Cl, ec);
      dep_N[gd] = N;
      dep_K[gd] = K;
    }
    // loops whose trip register can be elided (Sec. 5.1: only offset-0
    // dependencies carried there, or none), and their control counts
    for (int32_t l = 1; l < nl; ++l)              // the barrier fallback's barriers (shared trips)
      if (S.fbar[l]) pi.fb_iters += tot(l, 0);
    for (int32_t k = 0; k < nd; ++k) part.n_bar_deps += S.dep_bar[k];
    // code-size proxy (the code-size comparison of Sec. 7, RQ2): the looped
    // program holds each datapath instruction once, per waited dependency
    // the per-loop wait-value ops of Table 1 and the wait, per loop and
    // engine its control (r-hat := 0 at the statement, branch, r++, r-hat++),
    // and per engine one barrier per loop that ends its iterations with a
    // fallback barrier; the unrolled program holds one instruction per
    // instance and one static wait per waited pair
    {
      int64_t waited = 0, fb_loops = 0;
      for (int32_t k = 0; k < nd; ++k) waited += S.dep_bar[k] ? 0 : 1;
      for (int32_t l = 1; l < nl; ++l) fb_loops += S.fbar[l] ? 1 : 0;
      part.code_looped += nx + (kCodeWaitOps + 1) * waited + (int64_t)ne * (kCodeLoopOps * (nl - 1) + fb_loops);
      part.code_unrolled += pi.n_inst + pi.n_pairs;
    }
    lflag[l0] = 0;
    for (int32_t l = 1; l < nl; ++l) {
      lflag[l0 + l] = S.needs_rhat[l] ? 0 : 1;
      if (S.needs_rhat[l]) continue;
      for (int32_t e = 0; e < ne; ++e) {
        pi.el_stmt += tot(par[l], e);
        pi.el_iter += tot(l, e);
      }
    }
    // semaphores that some dependency waits on, per mode, with their history
    // slots: mode 0 = one per producer instruction (one increment per
    // iteration); mode 1 = one per (loop, engine) (N increments per
    // iteration); mode 2 = one per engine (one increment per instance of the
    // engine, numbered by the instance's ordinal)
    auto& inst_eng = S.inst_eng;
    inst_eng.assign(ne, 0);
    for (int32_t x = 0; x < nx; ++x)
      inst_eng[d.instr_engine[x0 + x]] += tot(d.instr_loop[x0 + x], d.instr_engine[x0 + x]);
    auto sem_key = [&](int m, int32_t x) {
      const int32_t e = d.instr_engine[x0 + x];
      return m == 0 ? x : m == 1 ? d.instr_loop[x0 + x] * ne + e : e;
    };
    // per-engine waits: loops strictly between the top level and the producer's loop
    auto levels = [&](int32_t px) { return std::max(0, S.depth[d.instr_loop[x0 + px]] - 1); };
    for (int32_t k = 0; k < nd; ++k) {
      if (S.dep_bar[k]) continue;                  // not waited on
      const int64_t gd = d0 + k;
      S.x_levels[d.dep_cons[gd]] += levels(d.dep_prod[gd]);
      pi.pair_levels += (int64_t)levels(d.dep_prod[gd]) *
                        tot(d.instr_loop[x0 + d.dep_cons[gd]], d.instr_engine[x0 + d.dep_cons[gd]]);
    }
    // dependencies grouped by consumer, stable by dependency id (a counting
    // sort); a consumer's dependencies start at x_dep_begin (d0 if none)
    auto& by_cons = S.by_cons;
    by_cons.resize(nd);
    auto& next = S.cons_next;
    next.resize(nx);
    for (int32_t k = 0; k < nd; ++k)
      if (!S.dep_bar[k]) S.x_ndeps[d.dep_cons[d0 + k]]++;
    for (int32_t x = 0, at = 0; x < nx; ++x) {
      if (S.x_ndeps[x] > 0) S.x_dep_begin[x] = d0 + at;
      next[x] = at;
      at += S.x_ndeps[x];
    }
    int32_t nw = 0;                                // waited dependencies, grouped first
    for (int32_t k = 0; k < nd; ++k)
      if (!S.dep_bar[k]) { by_cons[next[d.dep_cons[d0 + k]]++] = k; ++nw; }
    // Sec. 6.2's reductions.  CSE: per instruction, the counts its wait ops
    // are made of when the waits of one engine in one visit of a straight-
    // line segment are taken in program order (CostTables in enc.h).  LICM:
    // per (loop, engine), the producer engines whose cached path sums the
    // engine updates at the loop's iteration starts; the bound's terms.
    {
      auto& seen = S.cse_seen;
      for (int32_t l = 0; l < nl; ++l) {
        seen.clear();
        for (int32_t i = S.body_ptr[l]; i < S.body_ptr[l + 1]; ++i) {
          const int32_t x = S.body[i];
          if (x < 0) { seen.clear(); continue; }      // a child loop ends the segment
          const int32_t ex = d.instr_engine[x0 + x];
          int4 c = make_int4(0, 0, 0, 0);
          int32_t lvr = 0;
          for (int32_t j = 0; j < S.x_ndeps[x]; ++j) {
            const int32_t k = by_cons[S.x_dep_begin[x] - d0 + j];
            const int64_t gd = d0 + k;
            const int32_t px = d.dep_prod[gd], lev = levels(px);
            const std::array<int32_t, 6> w = {ex, px, d.dep_k[gd], S.dep_S[k], d.instr_loop[x0 + px],
                                              d.instr_engine[x0 + px]};
            bool same = false, mask = false, outer = false;
            for (const auto& o : seen) {
              if (o[0] != ex) continue;
              same = same || (o[1] == w[1] && o[2] == w[2]);     // the same value
              mask = mask || (o[3] == w[3] && o[2] == w[2]);     // the same isGT(r-hat_S, k)
              outer = outer || (o[4] == w[4] && o[5] == w[5]);   // the same outer path sum
            }
            lvr += lev > 0 ? 1 : 0;
            if (!same) {
              ++c.x;
              if (mask) ++c.y;
              if (!outer) { c.z += lev > 0 ? 1 : 0; c.w += lev; }
            }
            seen.push_back(w);
          }
          xcse[x0 + x] = c;
          xlvr[x0 + x] = lvr;
        }
      }
      S.pe_of.assign((size_t)nl * ne, 0u);
      for (int32_t k = 0; k < nd; ++k) {
        if (S.dep_bar[k]) continue;
        const int64_t gd = d0 + k;
        const int32_t px = d.dep_prod[gd], cx = d.dep_cons[gd];
        const int32_t Pl = d.instr_loop[x0 + px], ec = d.instr_engine[x0 + cx];
        if (S.depth[Pl] > 1) pi.lv_pairs += tot(d.instr_loop[x0 + cx], ec);
        for (int32_t l = par[Pl]; l > 0; l = par[l]) S.pe_of[(size_t)l * ne + ec] |= 1u << d.instr_engine[x0 + px];
      }
    }
    auto& sem_of = S.sem_of;
    auto& sem_hist = S.sem_hist;
    sem_of.resize(std::max(nx, nl * ne));
    for (int m = 0; m < kModes; ++m) {
      std::fill(sem_of.begin(), sem_of.end(), -1);
      sem_hist.clear();
      for (int32_t k = 0; k < nd; ++k) {
        if (S.dep_bar[k]) continue;                // not waited on: no semaphore of its own
        const int64_t gd = d0 + k;
        const int32_t px = d.dep_prod[gd];
        const int32_t Pl = d.instr_loop[x0 + px];
        const int32_t key = sem_key(m, px);
        if (sem_of[key] < 0) {
          sem_of[key] = (int32_t)sem_hist.size();
          sem_hist.push_back(hist_len[m]);
          const int32_t ep = d.instr_engine[x0 + px];
          hist_len[m] += m == 0 ? tot(Pl, ep) : m == 1 ? dep_N[gd] * tot(Pl, ep) : inst_eng[ep];
        }
      }
      pi.nsem[m] = (int32_t)sem_hist.size();
      pi.semhb_off[m] = (int32_t)semhb.size();
      semhb.insert(semhb.end(), sem_hist.begin(), sem_hist.end());
      part.semhb_mode.insert(part.semhb_mode.end(), sem_hist.size(), (uint8_t)m);
      for (int32_t x = 0; x < nx; ++x) {
        const int32_t l = d.instr_loop[x0 + x];
        const int32_t s = sem_of[sem_key(m, x)];
        S.x_own[m][x] = s;
        if (s >= 0) {
          S.x_hstride[m][x] = m == 0 ? 1 : m == 1 ? S.nloop_eng[(size_t)l * ne + d.instr_engine[x0 + x]] : -1;
          S.x_koff[m][x] = m == 0 ? 1 : m == 1 ? S.rank[x] : 0;
        }
        xsem[(size_t)m * NX + x0 + x] =
            make_int4(s, S.x_hstride[m][x], S.x_koff[m][x], m == 2 ? S.x_levels[x] : 0);
      }
      for (int32_t i = 0; i < nw; ++i) {
        const int64_t gd = d0 + by_cons[i];
        dsem[(size_t)m * ND + d0 + i] = sem_of[sem_key(m, d.dep_prod[gd])];
        if (m == 0) { dseg[d0 + i] = seg[gd]; ddep[d0 + i] = (int32_t)gd; }
      }
      for (int32_t i = nw; i < nd; ++i) {          // slots of barrier-fallback dependencies: unused
        dsem[(size_t)m * ND + d0 + i] = -1;
        if (m == 0) { dseg[d0 + i] = 0; ddep[d0 + i] = (int32_t)(d0 + i); }
      }
    }
    // per-(loop, engine) op records: own instructions and child loops in body
    // order, then an END record
    for (int32_t l = 0; l < nl; ++l)
      for (int32_t e = 0; e < ne; ++e) {
        const int32_t first = (int32_t)ops.size();
        op_ptr.push_back(first);
        bool has_loop = false;
        for (int32_t i = S.body_ptr[l]; i < S.body_ptr[l + 1]; ++i) {
          const int32_t it = S.body[i];
          if (it < 0) {
            const int32_t m = -it - 1;
            const int64_t rp = space(m, e).rowptr_off;
            ops.push_back(make_int4(OP_LOOP, pi.le_base + m * ne, (int32_t)(uint32_t)(rp & 0xffffffffu),
                                    (int32_t)(rp >> 32)));
            has_loop = true;
          } else if (d.instr_engine[x0 + it] == e) {
            ops.push_back(make_int4(x0 + it, d.instr_latency[x0 + it], S.x_ndeps[it], S.x_dep_begin[it]));
          }
        }
        const int32_t end_idx = (int32_t)ops.size();
        ops.push_back(make_int4(OP_END, 0, 0, 0));
        rowinfo.push_back(make_int2(end_idx, (has_loop ? 1 : 0) | (lflag[l0 + l] ? 2 : 0) | (S.fbar[l] ? 4 : 0)));
        const int32_t nh = __builtin_popcount(S.pe_of[(size_t)l * ne + e]);
        part.hoist.push_back(nh);
        pi.licm_upd += (int64_t)nh * tot(l, e);
        // next LOOP or END record at or after each record of the row
        opstop.resize(ops.size());
        int32_t next = end_idx;
        for (int32_t r = end_idx; r >= first; --r) {
          if (ops[r].x < 0) next = r;
          opstop[r] = next;
        }
      }
    // program-order sweep plan: per loop, its body cut at child loops into
    // straight-line segments, each segment in chunks of <= 32 engine-sorted lanes
    const size_t plan_first_loop = plan_ptr.size(), plan_first_item = plan.size();
    for (int32_t l = 0; l < nl; ++l) {
      plan_ptr.push_back((int32_t)plan.size());
      int32_t seg0 = S.body_ptr[l], nseg = 0, nloops = 0;   // current segment: body[seg0 .. i)
      for (int32_t i = S.body_ptr[l]; i <= S.body_ptr[l + 1]; ++i) {
        const bool at_end = i == S.body_ptr[l + 1];
        const int32_t it = at_end ? -1 : S.body[i];
        if (!at_end && it >= 0) continue;
        if (i > seg0) {
          ++nseg;
          const int32_t first_chunk = (int32_t)chunks.size();
          for (int32_t b = seg0; b < i; b += 32) {
            // up to 32 records, engine-major and in body order within an
            // engine (a counting sort by engine)
            const int32_t n = std::min<int32_t>(32, i - b);
            int32_t cnt[33] = {0}, piece[32];
            for (int32_t j = 0; j < n; ++j) ++cnt[d.instr_engine[x0 + S.body[b + j]] + 1];
            for (int32_t e = 0; e < ne; ++e) cnt[e + 1] += cnt[e];
            for (int32_t j = 0; j < n; ++j) piece[cnt[d.instr_engine[x0 + S.body[b + j]]]++] = S.body[b + j];
            add_chunk(d, x0, S, piece, nullptr, n, 1, chunks, lrec, lmeta);
          }
          plan.push_back(make_int4(ITEM_SEG, first_chunk, (int32_t)chunks.size() - first_chunk, -1));
        }
        seg0 = i + 1;
        if (!at_end) {
          ++nloops;
          plan.push_back(make_int4(ITEM_LOOP, l0 + (-it - 1), lflag[l0 + (-it - 1)], 0));
        }
      }
      // a short body with no child loop: a template of several iterations
      const int32_t L = S.body_ptr[l + 1] - S.body_ptr[l];
      if (nloops == 0 && nseg == 1 && L >= 1 && L <= 16) {
        const int32_t k = 32 / L;
        int32_t recs[32], copies[32], n = 0;
        for (int32_t e = 0; e < ne; ++e)
          for (int32_t c = 0; c < k; ++c)
            for (int32_t i = S.body_ptr[l]; i < S.body_ptr[l + 1]; ++i)
              if (d.instr_engine[x0 + S.body[i]] == e) { recs[n] = S.body[i]; copies[n++] = c; }
        plan.back().w = (int32_t)chunks.size();
        add_chunk(d, x0, S, recs, copies, n, k, chunks, lrec, lmeta);
      }
    }
    // per loop statement, what the walker needs without further lookups:
    // the child's rowptr offset, and the chunk that holds its whole body
    // (barrier-free: the multi-iteration template if there is one), or -1
    paux.resize(plan.size(), make_int4(0, 0, -1, -1));
    for (size_t i = plan_first_item; i < plan.size(); ++i) {
      if (plan[i].x != ITEM_LOOP) continue;
      const int32_t m = plan[i].y - l0;
      const size_t b = plan_ptr[plan_first_loop + m];
      const size_t e = m + 1 < nl ? (size_t)plan_ptr[plan_first_loop + m + 1] : plan.size();
      int32_t bf = -1, bb = -1;
      if (e - b == 1 && plan[b].x == ITEM_SEG) {
        if (plan[b].z == 1) bf = bb = plan[b].y;
        if (plan[b].w >= 0) bf = plan[b].w;
      }
      const int64_t rp = loop[l0 + m].rowptr_off;
      paux[i] = make_int4((int32_t)(uint32_t)(rp & 0xffffffffu), (int32_t)(rp >> 32), bf, bb);
    }
    for (int m = 0; m < kModes; ++m) part.nsem_max[m] = std::max(part.nsem_max[m], pi.nsem[m]);
    part.ne_max = std::max(part.ne_max, ne);
    part.depth_max = std::max(part.depth_max, depth_max);
    if ((int64_t)ops.size() > kI32Max) raise(SYNC_ERR_OVERFLOW, "op records exceed INT32_MAX entries");
  }
  };

  // Blocks of consecutive programs of about equal work, one per thread.
  std::vector<int64_t> work(P), erow_of(P + 1, 0);
  for (int32_t p = 0; p < P; ++p) {
    const int64_t nl = d.prog_loop_ptr[p + 1] - d.prog_loop_ptr[p];
    const int64_t ne = std::max<int64_t>(1, std::min<int64_t>(32, d.prog_n_engines[p]));
    const int64_t trips = div || nl == 0 ? nl * ne : d.trip_ptr[d.prog_loop_ptr[p + 1]] - d.trip_ptr[d.prog_loop_ptr[p]];
    work[p] = 16 + (nl + d.prog_instr_ptr[p + 1] - d.prog_instr_ptr[p]) * ne + (d.prog_dep_ptr[p + 1] - d.prog_dep_ptr[p]) +
              std::max<int64_t>(trips, 0);
    erow_of[p + 1] = erow_of[p] + nl * d.prog_n_engines[p];
  }
  const int n_threads = load_threads(P);
  std::vector<int32_t> cut(n_threads + 1, P);
  {
    int64_t total = 0;
    for (int64_t w : work) total += w;
    int64_t acc = 0;
    int b = 1;
    cut[0] = 0;
    for (int32_t p = 0; p < P && b < n_threads; ++p) {
      acc += work[p];
      while (b < n_threads && acc * n_threads >= total * b) cut[b++] = p + 1;
    }
  }
  std::vector<Part> parts(n_threads);
  {
    std::vector<std::thread> pool;
    for (int t = 0; t < n_threads; ++t) {
      auto job = [&, t] {
        try {
          run_block(parts[t], cut[t], cut[t + 1], erow_of[cut[t]]);
        } catch (...) {
          parts[t].error = std::current_exception();
        }
      };
      if (t + 1 < n_threads) pool.emplace_back(job); else job();
    }
    for (auto& th : pool) th.join();
    for (auto& pt : parts)
      if (pt.error) std::rethrow_exception(pt.error);
  }

  // ------------------------------------------------- join the blocks
  // Each block's bases in every space are the sizes of the blocks before it;
  // every block then copies itself into place, shifting the offsets it holds.
  struct Base {
    int64_t rowptr, iters, pairs, derived, path, ord, inst, hist[kModes];
    int64_t rowptr_host, ops, rows, plan, chunks, lanes, semhb, xloops, jobs, opstop, pairs_raw;
  };
  std::vector<Base> base(n_threads + 1);
  std::memset(base.data(), 0, sizeof(Base) * base.size());
  for (int t = 0; t < n_threads; ++t) {
    const Part& pt = parts[t];
    Base nb = base[t];
    nb.rowptr += pt.rowptr_len; nb.iters += pt.n_iters; nb.pairs += pt.n_pairs_padded;
    nb.derived += pt.n_derived; nb.path += (int64_t)pt.path.size(); nb.ord += pt.n_ord; nb.inst += pt.n_inst;
    for (int m = 0; m < kModes; ++m) nb.hist[m] += pt.hist_len[m];
    nb.rowptr_host += (int64_t)pt.rowptr_host.size(); nb.ops += (int64_t)pt.ops.size();
    nb.rows += (int64_t)pt.op_ptr.size(); nb.plan += (int64_t)pt.plan.size(); nb.chunks += (int64_t)pt.chunks.size();
    nb.lanes += (int64_t)pt.lrec.size(); nb.semhb += (int64_t)pt.semhb.size(); nb.xloops += (int64_t)pt.xloops.size();
    nb.jobs += (int64_t)pt.jobs.size(); nb.opstop += (int64_t)pt.opstop.size(); nb.pairs_raw += pt.n_pairs;
    base[t + 1] = nb;
    for (int m = 0; m < kModes; ++m) h.nsem_max[m] = std::max(h.nsem_max[m], pt.nsem_max[m]);
    h.ne_max = std::max(h.ne_max, pt.ne_max);
    h.depth_max = std::max(h.depth_max, pt.depth_max);
  }
  const Base& all = base[n_threads];
  if (all.ops > kI32Max) raise(SYNC_ERR_OVERFLOW, "op records exceed INT32_MAX entries");
  HostVec<int32_t> rowptr_host(all.rowptr_host);
  HostVec<int64_t> path(all.path);
  HostVec<int32_t> op_ptr(all.rows), opstop(all.opstop);
  HostVec<int2> rowinfo(all.rows);
  HostVec<int32_t> hoist(all.rows);
  HostVec<int4> ops(all.ops);
  HostVec<int64_t> semhb(all.semhb);
  HostVec<int32_t> plan_ptr(NL);             // one entry per loop; the blocks own consecutive loops
  HostVec<int4> plan(all.plan), paux(all.plan), chunks(all.chunks), lrec(all.lanes), lmeta(all.lanes);
  HostVec<LoopInfo> xloops(all.xloops);
  HostVec<uint8_t> reads_rowptr(all.xloops);
  HostVec<DeriveJob> jobs(all.jobs);
  const int64_t n_ord = all.ord, n_derived = all.derived, n_pairs = all.pairs_raw, n_pairs_padded = all.pairs;
  const int64_t n_inst = all.inst, n_iters = all.iters;
  std::vector<int64_t> hist_len(all.hist, all.hist + kModes);
  bool ord_overflow = false;
  for (const Part& pt : parts) ord_overflow = ord_overflow || pt.ord_overflow;
  h.n_bar_deps = 0;
  for (const Part& pt : parts) {
    h.n_bar_deps += pt.n_bar_deps;
    h.sz.code_bytes_looped += SYNC_CODE_BYTES_PER_INSTR * pt.code_looped;
    h.sz.code_bytes_unrolled += SYNC_CODE_BYTES_PER_INSTR * pt.code_unrolled;
  }
  auto join_block = [&](int t) {
    Part& pt = parts[t];
    const Base& B = base[t];
    const int32_t b_ops = (int32_t)B.ops, b_rows = (int32_t)B.rows, b_plan = (int32_t)B.plan;
    const int32_t b_chunks = (int32_t)B.chunks, b_lanes = (int32_t)B.lanes, b_semhb = (int32_t)B.semhb;
    // indexed by id: the block's programs, loops, instructions, dependencies
    for (int32_t p = cut[t]; p < cut[t + 1]; ++p) {
      ProgInfo& pi = prog[p];
      pi.le_base += b_rows;
      for (int m = 0; m < kModes; ++m) pi.semhb_off[m] += b_semhb;
      for (int32_t l = d.prog_loop_ptr[p]; l < d.prog_loop_ptr[p + 1]; ++l) {
        loop[l].rowptr_off += B.rowptr;
        loop[l].pidx_off += B.iters;
      }
      for (int32_t x = d.prog_instr_ptr[p]; x < d.prog_instr_ptr[p + 1]; ++x) {
        inst_off[x] += B.inst;
        if (ord_off[x] >= 0) ord_off[x] += B.ord;
      }
      for (int32_t k = d.prog_dep_ptr[p]; k < d.prog_dep_ptr[p + 1]; ++k) {
        DepInfo& D = dep[k];
        D.seg_off += B.pairs;
        D.src += B.derived;
        D.tstart += B.derived;
        D.path += B.path;
        D.ordp += B.ord;
        seg[k] += B.pairs;
        dseg[k] += B.pairs;
      }
    }
    // appended: into place, shifting the offsets they hold
    std::copy(pt.rowptr_host.begin(), pt.rowptr_host.end(), rowptr_host.begin() + B.rowptr_host);
    for (size_t i = 0; i < pt.path.size(); ++i)
      path[B.path + i] = pt.path[i] + (pt.path_kind[i] ? B.rowptr : B.iters);
    for (size_t i = 0; i < pt.op_ptr.size(); ++i) op_ptr[B.rows + i] = pt.op_ptr[i] + b_ops;
    for (size_t i = 0; i < pt.rowinfo.size(); ++i) {
      rowinfo[B.rows + i] = make_int2(pt.rowinfo[i].x + b_ops, pt.rowinfo[i].y);
      hoist[B.rows + i] = pt.hoist[i];
    }
    for (size_t i = 0; i < pt.opstop.size(); ++i) opstop[B.opstop + i] = pt.opstop[i] + b_ops;
    for (size_t i = 0; i < pt.ops.size(); ++i) {
      int4 v = pt.ops[i];
      if (v.x == OP_LOOP) {
        const int64_t rp = (int64_t)(((uint64_t)(uint32_t)v.w << 32) | (uint32_t)v.z) + B.rowptr;
        v = make_int4(OP_LOOP, v.y + b_rows, (int32_t)(uint32_t)(rp & 0xffffffffu), (int32_t)(rp >> 32));
      }
      ops[B.ops + i] = v;
    }
    for (size_t i = 0; i < pt.semhb.size(); ++i) semhb[B.semhb + i] = pt.semhb[i] + B.hist[pt.semhb_mode[i]];
    const int32_t l_first = d.prog_loop_ptr[cut[t]];
    for (size_t i = 0; i < pt.plan_ptr.size(); ++i) plan_ptr[l_first + i] = pt.plan_ptr[i] + b_plan;
    for (size_t i = 0; i < pt.plan.size(); ++i) {
      int4 v = pt.plan[i];
      if (v.x == ITEM_SEG) {
        v.y += b_chunks;
        if (v.w >= 0) v.w += b_chunks;
      }
      plan[B.plan + i] = v;
      int4 x = pt.paux[i];
      if (v.x == ITEM_LOOP) {
        const int64_t rp = (int64_t)(((uint64_t)(uint32_t)x.y << 32) | (uint32_t)x.x) + B.rowptr;
        x = make_int4((int32_t)(uint32_t)(rp & 0xffffffffu), (int32_t)(rp >> 32), x.z >= 0 ? x.z + b_chunks : -1,
                      x.w >= 0 ? x.w + b_chunks : -1);
      }
      paux[B.plan + i] = x;
    }
    for (size_t i = 0; i < pt.chunks.size(); ++i) {
      const int4 v = pt.chunks[i];
      chunks[B.chunks + i] = make_int4(v.x + b_lanes, v.y, v.z, v.w);
    }
    std::copy(pt.lrec.begin(), pt.lrec.end(), lrec.begin() + B.lanes);
    std::copy(pt.lmeta.begin(), pt.lmeta.end(), lmeta.begin() + B.lanes);
    for (size_t i = 0; i < pt.xloops.size(); ++i) {
      LoopInfo L = pt.xloops[i];
      L.rowptr_off += B.rowptr;
      L.pidx_off += B.iters;
      xloops[B.xloops + i] = L;
    }
    std::copy(pt.reads_rowptr.begin(), pt.reads_rowptr.end(), reads_rowptr.begin() + B.xloops);
    for (size_t i = 0; i < pt.jobs.size(); ++i) {
      DeriveJob J = pt.jobs[i];
      J.out += B.derived;
      if (J.kind == DERIVE_TSTART) {
        J.a += B.iters;
        J.b += B.rowptr;
      } else {
        J.a += B.path;
      }
      jobs[B.jobs + i] = J;
    }
    Part released;
    std::swap(pt, released);                     // the block's memory goes with it
  };
  {
    std::vector<std::thread> pool;
    for (int t = 0; t + 1 < n_threads; ++t) pool.emplace_back(join_block, t);
    join_block(n_threads - 1);
    for (auto& th : pool) th.join();
  }
  op_ptr.push_back((int32_t)ops.size());
  plan_ptr.push_back((int32_t)plan.size());
  seg[ND] = n_pairs_padded;

  // tile tables: table[t] = largest i < n with start(i) <= t * kTilePairs
  // (start nondecreasing), one extra entry n-1; all three in one pool of
  // threads, each table cut into slices of about 256k steps
  std::vector<std::thread> tile_pool;
  struct JoinAll {
    std::vector<std::thread>& v;
    ~JoinAll() { for (auto& th : v) if (th.joinable()) th.join(); }
  } tile_join{tile_pool};                      // also when something below throws
  auto tile_table = [&tile_pool, n_threads](std::vector<int32_t>& table, int64_t n_tiles, int64_t n, auto start) {
    table.assign(n_tiles + 1, n > 0 ? (int32_t)(n - 1) : 0);
    if (n == 0) return;
    auto fill = [&table, n, start](int64_t t0, int64_t t1) {
      int64_t lo = 0, hi = n - 1;                // largest i with start(i) <= t0 * kTilePairs
      while (lo < hi) {
        const int64_t mid = (lo + hi + 1) / 2;
        if (start(mid) <= t0 * kTilePairs) lo = mid; else hi = mid - 1;
      }
      for (int64_t t = t0, i = lo; t < t1; ++t) {
        while (i + 1 < n && start(i + 1) <= t * kTilePairs) ++i;
        table[t] = (int32_t)i;
      }
    };
    const int64_t nt = std::max<int64_t>(1, std::min<int64_t>(n_threads, (n_tiles + n) / (1 << 18)));
    for (int64_t k = 0; k < nt; ++k) tile_pool.emplace_back(fill, n_tiles * k / nt, n_tiles * (k + 1) / nt);
  };
  std::vector<int32_t> tile_first, tile_job, tile_loop;
  tile_table(tile_first, (n_pairs_padded + kTilePairs - 1) / kTilePairs, ND, [&seg](int64_t i) { return seg[i]; });
  tile_table(tile_job, (n_derived + kTilePairs - 1) / kTilePairs, (int64_t)jobs.size(),
             [&jobs](int64_t i) { return jobs[i].out; });
  tile_table(tile_loop, (n_iters + kTilePairs - 1) / kTilePairs, (int64_t)xloops.size(),
             [&xloops](int64_t i) { return xloops[i].pidx_off; });
  // programs in descending order of simulated work, equal work in program
  // order: a stable least-significant-digit radix sort (11-bit digits) of
  // the works' complements
  std::vector<int32_t> order(P);
  {
    std::vector<uint64_t> key(P);
    uint64_t all_bits = 0;
    for (int32_t p = 0; p < P; ++p) {
      const int64_t w = prog[p].n_inst + prog[p].n_pairs + (prog[p].n_stmt + prog[p].n_iter) * prog[p].ne;
      key[p] = ~(uint64_t)w;                     // w >= 0: larger work, smaller key
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
      order.swap(tmp);
    }
  }
  for (auto& th : tile_pool) th.join();      // the tables are read from here on

  h.sz.n_pairs = n_pairs;
  h.sz.n_pairs_padded = n_pairs_padded;
  h.sz.n_instances = n_inst;
  h.sz.n_loop_iters = n_iters;
  h.sz.n_programs = P;
  h.sz.n_loops = (int32_t)NL;
  h.sz.n_instrs = (int32_t)NX;
  h.sz.n_deps = (int32_t)ND;
  {
    // of the path pool the kernels read only the rowptr offsets from S's
    // child down to a nested producer's loop (clen per dependency); the
    // pidx offsets are read at load time only
    int64_t path_read = 0;
    for (int64_t d = 0; d < ND; ++d) path_read += dep[d].clen;
    int64_t sb = (int64_t)ND * (int64_t)sizeof(DepInfo) + 8 * (ND + 1) + 8 * path_read +
                 4 * (int64_t)tile_first.size();
    sb += 4 * n_derived;
    for (size_t l = 0; l < xloops.size(); ++l)
      if (reads_rowptr[l]) sb += 4 * ((int64_t)xloops[l].n_parent + 1);
    h.sz.struct_bytes = sb;
  }
  h.seg_host = std::move(seg);
  h.ord_off_host = std::move(ord_off);
  h.n_ord = n_ord;
  h.ord_overflow = ord_overflow;
  h.count_host = std::move(dep_count);
  h.n_chunks = n_pairs_padded / kChunk;

  // ---------------------------------------------------------------- device
  cuda_check(cudaSetDevice(device), "cudaSetDevice");
  h.device = device;
  cuda_check(cudaDeviceGetAttribute(&h.num_sms, cudaDevAttrMultiProcessorCount, device), "device attributes");
  h.loop = h.upload(loop, stream, "loop table");
  h.rowptr = h.upload(rowptr_host, stream, "rowptr");
  h.pidx = h.alloc<int32_t>(n_iters, "parent indices");
  h.dep = h.upload(dep, stream, "dependency table");
  h.seg = h.upload(h.seg_host, stream, "segment offsets");
  h.tile_first = h.upload(tile_first, stream, "tile table");
  h.path = h.upload(path, stream, "path pool");
  h.derived = h.alloc<int32_t>(n_derived, "derived trip starts and ancestors");
  DeriveJob* d_jobs = h.upload(jobs, stream, "derive jobs");
  int32_t* d_tile_job = h.upload(tile_job, stream, "derive tile table");
  int32_t* d_tile_loop = h.upload(tile_loop, stream, "loop tile table");
  h.prog = h.upload(prog, stream, "program table");
  h.order = h.upload(order, stream, "program order");
  h.op_ptr = h.upload(op_ptr, stream, "op record offsets");
  h.rowinfo = h.upload(rowinfo, stream, "row info");
  h.cost.hoist = h.upload(hoist, stream, "cached-sum counts");
  h.cost.xcse = h.upload(xcse, stream, "wait counts with CSE");
  h.cost.xlvr = h.upload(xlvr, stream, "cached-sum reads");
  h.ops = h.upload(ops, stream, "op records");
  h.opstop = h.upload(opstop, stream, "op stops");
  h.opsem = h.alloc<int4>(kModes * (int64_t)ops.size(), "op semaphore records");
  {
    h.dsem = h.upload(dsem, stream, "dependency semaphores");
  }
  h.n_ops = (int64_t)ops.size();
  h.dseg = h.upload(dseg, stream, "dependency segments");
  h.ddep = h.upload(ddep, stream, "consumer-grouped dependency ids");
  h.semhb = h.upload(semhb, stream, "semaphore history bases");
  h.inst_off = h.upload(inst_off, stream, "instance offsets");
  h.hist = h.alloc<int32_t>(*std::max_element(hist_len.begin(), hist_len.end()), "semaphore history");
  for (int m = 0; m < kModes; ++m) h.hist_len[m] = hist_len[m];
  h.next_slot = h.alloc<int32_t>(1, "program-slot counter");
  h.fallback = h.alloc<int32_t>((int64_t)P + 1, "fallback list");
  h.plan_ptr = h.upload(plan_ptr, stream, "sweep plan offsets");
  h.lflag = h.upload(lflag, stream, "loop flags");
  h.plan = h.upload(plan, stream, "sweep plan");
  h.paux = h.upload(paux, stream, "sweep loop statements");
  h.chunk = h.upload(chunks, stream, "sweep chunks");
  h.lrec = h.upload(lrec, stream, "sweep lanes");
  h.lmeta = h.upload(lmeta, stream, "sweep lane meta");
  h.lsem = h.alloc<int4>(kModes * (int64_t)lrec.size(), "sweep lane semaphores");
  const int4* d_xsem = h.upload(xsem, stream, "instruction semaphore records");
  h.n_lanes = (int64_t)lrec.size();
  LoopInfo* d_xloops = h.upload(xloops, stream, "iteration spaces");
  h.divergent = div;
  build_pieces(d, loop, rowptr_host, xsem, dep, h.seg_host, semhb, prog, inst_off, n_inst, stream, h);
  cuda_check(launch_expand(d_xloops, d_tile_loop, h.rowptr, h.pidx, n_iters, h.num_sms, stream), "expand");
  cuda_check(launch_sem_records(d_xsem, NX, h.ops, h.n_ops, h.lrec, h.n_lanes, h.opsem, h.lsem, h.num_sms, stream),
             "semaphore records");
  cuda_check(launch_derive(d_jobs, d_tile_job, h.rowptr, h.pidx, h.path, h.derived, n_derived, h.num_sms, stream),
             "derive");
  cuda_check(cudaStreamSynchronize(stream), "load");
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
  std::memcpy(offsets, h->seg_host.data(), h->seg_host.size() * sizeof(int64_t));
  if (counts) std::memcpy(counts, h->count_host.data(), h->count_host.size() * sizeof(int32_t));
  return SYNC_OK;
}

static ThrArgs thr_args(const sync_programs* h, sync_thr_mode mode) {
  ThrArgs a;
  a.dep = h->dep; a.derived = h->derived; a.ord = h->ord; a.seg = h->seg; a.tile_first = h->tile_first;
  a.path = h->path; a.rowptr = h->rowptr; a.pidx = h->pidx; a.n_chunks = h->n_chunks; a.mode = mode;
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
  int64_t* off = m->upload(h->ord_off_host, s, "engine-stream position offsets");
  cuda_check(launch_ordinals(h->prog, h->order, h->sz.n_programs, h->ne_max, h->op_ptr, h->ops, h->rowptr, off, ord,
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

const char* sync_last_error(void) { return g_err.c_str(); }

int64_t sync_kernel_launches(void) { return g_launches.load(std::memory_order_relaxed); }

}  // extern "C"
