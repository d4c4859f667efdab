// Schedule simulator, program-order sweep: one warp per program.
//
// Under a common loop tree every engine meets the same loop statements and
// iteration boundaries, so one walker per program can visit the tree once for
// all engines.  The body of each loop is cut at its child loops into
// straight-line segments; a segment is taken as one chunk of up to 32 datapath
// records (more chunks if longer), or -- barrier-free, for a short innermost
// body -- as several consecutive iterations at once.  The chunk's lanes are
// ordered engine-major, so each engine's events form a run of lanes:
//   - an engine's cursor obeys t' = max(t + A, B) per event (A its costs,
//     B the time its waits are satisfied plus the issue interval), maps that
//     compose associatively, so a segmented 5-step warp scan gives every
//     event the cursor before it; issue = max(cursor + wait ops, ready) and
//     in-order retirement is a segmented max-scan of issue + latency;
//   - a wait on a semaphore whose threshold increment happened in an earlier
//     chunk reads its retire time from the history array; an increment inside
//     the chunk is the k-th lane of the semaphore's lanes (increments come in
//     lane order), and these in-chunk waits are solved by repeating the scans
//     until no time changes (a least fixed point of the max-plus system;
//     times only grow, a cycle never settles and is a deadlock);
//   - a threshold beyond every increment up to this chunk points forward in
//     program order: the program is handed to the per-engine kernel.
// Barriers (barrier scheme) are a warp maximum of the engines' drained times.
// Per-engine cursor, last retire and instance count live in shared memory,
// read by the engine's lanes and written back by the last lane of its run.
#include "enc.h"

namespace syncgb {
namespace {

constexpr int kWarps = 8;                   // programs (warps) per CTA
constexpr int kMaxIntra = 4;                // in-chunk waits per lane before falling back
constexpr unsigned kFull = 0xffffffffu;
constexpr int32_t kNeg = -1;                // -infinity of the cursor maps (cursors, costs >= 0)
constexpr int SIM_FALLBACK = 9;             // internal: handed to the per-engine kernel

struct Frame { int32_t loop, item, g, g_end; };

// Shared memory of one warp (program), 16-byte aligned.
__host__ __device__ __forceinline__ size_t warp_bytes(int sem_cap, int frame_depth) {
  const size_t per = (size_t)20 * sem_cap + sizeof(Frame) * (size_t)frame_depth + 3 * 4 * 32;
  return (per + 15) & ~(size_t)15;
}

__device__ __forceinline__ unsigned long long sat_add(unsigned long long a, unsigned long long b) {
  const unsigned long long r = a + b;
  return r < a ? ~0ull : r;
}
__device__ __forceinline__ unsigned long long sat_mul(unsigned long long a, unsigned long long b) {
  return __umul64hi(a, b) ? ~0ull : a * b;
}
__device__ __forceinline__ unsigned lanemask_le() {
  unsigned m;
  asm("mov.u32 %0, %%lanemask_le;" : "=r"(m));
  return m;
}
// Lane of the k-th (1-based) set bit of m.
__device__ __forceinline__ int kth_bit(unsigned m, int k) {
  for (int i = 1; i < k; ++i) m &= m - 1;
  return __ffs(m) - 1;
}

__device__ __forceinline__ unsigned long long inst_term(int32_t issue, int32_t retire, uint32_t e,
                                                        uint32_t n) {
  uint32_t x = ((uint32_t)issue ^ (n * 0x9E3779B9u + e)) * 0x85EBCA6Bu;
  x ^= x >> 13;
  uint32_t y = ((uint32_t)retire ^ (n * 0xC2B2AE35u + e)) * 0x27D4EB2Fu;
  y ^= y >> 15;
  return ((unsigned long long)x << 32) | y;
}

template <bool BB>
__device__ __forceinline__ unsigned long long time_bound(const ProgInfo& pi, const sync_sim_params& q,
                                                         int32_t cwait) {
  typedef unsigned long long u64;
  u64 b = sat_add((u64)pi.agg_lat, sat_mul((u64)q.ii, (u64)pi.n_inst));
  if (BB) {
    b = sat_add(b, sat_mul(sat_mul((u64)pi.ne, (u64)pi.n_iter), (u64)q.c_branch));
    b = sat_add(b, sat_mul((u64)(pi.n_stmt + pi.n_iter), (u64)q.c_barrier));
  } else {
    b = sat_add(b, sat_mul((u64)cwait, (u64)pi.n_pairs));
    const u64 ctl = sat_add(sat_mul((u64)pi.n_stmt, (u64)q.c_regop),
                            sat_mul((u64)pi.n_iter, (u64)q.c_branch + 2ull * (u64)q.c_regop));
    b = sat_add(b, sat_mul((u64)pi.ne, ctl));
  }
  return b;
}

struct WarpSmem {
  int32_t* t;          // [32] engine cursors
  int32_t* lr;         // [32] engine last retire
  int32_t* nn;         // [32] engine datapath instances so far
  int32_t* semv;       // [cap] increments processed
  int64_t* semhb;      // [cap] history base
  uint32_t* grp;       // [cap] lanes of the current chunk that increment it
  int32_t* tag;        // [cap] chunk that wrote grp
  Frame* frames;       // [depth]
};

// One chunk: `copies` iterations (g .. g+copies-1) of a segment's records.
// Returns 0, SYNC_PROG_DEADLOCK or SIM_FALLBACK.
template <int MODE, bool BB, bool TL>
__device__ __forceinline__ int run_chunk(const SweepArgs& a, const WarpSmem& S, const int4 ch, int32_t g,
                                         int32_t copies, int32_t ctag, int lane,
                                         unsigned long long& chk) {
  const int32_t cwait = MODE == SYNC_THR_PERLOOP ? a.prm.c_wait_ops_perloop : a.prm.c_wait_ops_count;
  const int32_t iter_cost = BB ? a.prm.c_branch : a.prm.c_branch + 2 * a.prm.c_regop;
  const bool have = lane < ch.y;
  int4 rec = make_int4(0, 0, 0, 0), meta = make_int4(0, 0, lane, 0), sr = make_int4(-1, 0, 0, 0);
  if (have) {
    rec = __ldg(a.lrec + ch.x + lane);
    meta = __ldg(a.lmeta + ch.x + lane);
    sr = __ldg(a.lsem + ch.x + lane);
  }
  const bool valid = have && meta.y < copies;
  const int32_t e = meta.x, head = meta.z;
  const int32_t gl = g + meta.y;
  const int32_t t_in = S.t[e], lr_in = S.lr[e], n_in = S.nn[e];

  // semaphores incremented in this chunk: lanes in order of their increments
  const bool prod = valid && sr.x >= 0;
  const unsigned pm = __ballot_sync(kFull, prod);
  int32_t pub_own = 0;
  if (prod) {
    const unsigned peers = __match_any_sync(pm, sr.x);
    pub_own = S.semv[sr.x];
    if (lane == __ffs(peers) - 1) { S.grp[sr.x] = peers; S.tag[sr.x] = ctag; }
  }
  __syncwarp();

  // waits: earlier increments from the history, in-chunk ones by lane
  int32_t known = kNeg;                        // satisfied before this chunk (kNeg: none)
  int intra[kMaxIntra];
  int n_intra = 0;
  bool fallback = false;
  for (int j = 0; valid && j < rec.z; ++j) {
    const int32_t T = __ldg(a.thr + __ldg(a.dseg + rec.w + j) + gl);
    if (T <= 0) continue;
    const int32_t s = __ldg(a.dsem + rec.w + j);
    const int32_t pub = S.semv[s];
    if (T <= pub) { known = max(known, a.hist[S.semhb[s] + (T - 1)]); continue; }
    const unsigned m = S.tag[s] == ctag ? S.grp[s] : 0u;
    const int k = T - pub;
    if (k > __popc(m) || n_intra == kMaxIntra) { fallback = true; break; }
    intra[n_intra++] = kth_bit(m, k);
  }
  if (__ballot_sync(kFull, fallback)) return SIM_FALLBACK;

  const int32_t wcost = BB ? 0 : rec.z * cwait;
  const int32_t apre = (meta.w & LANE_ITER_START) ? iter_cost : 0;
  const int32_t A = valid ? apre + wcost + a.prm.ii : 0;
  int32_t r_intra = kNeg;                      // retire of in-chunk producers (lower bound)
  int32_t issue = 0, retire = 0, t_after = 0;
  const bool any_intra = __ballot_sync(kFull, n_intra > 0) != 0;
  const int passes = any_intra ? ch.y + 2 : 1;
  bool settled = false;
  for (int pass = 0; pass < passes; ++pass) {
    const int32_t ready = max(known, r_intra);
    const int32_t B0 = (valid && ready >= 0) ? ready + a.prm.ii : kNeg;
    // segmented inclusive scan of the cursor maps over the engine's run
    int32_t Ai = A, Bi = B0;
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t Ap = __shfl_up_sync(kFull, Ai, o), Bp = __shfl_up_sync(kFull, Bi, o);
      if (lane - o >= head) { Bi = max(Bp + Ai, Bi); Ai = Ap + Ai; }
    }
    int32_t Ae = __shfl_up_sync(kFull, Ai, 1), Be = __shfl_up_sync(kFull, Bi, 1);
    if (lane == head) { Ae = 0; Be = kNeg; }
    const int32_t tb = max(t_in + Ae, Be);
    t_after = max(t_in + Ai, Bi);
    issue = max(tb + apre + wcost, max(ready, 0));
    int32_t v = valid ? issue + rec.y : kNeg;
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t vp = __shfl_up_sync(kFull, v, o);
      if (lane - o >= head) v = max(v, vp);
    }
    retire = max(lr_in, v);
    // new lower bound from the in-chunk producers' retire times
    int32_t nr = kNeg;
#pragma unroll
    for (int i = 0; i < kMaxIntra; ++i) {
      const int32_t src = i < n_intra ? intra[i] : lane;
      const int32_t rv = __shfl_sync(kFull, retire, src);
      if (i < n_intra) nr = max(nr, rv);
    }
    if (!__ballot_sync(kFull, nr != r_intra)) { settled = true; break; }
    r_intra = nr;
  }
  if (!settled) return SYNC_PROG_DEADLOCK;   // a cycle of waits inside the chunk

  // publish increments, instance counts, checksum terms, engine state
  if (prod) {
    a.hist[S.semhb[sr.x] + (int64_t)sr.y * gl + (sr.z - 1)] = retire;
  }
  const unsigned vm = __ballot_sync(kFull, valid);
  const unsigned run_le = vm & lanemask_le() & ~((1u << head) - 1u);
  if (valid) {
    const uint32_t nj = (uint32_t)n_in + __popc(run_le);
    chk += inst_term(issue, retire, (uint32_t)e, nj);
    if (TL) {
      const int64_t o = __ldg(a.inst_off + rec.x) + gl;
      a.issue[o] = issue;
      a.retire[o] = retire;
    }
  }
  __syncwarp();
  if (prod && lane == 31 - __clz(__match_any_sync(pm, sr.x))) S.semv[sr.x] = pub_own + __popc(S.grp[sr.x]);
  if (have && (meta.w & LANE_RUN_LAST)) {
    S.t[e] = t_after;
    S.lr[e] = retire;
    S.nn[e] = n_in + __popc(run_le);
  }
  __syncwarp();
  // engines without records here still pass the iteration starts between copies
  if (copies > 1 && lane < 32 && !((ch.w >> lane) & 1)) S.t[lane] += (copies - 1) * iter_cost;
  __syncwarp();
  return 0;
}

template <int MODE, bool BB, bool TL>
__global__ void __launch_bounds__(kWarps * 32) k_sweep(const SweepArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  WarpSmem S;
  {
    unsigned char* p = smem_raw + wib * warp_bytes(a.sem_cap, a.frame_depth);
    S.semhb = reinterpret_cast<int64_t*>(p); p += 8 * a.sem_cap;
    S.frames = reinterpret_cast<Frame*>(p); p += sizeof(Frame) * a.frame_depth;
    S.t = reinterpret_cast<int32_t*>(p); p += 4 * 32;
    S.lr = reinterpret_cast<int32_t*>(p); p += 4 * 32;
    S.nn = reinterpret_cast<int32_t*>(p); p += 4 * 32;
    S.semv = reinterpret_cast<int32_t*>(p); p += 4 * a.sem_cap;
    S.grp = reinterpret_cast<uint32_t*>(p); p += 4 * a.sem_cap;
    S.tag = reinterpret_cast<int32_t*>(p);
  }
  const int32_t cwait = MODE == SYNC_THR_PERLOOP ? a.prm.c_wait_ops_perloop : a.prm.c_wait_ops_count;
  const int32_t iter_cost = BB ? a.prm.c_branch : a.prm.c_branch + 2 * a.prm.c_regop;

  for (;;) {
    int slot = 0;
    if (lane == 0) slot = atomicAdd(a.next_slot, 1);
    slot = __shfl_sync(kFull, slot, 0);
    if (slot >= a.n_programs) break;
    const int p = __ldg(a.order + slot);
    const ProgInfo pi = a.prog[p];
    if (time_bound<BB>(pi, a.prm, cwait) > 2147483647ull) {
      if (lane == 0) { a.makespan[p] = -1; a.checksum[p] = 0; a.status[p] = SYNC_PROG_OVERFLOW; }
      continue;
    }
    for (int i = lane; i < pi.nsem[MODE]; i += 32) {
      S.semv[i] = 0;
      S.semhb[i] = __ldg(a.semhb + pi.semhb_off[MODE] + i);
      S.tag[i] = -1;
    }
    S.t[lane] = 0; S.lr[lane] = 0; S.nn[lane] = 0;
    __syncwarp();
    unsigned long long chk = 0;
    int32_t loop = pi.loop_base, item = 0, g = 0, g_end = 1, sp = 0, ctag = 0;
    int32_t pbeg = __ldg(a.plan_ptr + loop), pend = __ldg(a.plan_ptr + loop + 1);
    int verdict = SYNC_PROG_OK;
    for (;;) {
      if (pbeg + item == pend) {                       // end of an iteration's body
        if (sp == 0) break;                            // the top-level loop runs once
        if (BB) {                                      // all-engine barrier: drain, release
          int32_t arr = lane < pi.ne ? max(S.t[lane], S.lr[lane]) : 0;
          arr = (int32_t)__reduce_max_sync(kFull, (unsigned)arr);
          __syncwarp();
          if (lane < pi.ne) S.t[lane] = arr + a.prm.c_barrier;
          __syncwarp();
        }
        if (++g < g_end) {
          if (lane < pi.ne) S.t[lane] += iter_cost;
          __syncwarp();
          item = 0;
        } else {
          const Frame f = S.frames[--sp];
          loop = f.loop; item = f.item; g = f.g; g_end = f.g_end;
          pbeg = __ldg(a.plan_ptr + loop);
          pend = __ldg(a.plan_ptr + loop + 1);
        }
        continue;
      }
      const int4 it = __ldg(a.plan + pbeg + item);
      if (it.x == ITEM_LOOP) {                         // a loop statement
        if (BB) {
          int32_t arr = lane < pi.ne ? max(S.t[lane], S.lr[lane]) : 0;
          arr = (int32_t)__reduce_max_sync(kFull, (unsigned)arr);
          __syncwarp();
          if (lane < pi.ne) S.t[lane] = arr + a.prm.c_barrier;
        } else if (lane < pi.ne) {
          S.t[lane] += a.prm.c_regop;
        }
        const LoopInfo L = a.loop[it.y];
        const int32_t lo = __ldg(a.rowptr + L.rowptr_off + g), hi = __ldg(a.rowptr + L.rowptr_off + g + 1);
        ++item;
        if (lo < hi) {
          __syncwarp();
          if (lane == 0) S.frames[sp] = Frame{loop, item, g, g_end};
          ++sp;
          loop = it.y; item = 0; g = lo; g_end = hi;
          pbeg = __ldg(a.plan_ptr + loop);
          pend = __ldg(a.plan_ptr + loop + 1);
          if (lane < pi.ne) S.t[lane] += iter_cost;
        }
        __syncwarp();
        continue;
      }
      // a straight-line segment
      if (!BB && it.w >= 0) {                          // several iterations at once
        const int4 ch = __ldg(a.chunk + it.w);
        const int32_t v = min(ch.z, g_end - g);
        verdict = run_chunk<MODE, BB, TL>(a, S, ch, g, v, ++ctag, lane, chk);
        if (verdict) break;
        g += v - 1;
        item = pend - pbeg;                            // continue at the END of iteration g
        continue;
      }
      for (int c = 0; c < it.z && !verdict; ++c)
        verdict = run_chunk<MODE, BB, TL>(a, S, __ldg(a.chunk + it.y + c), g, 1, ++ctag, lane, chk);
      if (verdict) break;
      ++item;
    }
    if (verdict == SIM_FALLBACK) {
      if (lane == 0) {
        a.status[p] = SIM_FALLBACK;
        const int i = atomicAdd(a.fallback, 1);
        a.fallback[1 + i] = p;
      }
      __syncwarp();
      continue;
    }
    int32_t ms = lane < pi.ne ? max(S.t[lane], S.lr[lane]) : 0;
    ms = (int32_t)__reduce_max_sync(kFull, (unsigned)ms);
    for (int o = 16; o > 0; o >>= 1) chk += __shfl_xor_sync(kFull, chk, o);
    if (lane == 0) {
      const bool ok = verdict == SYNC_PROG_OK;
      a.makespan[p] = ok ? ms : -1;
      a.checksum[p] = ok ? chk : 0ull;
      a.status[p] = verdict;
    }
    __syncwarp();
  }
}

template <int MODE, bool BB>
cudaError_t launch3(const SweepArgs& a, size_t smem, int num_sms, cudaStream_t s) {
  auto run = [&](auto kern) -> cudaError_t {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kWarps * 32, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    const long long want = ((long long)a.n_programs + kWarps - 1) / kWarps;
    const long long cap = (long long)num_sms * per_sm;
    const int grid = (int)(want < cap ? want : cap);
    e = cudaMemsetAsync(a.next_slot, 0, sizeof(int32_t), s);
    if (e == cudaSuccess) e = cudaMemsetAsync(a.fallback, 0, sizeof(int32_t), s);
    if (e != cudaSuccess) return e;
    kern<<<grid, kWarps * 32, smem, s>>>(a);
    return cudaGetLastError();
  };
  if (a.issue) return run(k_sweep<MODE, BB, true>);
  return run(k_sweep<MODE, BB, false>);
}

}  // namespace

size_t sweep_smem_bytes(int sem_cap, int frame_depth) {
  return kWarps * warp_bytes(sem_cap, frame_depth);
}

cudaError_t launch_sweep(const SweepArgs& a, bool barrier, int num_sms, cudaStream_t s) {
  if (a.n_programs == 0) return cudaSuccess;
  const size_t smem = sweep_smem_bytes(a.sem_cap, a.frame_depth);
  if (a.mode == SYNC_THR_PERLOOP)
    return barrier ? launch3<SYNC_THR_PERLOOP, true>(a, smem, num_sms, s)
                   : launch3<SYNC_THR_PERLOOP, false>(a, smem, num_sms, s);
  return barrier ? launch3<SYNC_THR_COUNT, true>(a, smem, num_sms, s)
                 : launch3<SYNC_THR_COUNT, false>(a, smem, num_sms, s);
}

}  // namespace syncgb
