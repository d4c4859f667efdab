// Schedule simulator: one warp per program, lane e = engine e.
//
// Every lane walks the common loop tree with its own cursor (a stack of
// frames in shared memory) and its own time t, visiting its engine's
// instructions and every loop's control points.  Lanes run independently in
// bursts of up to kBurst events and meet once per round at a __syncwarp:
//   - a datapath instruction waits on semaphores: the value of a semaphore
//     (increments processed so far) lives in shared memory, written only by
//     the owning engine's lane with a release store after the increment's
//     retire time was written to the history array; a waiting lane reads the
//     value with an acquire load and, once it reaches the threshold, takes
//     the retire time of that increment (the time the semaphore reached it);
//     otherwise it stops its burst and retries in the next round;
//   - a barrier (barrier scheme) stops the lane; when the ballot shows every
//     engine of the program at its barrier, the release time is the
//     warp-reduced maximum arrival plus the barrier cost;
//   - a round in which no lane moved is a deadlock (every lane saw the state
//     published before the previous __syncwarp and still could not move).
// Times are int32: a program whose static time bound exceeds INT32_MAX gets
// status 4 without being simulated, so no time can overflow.
#include "enc.h"

namespace syncgb {
namespace {

constexpr int kWarps = 4;       // warps per CTA
constexpr int kBurst = 16;      // events per lane between two warp meetings

enum : int { ST_RUN = 0, ST_BAR = 1, ST_DONE = 2 };
enum : int { R_MOVED = 0, R_BLOCKED = 1, R_BARRIER = 2, R_DONE = 3 };

struct Frame { int32_t loop, ptr, g, g_end; };

__device__ __forceinline__ int32_t ld_acquire(const int32_t* p) {
  int32_t v;
  asm volatile("ld.acquire.cta.shared.b32 %0, [%1];"
               : "=r"(v) : "r"((unsigned)__cvta_generic_to_shared(p)) : "memory");
  return v;
}
__device__ __forceinline__ void st_release(int32_t* p, int32_t v) {
  asm volatile("st.release.cta.shared.b32 [%0], %1;"
               :: "r"((unsigned)__cvta_generic_to_shared(p)), "r"(v) : "memory");
}

__device__ __forceinline__ unsigned long long sat_add(unsigned long long a, unsigned long long b) {
  const unsigned long long r = a + b;
  return r < a ? ~0ull : r;
}
__device__ __forceinline__ unsigned long long sat_mul(unsigned long long a, unsigned long long b) {
  return __umul64hi(a, b) ? ~0ull : a * b;
}

__device__ __forceinline__ unsigned long long inst_term(int32_t issue, int32_t retire, int32_t e,
                                                        long long n) {
  return ((unsigned long long)(uint32_t)issue * 0x9E3779B97F4A7C15ull) ^
         ((unsigned long long)(uint32_t)retire * 0xC2B2AE3D27D4EB4Full) ^
         ((unsigned long long)n * 0x165667B19E3779F9ull + (unsigned long long)e);
}

// Lane-private state of one engine.
struct Lane {
  int32_t cur, ptr, pend, g, g_end, sp;
  int32_t t, lastret, arrival;
  long long n;
  unsigned long long chk;
  bool bar_passed;
};

template <int MODE, bool BB, bool TL>
__device__ __forceinline__ int step(const SimArgs& a, const ProgInfo& pi, Lane& L, Frame* stk,
                                    int32_t* sem, int lane, int32_t iter_cost, int32_t cwait) {
  if (L.ptr == L.pend) {                       // end of an iteration's body
    if (L.sp == 0) return R_DONE;              // the top-level loop runs once
    if (BB && !L.bar_passed) { L.arrival = max(L.t, L.lastret); return R_BARRIER; }
    L.bar_passed = false;
    if (++L.g < L.g_end) {                     // next iteration starts
      L.t += iter_cost;
      L.ptr = __ldg(a.op_ptr + pi.le_base + (L.cur - pi.loop_base) * pi.ne + lane);
      return R_MOVED;
    }
    const Frame f = stk[--L.sp];               // loop exit
    L.cur = f.loop; L.ptr = f.ptr; L.g = f.g; L.g_end = f.g_end;
    L.pend = __ldg(a.op_ptr + pi.le_base + (L.cur - pi.loop_base) * pi.ne + lane + 1);
    return R_MOVED;
  }
  const int32_t op = __ldg(a.ops + L.ptr);
  if (op < 0) {                                // a loop statement
    if (BB && !L.bar_passed) { L.arrival = max(L.t, L.lastret); return R_BARRIER; }
    L.bar_passed = false;
    if (!BB) L.t += a.prm.c_regop;
    const int32_t m = -op - 1;
    const int64_t rp = __ldg(&a.loop[m].rowptr_off) + L.g;
    const int32_t lo = __ldg(a.rowptr + rp), hi = __ldg(a.rowptr + rp + 1);
    ++L.ptr;
    if (lo < hi) {
      stk[L.sp++] = Frame{L.cur, L.ptr, L.g, L.g_end};
      const int32_t row = pi.le_base + (m - pi.loop_base) * pi.ne + lane;
      L.cur = m; L.g = lo; L.g_end = hi;
      L.ptr = __ldg(a.op_ptr + row);
      L.pend = __ldg(a.op_ptr + row + 1);
      L.t += iter_cost;
    }
    return R_MOVED;
  }
  // datapath instruction `op` in global iteration L.g of its loop
  const InstrSim& X = a.instr[op];
  const int32_t ndeps = __ldg(&X.ndeps);
  const int32_t dep_begin = __ldg(&X.dep_begin);
  const int32_t tw = L.t + (BB ? 0 : ndeps * cwait);
  int32_t ready = 0;
  for (int j = 0; j < ndeps; ++j) {
    const ConsDep& C = a.cdep[dep_begin + j];
    const int32_t T = __ldg(a.thr + __ldg(&C.seg_off) + L.g);
    if (T <= 0) continue;
    const int32_t s = __ldg(&C.tsem[MODE]);
    if (ld_acquire(sem + s) < T) return R_BLOCKED;   // semaphore below threshold
    ready = max(ready, a.hist[__ldg(&C.thist[MODE]) + (T - 1)]);
  }
  const int32_t issue = max(tw, ready);
  const int32_t retire = max(issue + __ldg(&X.lat), L.lastret);
  L.t = issue + a.prm.ii;
  L.lastret = retire;
  const int32_t s = __ldg(&X.own_sem[MODE]);
  if (s >= 0) {                                // someone waits on this semaphore
    a.hist[__ldg(&X.hbase[MODE]) + (int64_t)__ldg(&X.hstride[MODE]) * L.g] = retire;
    st_release(sem + s, sem[s] + 1);
  }
  ++L.n;
  L.chk += inst_term(issue, retire, lane, L.n);
  if (TL) {
    const int64_t o = __ldg(&X.inst_off) + L.g;
    a.issue[o] = issue;
    a.retire[o] = retire;
  }
  ++L.ptr;
  return R_MOVED;
}

template <int MODE, bool BB, bool TL>
__global__ void __launch_bounds__(kWarps * 32) k_simulate(const SimArgs a) {
  extern __shared__ __align__(16) int32_t smem[];
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  const int per_warp = a.sem_ints + a.ne_max * a.frame_depth * 4;
  int32_t* sem = smem + wib * per_warp;
  Frame* stk = reinterpret_cast<Frame*>(sem + a.sem_ints) + (lane < a.ne_max ? lane : 0) * a.frame_depth;
  const int32_t cwait = MODE == SYNC_THR_PERLOOP ? a.prm.c_wait_ops_perloop : a.prm.c_wait_ops_count;
  const int32_t iter_cost = BB ? a.prm.c_branch : a.prm.c_branch + 2 * a.prm.c_regop;
  const long long n_warps = (long long)gridDim.x * kWarps;

  for (long long slot = (long long)blockIdx.x * kWarps + wib; slot < a.n_programs; slot += n_warps) {
    const int p = __ldg(a.order + slot);
    const ProgInfo pi = a.prog[p];
    // static time bound (identical in every lane)
    unsigned long long bound = (unsigned long long)pi.agg_lat;
    bound = sat_add(bound, sat_mul((unsigned long long)a.prm.ii, (unsigned long long)pi.n_inst));
    if (BB) {
      bound = sat_add(bound, sat_mul(sat_mul((unsigned long long)pi.ne, (unsigned long long)pi.n_iter),
                                     (unsigned long long)a.prm.c_branch));
      bound = sat_add(bound, sat_mul((unsigned long long)(pi.n_stmt + pi.n_iter),
                                     (unsigned long long)a.prm.c_barrier));
    } else {
      bound = sat_add(bound, sat_mul((unsigned long long)cwait, (unsigned long long)pi.n_pairs));
      const unsigned long long ctl =
          sat_add(sat_mul((unsigned long long)pi.n_stmt, (unsigned long long)a.prm.c_regop),
                  sat_mul((unsigned long long)pi.n_iter,
                          (unsigned long long)a.prm.c_branch + 2ull * (unsigned long long)a.prm.c_regop));
      bound = sat_add(bound, sat_mul((unsigned long long)pi.ne, ctl));
    }
    if (bound > 2147483647ull) {
      if (lane == 0) { a.makespan[p] = -1; a.checksum[p] = 0; a.status[p] = SYNC_PROG_OVERFLOW; }
      continue;
    }
    for (int i = lane; i < pi.nsem[MODE]; i += 32) sem[i] = 0;
    __syncwarp();

    const bool active = lane < pi.ne;
    Lane L;
    L.cur = pi.loop_base; L.g = 0; L.g_end = 1; L.sp = 0;
    L.ptr = active ? __ldg(a.op_ptr + pi.le_base + lane) : 0;
    L.pend = active ? __ldg(a.op_ptr + pi.le_base + lane + 1) : 0;
    L.t = 0; L.lastret = 0; L.arrival = 0; L.n = 0; L.chk = 0; L.bar_passed = false;
    int state = active ? ST_RUN : ST_DONE;
    // every round moves at least one event or releases a barrier, so events
    // plus barriers bound the rounds; exceeding it would be a defect (status 8)
    const long long guard = pi.n_inst + 4ll * (pi.n_stmt + pi.n_iter) * (pi.ne + 1) + 64;
    long long rounds = 0;
    int result = SYNC_PROG_OK;
    for (;;) {
      bool moved = false;
      if (state == ST_RUN) {
        for (int b = 0; b < kBurst; ++b) {
          const int r = step<MODE, BB, TL>(a, pi, L, stk, sem, lane, iter_cost, cwait);
          if (r == R_MOVED) { moved = true; continue; }
          if (r == R_BARRIER) { state = ST_BAR; moved = true; }
          else if (r == R_DONE) { state = ST_DONE; moved = true; }
          break;
        }
      }
      __syncwarp();
      const unsigned any_moved = __ballot_sync(0xffffffffu, moved);
      const unsigned at_bar = __ballot_sync(0xffffffffu, state == ST_BAR);
      const unsigned running = __ballot_sync(0xffffffffu, state == ST_RUN);
      const unsigned lanes = pi.ne >= 32 ? 0xffffffffu : ((1u << pi.ne) - 1u);
      if (++rounds > guard) { result = SYNC_PROG_ROUND_GUARD; break; }
      if (BB && at_bar == lanes) {             // every engine drained: release
        const int32_t rel = (int32_t)__reduce_max_sync(0xffffffffu, (unsigned)(state == ST_BAR ? L.arrival : 0)) +
                            a.prm.c_barrier;
        if (state == ST_BAR) { L.t = rel; state = ST_RUN; L.bar_passed = true; }
        continue;
      }
      if (running == 0 && at_bar == 0) break;  // all engines done
      if (any_moved == 0) { result = SYNC_PROG_DEADLOCK; break; }
    }
    int32_t ms = active ? max(L.t, L.lastret) : 0;
    ms = (int32_t)__reduce_max_sync(0xffffffffu, (unsigned)ms);
    unsigned long long chk = active ? L.chk : 0ull;
    for (int o = 16; o > 0; o >>= 1) chk += __shfl_xor_sync(0xffffffffu, chk, o);
    if (lane == 0) {
      const bool ok = result == SYNC_PROG_OK;
      a.makespan[p] = ok ? ms : -1;
      a.checksum[p] = ok ? chk : 0ull;
      a.status[p] = result;
    }
    __syncwarp();
  }
}

template <int MODE, bool BB>
cudaError_t launch3(const SimArgs& a, int grid, size_t smem, cudaStream_t s) {
  cudaError_t e;
  if (a.issue) {
    e = cudaFuncSetAttribute(k_simulate<MODE, BB, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_simulate<MODE, BB, true><<<grid, kWarps * 32, smem, s>>>(a);
  } else {
    e = cudaFuncSetAttribute(k_simulate<MODE, BB, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_simulate<MODE, BB, false><<<grid, kWarps * 32, smem, s>>>(a);
  }
  return cudaGetLastError();
}

}  // namespace

size_t simulate_smem_per_warp(int sem_ints, int frame_depth, int ne_max) {
  return (size_t)(sem_ints + ne_max * frame_depth * 4) * sizeof(int32_t);
}

cudaError_t launch_simulate(const SimArgs& a, bool barrier, int num_sms, cudaStream_t s) {
  if (a.n_programs == 0) return cudaSuccess;
  const size_t smem = kWarps * simulate_smem_per_warp(a.sem_ints, a.frame_depth, a.ne_max);
  const long long want = ((long long)a.n_programs + kWarps - 1) / kWarps;
  // 16 resident CTAs (64 warps) per SM at most; programs beyond that are
  // picked up grid-stride in descending-work order
  const long long cap = (long long)num_sms * 16;
  const int grid = (int)(want < cap ? want : cap);
  if (a.mode == SYNC_THR_PERLOOP)
    return barrier ? launch3<SYNC_THR_PERLOOP, true>(a, grid, smem, s)
                   : launch3<SYNC_THR_PERLOOP, false>(a, grid, smem, s);
  return barrier ? launch3<SYNC_THR_COUNT, true>(a, grid, smem, s)
                 : launch3<SYNC_THR_COUNT, false>(a, grid, smem, s);
}

}  // namespace syncgb
