// Schedule simulator: one CTA per program at a time, warp e = engine e.
//
// Each warp walks the common loop tree for its engine (current row of op
// records, iteration range, a stack of frames in shared memory), but instead
// of one event per step it takes up to 32 consecutive events of its stream at
// once, one per lane:
//   - inside a loop body with no child loop (barrier-free), the events run on
//     across iteration boundaries (the body's records repeat, the END record
//     between two iterations is an iteration start);
//   - otherwise they stop at the next child loop or END record, which the
//     whole warp then handles as one control step (loop statement, next
//     iteration, loop exit, barrier).
// The engine's cursor obeys t' = max(t + A, B) for every event -- A the cost
// of the event (wait ops, issue interval, iteration start), B the time its
// waits become satisfied plus the issue interval (or -inf) -- and these
// max-plus affine maps compose associatively, so a 5-step warp scan gives
// every lane the cursor before its event; issue = max(cursor + wait ops,
// ready), and retire (in-order retirement) is a max-scan of issue + latency.
//
// Waits: a semaphore's value (its increments processed so far) and the
// history base of its retire times live in shared memory; only the owning
// engine's warp writes them -- the retire times to the history array first,
// then, after __syncwarp, one release store of the semaphore's new value per
// semaphore touched by the chunk.  A lane whose wait is not yet satisfied
// cuts the chunk before itself; a warp whose first event is blocked polls
// that semaphore a bounded number of times, then ends its round.
// Barriers (barrier scheme) are met in shared memory: each engine stores its
// arrival time and counts itself in; the last one computes the release (the
// maximum arrival plus the barrier cost) and advances a generation counter,
// which the others poll a bounded number of times before ending their round.
// Warps meet once per round at a CTA barrier; a round in which no warp moved
// is a deadlock.
//
// CTAs are persistent and fetch program ids from a counter in descending-work
// order.  Times are int32: a program whose static time bound exceeds
// INT32_MAX gets status 4 without being simulated, so no time can overflow.
#include "cost.cuh"
#include "waitval.cuh"

namespace syncgb {
namespace {

constexpr int kChunks = 16;                 // chunks per warp per round
constexpr int kSpin = 64;                   // polls of a semaphore or barrier per round
// A program still running after this many SM clock cycles (about 2 s) stops at
// the next round boundary with SYNC_PROG_TIMEOUT, so a launch always ends;
// the deterministic round guard (status 8) stays the only defect verdict.
constexpr long long kWatchdogCycles = 4000000000ll;
constexpr unsigned kFull = 0xffffffffu;
// "-infinity" of the max-plus maps t' = max(t + A, B): cursors are >= 0 and
// costs A >= 0, so a composed term -1 + (later costs) never exceeds the
// t + (all costs) term and -1 acts exactly as -infinity in int32.
constexpr int32_t kNeg = -1;

enum : int { ST_RUN = 0, ST_BAR = 1, ST_DONE = 2 };

struct Frame { int32_t row, ptr, g, g_end, lo; };   // lo: start of the trip of iteration g

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
__device__ __forceinline__ unsigned lanemask_le() {
  unsigned m;
  asm("mov.u32 %0, %%lanemask_le;" : "=r"(m));
  return m;
}

__device__ __forceinline__ int64_t lohi(int32_t lo, int32_t hi) {
  return (int64_t)(((uint64_t)(uint32_t)hi << 32) | (uint32_t)lo);
}

// Per-instance checksum term (see include/sync.h).
__device__ __forceinline__ unsigned long long inst_term(int32_t issue, int32_t retire, uint32_t e,
                                                        uint32_t n) {
  uint32_t x = ((uint32_t)issue ^ (n * 0x9E3779B9u + e)) * 0x85EBCA6Bu;
  x ^= x >> 13;
  uint32_t y = ((uint32_t)retire ^ (n * 0xC2B2AE35u + e)) * 0x27D4EB2Fu;
  y ^= y >> 15;
  return ((unsigned long long)x << 32) | y;
}


struct Smem {
  int64_t* semhb;          // [sem_cap]
  int32_t* sem;            // [sem_cap]
  int32_t* w_moved;        // [warps]
  int32_t* w_state;
  int32_t* w_arrival;      // barrier arrival times
  int32_t* w_ms;
  unsigned long long* w_chk;
  int32_t* slot;           // [4]: program slot, barrier count, generation, release
  Frame* frames;           // [warps][frame_depth]
  unsigned long long* tally;  // [3] fused check: unsafe, over-synchronised, first offending pair
};

// Engine state, identical in the 32 lanes of the engine's warp.
struct Eng {
  int32_t row, pbeg, rend, ptr, g, g_end, sp;
  int32_t lo;              // start of the current trip
  int32_t ic;              // iteration-start cost of the current row's loop
  bool loops;              // the current row holds a child loop
  bool fbar;               // barrier-free: the current row's loop ends each iteration
                           // with a barrier-fallback barrier
  int32_t t, lastret;
  int32_t bar_gen;         // barrier generation this engine waits to see pass
  uint32_t n;              // datapath instances issued so far
  int state;
  bool bar_passed;
};

// Arrive at the program's next barrier; the last engine to arrive releases it.
// Returns true once the barrier has been released for this engine.
template <bool BB>
__device__ __forceinline__ bool barrier_arrive(const SimArgs& a, const Smem& S, Eng& E, int w, int lane,
                                              int ne) {
  E.bar_gen = ld_acquire(S.slot + 2);
  int last = 0;
  if (lane == 0) {
    S.w_arrival[w] = max(E.t, E.lastret);
    __threadfence_block();
    last = atomicAdd(S.slot + 1, 1) == ne - 1;
    if (last) {
      __threadfence_block();
      int32_t rel = 0;
      for (int i = 0; i < ne; ++i) rel = max(rel, *(volatile int32_t*)(S.w_arrival + i));
      S.slot[3] = rel + a.prm.c_barrier;
      S.slot[1] = 0;
      st_release(S.slot + 2, E.bar_gen + 1);
    }
  }
  E.state = ST_BAR;
  return __shfl_sync(kFull, last, 0) != 0;
}

// Has the barrier this engine waits at been released?  Polls at most kSpin times.
__device__ __forceinline__ bool barrier_poll(const Smem& S, const Eng& E, int spins) {
  for (int i = 0;; ++i) {
    if (ld_acquire(S.slot + 2) != E.bar_gen) return true;
    if (i >= spins) return false;
  }
}

template <int MODE, bool BB, bool TL>
__device__ __forceinline__ void set_row(const SimArgs& a, Eng& E, int32_t row) {
  E.row = row;
  E.pbeg = __ldg(a.op_ptr + row);
  const int2 ri = __ldg(a.rowinfo + row);
  E.rend = ri.x;
  E.loops = (ri.y & 1) != 0;
  E.fbar = !BB && (ri.y & 4) != 0;
  // barrier-free with trip-register elision, a loop carrying no offset > 0
  // has no r-hat++ at its iteration starts
  const int32_t ic = BB ? a.prm.c_branch : a.prm.c_branch + 2 * a.prm.c_regop;
  E.ic = (!BB && a.prm.trip_register_elision && (ri.y & 2) ? ic - a.prm.c_regop : ic) + hoist_ops<MODE, BB>(a, row);
}

// Fused simulation: the wait value of consumer-grouped dependency r for the
// engine's instance at global iteration gj of its current loop, from the
// engine's loop state (the register form of Sec. 5.1, r_S and r-hat_S read
// off the level of S); with the optional check, the Eq. (1) minimum beside
// it, mismatches counted in nu / no and the smallest offending pair in first.
template <int MODE>
__device__ __forceinline__ int32_t fused_value(const SimArgs& a, const Frame* frames, const Eng& E, int r,
                                               int32_t gj, unsigned& nu, unsigned& no,
                                               unsigned long long& first) {
  const DepInfo& D = a.dep[__ldg(a.ddep + r)];
  int32_t gs = gj, st = E.lo;
  if (D.up > 0) {
    const Frame f = frames[E.sp - D.up];
    gs = f.g;
    st = f.lo;
  }
  const int32_t T = wait_value(a, D, gs, st, MODE);
  if (a.chk_counts) {
    const int32_t m = minimum(a, D, gs, st, MODE);
    if (T != m) {
      if (T < m) ++nu; else ++no;
      const unsigned long long q = (unsigned long long)(__ldg(a.dseg + r) + gj);
      first = q < first ? q : first;
    }
  }
  return T;
}

// One round of engine w: up to kChunks chunks or control steps.
template <int MODE, bool BB, bool TL, bool FUSED>
__device__ __forceinline__ bool run_engine(const SimArgs& a, const Smem& S, Eng& E, int w, int lane,
                                           int ne, unsigned long long& chk) {
  const int32_t ii = a.prm.ii;
  Frame* frames = S.frames + w * a.frame_depth;
  bool moved = false;
  int spins = kSpin;
  if (E.state == ST_BAR) {                           // waiting at a barrier
    if (!barrier_poll(S, E, spins)) return false;
    E.t = *(volatile int32_t*)(S.slot + 3);
    E.state = ST_RUN;
    E.bar_passed = true;
    moved = true;
  }
  for (int c = 0; c < kChunks; ++c) {
    const int4 r0 = __ldg(a.ops + E.ptr);
    const bool at_end = r0.x == OP_END && E.sp != 0;
    if ((BB ? r0.x == OP_LOOP || at_end : E.fbar && at_end) && !E.bar_passed) {
      // an all-engine barrier before the loop statement / after the iteration
      // (barrier-free: after each iteration of a loop with a fallback barrier)
      moved = true;
      if (!barrier_arrive<BB>(a, S, E, w, lane, ne) && !barrier_poll(S, E, spins)) return true;
      E.t = *(volatile int32_t*)(S.slot + 3);
      E.state = ST_RUN;
      E.bar_passed = true;
    }
    if (r0.x == OP_LOOP) {                           // a loop statement
      E.bar_passed = false;
      if (!BB) {                                     // r-hat := 0, unless the child has none
        const bool el = a.prm.trip_register_elision && (__ldg(a.rowinfo + r0.y + w).y & 2);
        E.t += el ? 0 : a.prm.c_regop;
      }
      const int64_t rp = lohi(r0.z, r0.w) + E.g;
      const int32_t lo = __ldg(a.rowptr + rp), hi = __ldg(a.rowptr + rp + 1);
      ++E.ptr;
      if (lo < hi) {
        __syncwarp();
        if (lane == 0) frames[E.sp] = Frame{E.row, E.ptr, E.g, E.g_end, E.lo};
        ++E.sp;
        set_row<MODE, BB, TL>(a, E, r0.y + w);
        E.ptr = E.pbeg;
        E.g = lo;
        E.g_end = hi;
        E.lo = lo;
        E.t += E.ic;
      }
      moved = true;
      continue;
    }
    if (r0.x == OP_END) {                            // end of an iteration's body
      if (E.sp == 0) { E.state = ST_DONE; return true; }   // the top-level loop runs once
      E.bar_passed = false;
      if (++E.g < E.g_end) {
        E.t += E.ic;
        E.ptr = E.pbeg;
      } else {
        __syncwarp();
        const Frame f = frames[--E.sp];
        set_row<MODE, BB, TL>(a, E, f.row);
        E.ptr = f.ptr; E.g = f.g; E.g_end = f.g_end; E.lo = f.lo;
      }
      moved = true;
      continue;
    }
    // ---- a chunk of datapath events (and, run-on, iteration starts)
    const bool periodic = !BB && !E.loops && !E.fbar;
    const int32_t period = E.rend - E.pbeg + 1;      // the body's records and its END
    int32_t idx, gj;
    bool valid, is_end;
    if (periodic) {
      const int32_t off = (E.ptr - E.pbeg) + lane;
      const int32_t it = off / period;
      idx = E.pbeg + (off - it * period);
      gj = E.g + it;
      is_end = idx == E.rend;
      valid = gj < E.g_end && !(is_end && gj == E.g_end - 1);   // stop before the loop exit
    } else {
      const int32_t stop = __ldg(a.opstop + E.ptr);
      idx = E.ptr + lane;
      gj = E.g;
      is_end = false;
      valid = idx < stop;
    }
    const int32_t nev = __popc(__ballot_sync(kFull, valid));
    const bool dp = valid && !is_end;
    int4 rec = make_int4(0, 0, 0, 0), srec = make_int4(-1, 0, 0, 0);
    if (dp) {
      rec = __ldg(a.ops + idx);
      srec = __ldg(a.opsem + idx);
    }
    // waits: every dependency's semaphore must have reached the threshold
    int32_t ready = 0, bsem = 0, bthr = 0;
    bool waited = false, blocked = false;
    unsigned nu = 0, no = 0;                         // fused check, this lane's dependencies
    unsigned long long first = ~0ull;
    for (int j = 0; dp && j < rec.z; ++j) {
      const int32_t T = FUSED ? fused_value<MODE>(a, frames, E, rec.w + j, gj, nu, no, first)
                              : __ldg(a.thr + __ldg(a.dseg + rec.w + j) + gj);
      if (T <= 0) continue;
      const int32_t s = __ldg(a.dsem + rec.w + j);
      if (ld_acquire(S.sem + s) < T) { blocked = true; bsem = s; bthr = T; break; }
      ready = max(ready, a.hist[S.semhb[s] + (T - 1)]);
      waited = true;
    }
    const unsigned bm = __ballot_sync(kFull, blocked);
    const int32_t cut = bm ? min(nev, __ffs(bm) - 1) : nev;
    if (cut == 0) {                                  // blocked at the first event
      const int32_t s = __shfl_sync(kFull, bsem, 0), T = __shfl_sync(kFull, bthr, 0);
      for (;;) {                                     // poll the semaphore, bounded
        if (spins <= 0) return moved;
        --spins;
        if (ld_acquire(S.sem + s) >= T) break;
      }
      --c;                                           // retry this chunk
      continue;
    }
    const bool in = lane < cut;
    if (FUSED && in && (nu | no)) {                  // consumed events only (a cut one is re-evaluated)
      if (nu) atomicAdd(S.tally + 0, (unsigned long long)nu);
      if (no) atomicAdd(S.tally + 1, (unsigned long long)no);
      atomicMin(S.tally + 2, first);
    }
    // cursor maps t' = max(t + A, B), inclusive scan over the lanes
    const int32_t wcost = BB ? 0 : wait_ops<MODE>(a, rec, srec.w);
    int32_t A = 0, B = kNeg;
    if (in) {
      if (dp) { A = wcost + ii; B = waited ? ready + ii : kNeg; }
      else A = E.ic;
    }
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t Ap = __shfl_up_sync(kFull, A, o), Bp = __shfl_up_sync(kFull, B, o);
      if (lane >= o) { B = max(Bp + A, B); A = Ap + A; }
    }
    int32_t Ae = __shfl_up_sync(kFull, A, 1), Be = __shfl_up_sync(kFull, B, 1);
    if (lane == 0) { Ae = 0; Be = kNeg; }
    const int32_t tb = max(E.t + Ae, Be);           // cursor before the event
    int32_t issue = 0, v = INT_MIN;
    if (in && dp) {
      issue = max(tb + wcost, ready);
      v = issue + rec.y;
    }
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t vp = __shfl_up_sync(kFull, v, o);
      if (lane >= o) v = max(v, vp);
    }
    const int32_t retire = max(E.lastret, v);       // in-order retirement
    // publish this chunk's semaphore increments: per-engine semaphores count
    // the engine's instances, the others a fixed number per iteration
    const unsigned dm = __ballot_sync(kFull, in && dp);
    const uint32_t nj = E.n + __popc(dm & lanemask_le());   // the instance's position in the engine's stream
    const bool prod = in && dp && srec.x >= 0;
    const int32_t ninc = srec.y < 0 ? (int32_t)nj : srec.y * gj + srec.z;
    if (prod) a.hist[S.semhb[srec.x] + (ninc - 1)] = retire;
    __syncwarp();                                    // orders the warp's history writes
    const unsigned pm = __ballot_sync(kFull, prod);
    if (prod) {
      const unsigned peers = __match_any_sync(pm, srec.x);
      if (lane == 31 - __clz(peers)) st_release(S.sem + srec.x, ninc);
    }
    if (in && dp) {
      chk += inst_term(issue, retire, (uint32_t)w, nj);
      if (TL) {
        const int64_t o = __ldg(a.inst_off + rec.x) + gj;
        a.issue[o] = issue;
        a.retire[o] = retire;
      }
    }
    E.n += __popc(dm);
    // advance to the event after lane cut-1
    E.t = __shfl_sync(kFull, max(E.t + A, B), cut - 1);
    E.lastret = __shfl_sync(kFull, retire, cut - 1);
    if (periodic) {
      const int32_t off = (E.ptr - E.pbeg) + cut;
      const int32_t it = off / period;
      E.g += it;
      E.ptr = E.pbeg + (off - it * period);
    } else {
      E.ptr += cut;
    }
    moved = true;
  }
  return moved;
}

// Up to 32 engines: 1024 threads, so at most 64 registers a thread.
template <int MODE, bool BB, bool TL, bool FUSED>
__global__ void __launch_bounds__(1024) k_simulate(const SimArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int W = a.warps;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  Smem S;
  {
    unsigned char* p = smem_raw;
    S.semhb = reinterpret_cast<int64_t*>(p); p += 8 * a.sem_cap;
    S.tally = reinterpret_cast<unsigned long long*>(p); p += 3 * 8;
    S.w_chk = reinterpret_cast<unsigned long long*>(p); p += 8 * W;
    S.frames = reinterpret_cast<Frame*>(p); p += sizeof(Frame) * W * a.frame_depth;
    S.sem = reinterpret_cast<int32_t*>(p); p += 4 * a.sem_cap;
    S.w_moved = reinterpret_cast<int32_t*>(p); p += 4 * W;
    S.w_state = reinterpret_cast<int32_t*>(p); p += 4 * W;
    S.w_arrival = reinterpret_cast<int32_t*>(p); p += 4 * W;
    S.w_ms = reinterpret_cast<int32_t*>(p); p += 4 * W;
    S.slot = reinterpret_cast<int32_t*>(p);   // 4 ints
  }
  const int32_t cwait = MODE == SYNC_THR_COUNT ? a.prm.c_wait_ops_count : a.prm.c_wait_ops_perloop;

  for (;;) {
    __syncthreads();
    if (threadIdx.x == 0) *S.slot = atomicAdd(a.next_slot, 1);
    __syncthreads();
    const int slot = *S.slot;
    const int limit = a.only ? *(volatile const int32_t*)a.only : a.n_programs;
    if (slot >= limit) break;
    const int p = a.only ? a.only[1 + slot] : __ldg(a.order + slot);
    const ProgInfo pi = a.prog[p];
    if (time_bound<MODE, BB>(pi, a.prm, cwait) > 2147483647ull) {
      if (threadIdx.x == 0) { a.makespan[p] = -1; a.checksum[p] = 0; a.status[p] = SYNC_PROG_OVERFLOW; }
      continue;
    }
    for (int i = threadIdx.x; i < pi.nsem[MODE]; i += blockDim.x) {
      S.sem[i] = 0;
      S.semhb[i] = __ldg(a.semhb + pi.semhb_off[MODE] + i);
    }
    if (threadIdx.x == 0) {
      S.slot[1] = 0; S.slot[2] = 0; S.slot[3] = 0;
      S.tally[0] = S.tally[1] = 0;
      S.tally[2] = ~0ull;
    }
    const bool live = w < pi.ne;
    Eng E;
    E.sp = 0; E.g = 0; E.g_end = 1; E.lo = 0;
    E.t = 0; E.lastret = 0; E.bar_gen = 0; E.n = 0;
    E.state = live ? ST_RUN : ST_DONE;
    E.bar_passed = false;
    E.row = 0; E.pbeg = 0; E.rend = 0; E.loops = false; E.fbar = false; E.ptr = 0; E.ic = 0;
    if (live) {
      set_row<MODE, BB, TL>(a, E, pi.le_base + w);
      E.ptr = E.pbeg;
    }
    unsigned long long chk = 0;
    // every round moves an event or releases a barrier
    const long long guard = pi.n_inst + 4ll * (pi.n_stmt + pi.n_iter) * (pi.ne + 1) + 64;
    long long rounds = 0;
    int verdict = -1;
    const long long started = clock64();
    __syncthreads();
    while (verdict < 0) {
      bool moved = false;
      if (E.state != ST_DONE) moved = run_engine<MODE, BB, TL, FUSED>(a, S, E, w, lane, pi.ne, chk);
      if (lane == 0) {
        S.w_moved[w] = moved;
        S.w_state[w] = E.state;
      }
      __syncthreads();
      bool any_moved = false;
      int n_live = 0;
      for (int i = 0; i < pi.ne; ++i) {
        any_moved |= S.w_moved[i] != 0;
        n_live += S.w_state[i] != ST_DONE;
      }
      // a barrier released after its waiters stopped polling is progress too
      const bool released = S.slot[2] != E.bar_gen && E.state == ST_BAR;
      const bool any_released = __syncthreads_or(released) != 0;
      // the watchdog reads thread 0's clock so that every thread agrees
      if (threadIdx.x == 0) S.w_ms[0] = clock64() - started > kWatchdogCycles;
      __syncthreads();
      if (++rounds > guard) verdict = SYNC_PROG_ROUND_GUARD;
      else if (S.w_ms[0]) verdict = SYNC_PROG_TIMEOUT;
      else if (n_live == 0) verdict = SYNC_PROG_OK;
      else if (!any_moved && !any_released) verdict = SYNC_PROG_DEADLOCK;
      __syncthreads();
    }
    for (int o = 16; o > 0; o >>= 1) chk += __shfl_xor_sync(kFull, chk, o);
    if (lane == 0) {
      S.w_chk[w] = live ? chk : 0ull;
      S.w_ms[w] = live ? max(E.t, E.lastret) : 0;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      unsigned long long ck = 0;
      int32_t ms = 0;
      for (int i = 0; i < pi.ne; ++i) { ck += S.w_chk[i]; ms = max(ms, S.w_ms[i]); }
      const bool ok = verdict == SYNC_PROG_OK;
      a.makespan[p] = ok ? ms : -1;
      a.checksum[p] = ok ? ck : 0ull;
      a.status[p] = verdict;
      // fused check: the pairs of programs that ran to the end
      if (FUSED && ok && a.chk_counts) {
        if (S.tally[0]) atomicAdd(a.chk_counts + 0, S.tally[0]);
        if (S.tally[1]) atomicAdd(a.chk_counts + 1, S.tally[1]);
        if (S.tally[2] != ~0ull) atomicMin(a.chk_first, S.tally[2]);
      }
    }
  }
}

template <int MODE, bool BB>
cudaError_t launch3(const SimArgs& a, size_t smem, int num_sms, cudaStream_t s) {
  auto run = [&](auto kern) -> cudaError_t {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int threads = 32 * a.warps;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, threads, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    const long long cap = (long long)num_sms * per_sm;
    const int grid = (int)(a.n_programs < cap ? a.n_programs : cap);
    e = cudaMemsetAsync(a.next_slot, 0, sizeof(int32_t), s);
    if (e != cudaSuccess) return e;
    kern<<<grid, threads, smem, s>>>(a);
    return launched();
  };
  if (a.dep) return a.issue ? run(k_simulate<MODE, BB, true, true>) : run(k_simulate<MODE, BB, false, true>);
  return a.issue ? run(k_simulate<MODE, BB, true, false>) : run(k_simulate<MODE, BB, false, false>);
}

}  // namespace

size_t simulate_smem_bytes(int warps, int sem_cap, int frame_depth) {
  return (size_t)12 * sem_cap + 3 * 8 + (size_t)8 * warps + sizeof(Frame) * (size_t)warps * frame_depth +
         (size_t)16 * warps + 16;
}

cudaError_t launch_simulate(const SimArgs& a, bool barrier, int num_sms, cudaStream_t s) {
  if (a.n_programs == 0) return cudaSuccess;
  const size_t smem = simulate_smem_bytes(a.warps, a.sem_cap, a.frame_depth);
  if (a.mode == SYNC_THR_PERLOOP)
    return barrier ? launch3<SYNC_THR_PERLOOP, true>(a, smem, num_sms, s)
                   : launch3<SYNC_THR_PERLOOP, false>(a, smem, num_sms, s);
  if (a.mode == SYNC_THR_PERENGINE)
    return barrier ? launch3<SYNC_THR_PERENGINE, true>(a, smem, num_sms, s)
                   : launch3<SYNC_THR_PERENGINE, false>(a, smem, num_sms, s);
  return barrier ? launch3<SYNC_THR_COUNT, true>(a, smem, num_sms, s)
                 : launch3<SYNC_THR_COUNT, false>(a, smem, num_sms, s);
}

}  // namespace syncgb
