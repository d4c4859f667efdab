// Piece-parallel simulation of large programs (PieceArgs in enc.h).
//
// A split program's top-level body is one loop L; its pieces are runs of
// consecutive iterations of L, each simulated by one warp with the sweep's
// code (k_sweep<..., PIECE>).  Exactness rests on two facts:
//   - every wait of a piece targets an increment the piece produces, which
//     the validation below checks against the thresholds of the call (a
//     program that fails it, or whose piece hits a deadlock or a wait
//     reaching forward, is simulated whole by the ordinary sweep), so a
//     piece depends on the rest of the program only through the engines'
//     cursors and last retire times at its start;
//   - under the timing model every time in a piece is the maximum, over
//     paths from those start values, of a start value plus a sum of costs
//     (all costs >= 0, no constant terms), so the piece's end state is a
//     max-plus linear map of its start state.  Barrier scheme: a barrier
//     release precedes every piece (every engine at the release time, the
//     last retires below it), so the map is a shift by the piece's duration.
//     Barrier-free: probe q runs the piece with state variable q at kProbe
//     and the others at 0; since no path weight reaches kProbe (the time
//     bound of a split program is below it), output o of probe q is
//     kProbe + M[o][q] when o depends on q and below kProbe otherwise.
// The pieces of a program are then composed in order (x_{j+1} = M_j x_j).  The
// same linearity holds for every instance's issue and retire times, which
// the piece runs store (per probe, with the instance's position in its
// engine's stream): a memory-bound pass then forms the true times from the
// start states -- shifted by the piece's start (barrier scheme), or the
// maximum over the probes of stored time - kProbe + start value (barrier-
// free) -- for the checksum and the timelines.
#include <algorithm>

#include "sweep.cuh"

namespace syncgb {
namespace {

constexpr int kValThreads = 256;
constexpr int kSpecRounds = 4;              // rounds of speculation before a program is simulated whole

// One block per piece: every pair of the piece's consumer instances must
// wait for nothing (threshold <= 0) or for an increment beyond its
// semaphore's published increments at the piece start.  The first piece of
// a program also checks the program's static time bound (below kProbe for
// the probes; the sweep reports an overflow itself).
template <int MODE, bool BB>
__global__ void __launch_bounds__(kValThreads) k_piece_validate(const SweepArgs a, const VDep* __restrict__ vdep,
                                                                const int32_t* __restrict__ cnt) {
  const int piece = blockIdx.x;
  const PieceInfo pc = a.pcs.piece[piece];
  if (*(volatile int32_t*)(a.pcs.fail + pc.split)) return;
  const SplitProg sp = a.pcs.split[pc.split];
  const int j = piece - sp.first_piece;
  if (j == 0 && threadIdx.x == 0) {
    const int32_t cwait = MODE == SYNC_THR_COUNT ? a.prm.c_wait_ops_count : a.prm.c_wait_ops_perloop;
    if (time_bound<MODE, BB>(a.prog[pc.prog], a.prm, cwait) >= (unsigned long long)kProbe)
      atomicExch(a.pcs.fail + pc.split, 1);
  }
  bool bad = false;
  for (int v = sp.vdep0; v < sp.vdep1; ++v) {
    const VDep D = vdep[v];
    const int32_t lo = __ldg(cnt + sp.cnt_base + (int64_t)j * sp.nx + D.cons);
    const int32_t hi = __ldg(cnt + sp.cnt_base + (int64_t)(j + 1) * sp.nx + D.cons);
    const int32_t pub = __ldg(a.pcs.pub + pc.pub_off[MODE] + D.sem[MODE]);
    for (int32_t g = lo + threadIdx.x; g < hi; g += kValThreads) {
      const int32_t T = __ldg(a.thr + D.seg + g);
      bad = bad || (T > 0 && T <= pub);
    }
  }
  if (__syncthreads_or(bad) && threadIdx.x == 0) atomicExch(a.pcs.fail + pc.split, 1);
}

// The state of a split program after L's statement, barrier-free: r-hat :=
// 0 on every engine (unless the trip register is elided), nothing retired.
__device__ __forceinline__ int32_t start_cursor(const SweepArgs& a, const SplitProg& sp) {
  const bool elide = a.prm.trip_register_elision && __ldg(a.lflag + sp.loop);
  return elide ? 0 : a.prm.c_regop;
}

// Slot of state variable v (cursor v < ne, last retire v - ne) in a 64-entry state.
__device__ __forceinline__ int slot_of(int v, int ne) { return v < ne ? v : 32 + v - ne; }

// One warp per split program: the pieces' start states in order, the
// program's makespan and status; the checksum is zeroed for the fix-up pass
// to accumulate.  Barrier scheme: every piece runs from a release, so it is
// shifted by its start (stored in shift).  Barrier-free, probed programs:
// the probes' end states give each piece's max-plus map (x at 64 * piece).
template <bool BB>
__global__ void k_piece_resolve(const SweepArgs a, int n_split) {
  const int w = (int)((blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5), lane = threadIdx.x & 31;
  if (w >= n_split) return;
  if (*(volatile int32_t*)(a.pcs.fail + w)) return;
  if (!BB && a.pcs.cls[w]) return;                 // speculated, not probed
  const SplitProg sp = a.pcs.split[w];
  const int ne = sp.ne;
  if (BB) {
    // after L's statement barrier every engine is at c_barrier; each piece
    // ends with a barrier release, its duration after its start
    int64_t R = a.prm.c_barrier;
    for (int j = 0; j < sp.n_pieces; ++j) {
      const int piece = sp.first_piece + j;
      if (lane == 0) a.pcs.shift[piece] = (int32_t)R;
      R += __ldg(a.pcs.out + (int64_t)piece * a.pcs.out_probes * 64);   // run 0, engine 0: the release
    }
    if (lane == 0) {
      a.makespan[sp.prog] = (int32_t)R;
      a.status[sp.prog] = SYNC_PROG_OK;
      a.checksum[sp.prog] = 0ull;
    }
    return;
  }
  const int nv = 2 * ne;
  // lane holds variables lane and lane + 32
  int64_t x0 = lane < ne ? start_cursor(a, sp) : 0, x1 = 0;
  for (int j = 0; j < sp.n_pieces; ++j) {
    const int piece = sp.first_piece + j;
    if (lane < nv) a.pcs.x[(int64_t)piece * 64 + slot_of(lane, ne)] = (int32_t)x0;
    if (lane + 32 < nv) a.pcs.x[(int64_t)piece * 64 + slot_of(lane + 32, ne)] = (int32_t)x1;
    int64_t y0 = -1, y1 = -1;                    // -1: no path (times are >= 0)
    const int32_t* o = a.pcs.out + (int64_t)piece * a.pcs.out_probes * 64;
    // the probes' outputs of this lane's variables, 8 loads in flight at a time
    for (int q0 = 0; q0 < nv; q0 += 8) {
      int32_t r0[8], r1[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int q = q0 + k;
        r0[k] = q < nv && lane < nv ? __ldg(o + (int64_t)q * 64 + slot_of(lane, ne)) : 0;
        r1[k] = q < nv && lane + 32 < nv ? __ldg(o + (int64_t)q * 64 + slot_of(lane + 32, ne)) : 0;
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int q = q0 + k;
        if (q >= nv) break;
        const int64_t xq = q < 32 ? __shfl_sync(0xffffffffu, x0, q) : __shfl_sync(0xffffffffu, x1, q - 32);
        if (r0[k] >= kProbe) y0 = max(y0, (int64_t)(r0[k] - kProbe) + xq);
        if (r1[k] >= kProbe) y1 = max(y1, (int64_t)(r1[k] - kProbe) + xq);
      }
    }
    x0 = y0;
    x1 = y1;
  }
  int64_t ms = 0;
  if (lane < nv) ms = max(ms, x0);
  if (lane + 32 < nv) ms = max(ms, x1);
  for (int o = 16; o > 0; o >>= 1) ms = max(ms, (int64_t)__shfl_xor_sync(0xffffffffu, ms, o));
  if (lane == 0) {
    a.makespan[sp.prog] = (int32_t)ms;
    a.status[sp.prog] = SYNC_PROG_OK;
    a.checksum[sp.prog] = 0ull;
  }
}

// Speculation, before the first round: every speculated program's first
// piece runs from its true start state; the others wait for a guess.
__global__ void k_spec_init(const SweepArgs a, int n_split) {
  const int w = (int)((blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5), lane = threadIdx.x & 31;
  if (w >= n_split || !a.pcs.cls[w] || *(volatile int32_t*)(a.pcs.fail + w)) return;
  const SplitProg sp = a.pcs.split[w];
  for (int j = lane; j < sp.n_pieces; j += 32) {
    a.pcs.need[sp.first_piece + j] = j == 0;
    a.pcs.has[sp.first_piece + j] = 0;
  }
  if (lane < 32) {
    a.pcs.xhat[(int64_t)sp.first_piece * 64 + lane] = lane < sp.ne ? start_cursor(a, sp) : 0;
    a.pcs.xhat[(int64_t)sp.first_piece * 64 + 32 + lane] = 0;
  }
  if (lane == 0) a.pcs.vp[w] = 0;
}

// Speculation, after a round: one warp per speculated program walks its
// pieces from the first one not yet accepted, with that piece's true start
// state.  A piece that ran from the true start plus one shift c for every
// state variable is accepted (its times and end state are the stored ones
// plus c, the timing model being max-plus homogeneous), and the next piece's
// true start is its end state.  At the first piece that has not run, every
// remaining piece is guessed to start like it; at the first rejected one, it
// runs again from its true start and every later piece from the end state
// of its predecessor's last run.  After the last round a program with
// pieces left is simulated whole by the sweep.
__global__ void k_spec_resolve(const SweepArgs a, int n_split, int last_round) {
  const int w = (int)((blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5), lane = threadIdx.x & 31;
  if (w >= n_split || !a.pcs.cls[w] || *(volatile int32_t*)(a.pcs.fail + w)) return;
  const SplitProg sp = a.pcs.split[w];
  const int ne = sp.ne, n = sp.n_pieces;
  int j = a.pcs.vp[w];
  if (j >= n) return;
  // the true start of piece j, lane v < ne: cursor v, lane 32 + v: retire v
  int64_t xt = 0, xr = 0;
  if (lane < ne) {
    if (j == 0) { xt = start_cursor(a, sp); xr = 0; }
    else {
      xt = a.pcs.x[(int64_t)(sp.first_piece + j) * 64 + lane];
      xr = a.pcs.x[(int64_t)(sp.first_piece + j) * 64 + 32 + lane];
    }
  }
  for (; j < n; ++j) {
    const int piece = sp.first_piece + j;
    if (!*(volatile int32_t*)(a.pcs.has + piece)) {
      // never ran: guess that every remaining piece starts like this one
      for (int k = j; k < n; ++k) {
        if (lane < ne) {
          a.pcs.xhat[(int64_t)(sp.first_piece + k) * 64 + lane] = (int32_t)xt;
          a.pcs.xhat[(int64_t)(sp.first_piece + k) * 64 + 32 + lane] = (int32_t)xr;
        }
        if (lane == 0) a.pcs.need[sp.first_piece + k] = 1;
      }
      break;
    }
    const int64_t ht = lane < ne ? a.pcs.xhat[(int64_t)piece * 64 + lane] : 0;
    const int64_t hr = lane < ne ? a.pcs.xhat[(int64_t)piece * 64 + 32 + lane] : 0;
    const int64_t c = __shfl_sync(0xffffffffu, xt - ht, 0);
    if (__all_sync(0xffffffffu, lane >= ne || (xt - ht == c && xr - hr == c))) {
      if (lane == 0) a.pcs.shift[piece] = (int32_t)c;
      if (lane < ne) {                            // the next piece's true start
        xt = a.pcs.out[(int64_t)piece * a.pcs.out_probes * 64 + lane] + c;
        xr = a.pcs.out[(int64_t)piece * a.pcs.out_probes * 64 + 32 + lane] + c;
        if (j + 1 < n) {
          a.pcs.x[(int64_t)(piece + 1) * 64 + lane] = (int32_t)xt;
          a.pcs.x[(int64_t)(piece + 1) * 64 + 32 + lane] = (int32_t)xr;
        }
      }
      continue;
    }
    // rejected: again from its true start; the later pieces from their
    // predecessors' last end states (read before any is overwritten)
    for (int k = n - 1; k > j; --k) {
      if (lane < ne) {
        const int pk = sp.first_piece + k;
        a.pcs.xhat[(int64_t)pk * 64 + lane] = a.pcs.out[(int64_t)(pk - 1) * a.pcs.out_probes * 64 + lane];
        a.pcs.xhat[(int64_t)pk * 64 + 32 + lane] = a.pcs.out[(int64_t)(pk - 1) * a.pcs.out_probes * 64 + 32 + lane];
      }
      if (lane == 0) a.pcs.need[sp.first_piece + k] = 1;
    }
    if (lane < ne) {
      a.pcs.xhat[(int64_t)piece * 64 + lane] = (int32_t)xt;
      a.pcs.xhat[(int64_t)piece * 64 + 32 + lane] = (int32_t)xr;
    }
    if (lane == 0) a.pcs.need[piece] = 1;
    break;
  }
  if (lane == 0) a.pcs.vp[w] = j;
  if (j == n) {                                  // every piece accepted
    int64_t ms = lane < ne ? max(xt, xr) : 0;
    for (int o = 16; o > 0; o >>= 1) ms = max(ms, (int64_t)__shfl_xor_sync(0xffffffffu, ms, o));
    if (lane == 0) {
      a.makespan[sp.prog] = (int32_t)ms;
      a.status[sp.prog] = SYNC_PROG_OK;
      a.checksum[sp.prog] = 0ull;
    }
  } else if (last_round && lane == 0) {
    atomicExch(a.pcs.fail + w, 1);
  }
}

// Blocks (piece, y): instructions y, y + gridDim.y, ... of the piece's
// program; every instance of the piece gets its true issue and retire times
// from the stored ones (see the top of this file) and adds its checksum
// term; the timelines, if requested, are written here.  Stored times of
// single runs (barrier scheme, speculated pieces) are in `one` (issue,
// retire, position in the engine's stream per instance of the split
// programs, one_len of them), those of the probes in a.pcs.ptimes.
template <bool BB>
__global__ void __launch_bounds__(kValThreads) k_piece_fixup(const SweepArgs a, const int32_t* __restrict__ cnt,
                                                             const int32_t* __restrict__ one, int64_t one_len) {
  __shared__ int32_t xs[64];
  __shared__ unsigned long long part[kValThreads / 32];
  const int piece = blockIdx.x;
  const PieceInfo pc = a.pcs.piece[piece];
  if (*(volatile int32_t*)(a.pcs.fail + pc.split)) return;
  const SplitProg sp = a.pcs.split[pc.split];
  const bool shifted = BB || a.pcs.cls[pc.split];
  const int j = piece - sp.first_piece, ne = sp.ne, nv = 2 * ne;
  if (threadIdx.x < 64) xs[threadIdx.x] = shifted ? 0 : a.pcs.x[(int64_t)piece * 64 + threadIdx.x];
  __syncthreads();
  const int32_t c = shifted ? a.pcs.shift[piece] : 0;
  const int32_t* __restrict__ pt = shifted ? one : a.pcs.ptimes;
  const int64_t N = shifted ? one_len : a.pcs.plen, tl = pc.tl[shifted ? 0 : 1];
  const int64_t ordv = 2 * (int64_t)(shifted ? 1 : a.pcs.probes) * N;
  unsigned long long chk = 0;
  for (int x = blockIdx.y; x < sp.nx; x += gridDim.y) {
    const int32_t lo = __ldg(cnt + sp.cnt_base + (int64_t)j * sp.nx + x);
    const int32_t hi = __ldg(cnt + sp.cnt_base + (int64_t)(j + 1) * sp.nx + x);
    if (lo >= hi) continue;
    const int64_t o0 = __ldg(a.inst_off + sp.x0 + x);
    const uint32_t e = (uint32_t)__ldg(a.pcs.xeng + sp.x0 + x);
    for (int32_t g = lo + (int32_t)threadIdx.x; g < hi; g += kValThreads) {
      const int64_t o = o0 + g, i = o + tl;
      int32_t issue, retire;
      if (shifted) {
        issue = __ldg(pt + i) + c;
        retire = __ldg(pt + N + i) + c;
      } else {
        int64_t bi = -1, br = -1;
        for (int q = 0; q < nv; ++q) {
          const int32_t xq = xs[slot_of(q, ne)];
          const int32_t ti = __ldg(pt + 2 * q * N + i), tr = __ldg(pt + (2 * q + 1) * N + i);
          if (ti >= kProbe) bi = max(bi, (int64_t)(ti - kProbe) + xq);
          if (tr >= kProbe) br = max(br, (int64_t)(tr - kProbe) + xq);
        }
        issue = (int32_t)bi;
        retire = (int32_t)br;
      }
      chk += inst_term(issue, retire, e, (uint32_t)__ldg(pt + ordv + i));
      if (a.issue) {
        a.issue[o] = issue;
        a.retire[o] = retire;
      }
    }
  }
  for (int o = 16; o > 0; o >>= 1) chk += __shfl_xor_sync(0xffffffffu, chk, o);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = chk;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long t = 0;
    for (int w = 0; w < kValThreads / 32; ++w) t += part[w];
    atomicAdd(a.checksum + sp.prog, t);
  }
}

template <class K>
cudaError_t launch_items(K kern, const SweepArgs& a, int64_t items, size_t smem, int num_sms, cudaStream_t s) {
  if (items <= 0) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kWarps * 32, smem);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) return cudaErrorInvalidConfiguration;
  const long long want = (items + kWarps - 1) / kWarps;
  const long long cap = (long long)num_sms * per_sm;
  const int grid = (int)(want < cap ? want : cap);
  e = cudaMemsetAsync(a.next_slot, 0, sizeof(int32_t), s);
  if (e != cudaSuccess) return e;
  kern<<<grid, kWarps * 32, smem, s>>>(a);
  return launched();
}

template <int MODE, bool BB>
cudaError_t pieces(const SweepArgs& a, const PieceLaunch& L, int num_sms, cudaStream_t s) {
  const size_t smem = sweep_smem_bytes(a.sem_cap, a.frame_depth, a.ring);
  const int warp_blocks = (L.n_split * 32 + 255) / 256;
  k_piece_validate<MODE, BB><<<a.pcs.n_pieces, kValThreads, 0, s>>>(a, L.vdep, L.cnt);
  cudaError_t e = launched();
  if (e != cudaSuccess) return e;
  // barrier scheme, or barrier-free probes: one launch of runs storing
  // every instance's times, then the composition
  if (BB || L.n_probed > 0) {
    SweepArgs p = a;
    p.pcs.spec = 0;
    if (BB) { p.pcs.ptimes = L.one; p.pcs.plen = L.one_len; }
    e = launch_items(k_sweep<MODE, BB, true, false, true>, p, (int64_t)p.pcs.n_pieces * p.pcs.probes, smem,
                     num_sms, s);
    if (e != cudaSuccess) return e;
    k_piece_resolve<BB><<<warp_blocks, 256, 0, s>>>(p, L.n_split);
    if ((e = launched()) != cudaSuccess) return e;
  }
  // barrier-free speculation: rounds of runs and acceptance checks
  if (!BB && L.n_spec > 0) {
    SweepArgs p = a;
    p.pcs.spec = 1;
    p.pcs.probes = 1;
    p.pcs.ptimes = L.one;
    p.pcs.plen = L.one_len;
    k_spec_init<<<warp_blocks, 256, 0, s>>>(p, L.n_split);
    if ((e = launched()) != cudaSuccess) return e;
    for (int r = 0; r < kSpecRounds; ++r) {
      e = launch_items(k_sweep<MODE, BB, true, false, true>, p, p.pcs.n_pieces, smem, num_sms, s);
      if (e != cudaSuccess) return e;
      k_spec_resolve<<<warp_blocks, 256, 0, s>>>(p, L.n_split, r == kSpecRounds - 1);
      if ((e = launched()) != cudaSuccess) return e;
    }
  }
  // (piece, instruction slice) blocks: about 2048 or more in all
  const int ys = std::max(1, std::min(a.pcs.nx_max, (2048 + a.pcs.n_pieces - 1) / a.pcs.n_pieces));
  k_piece_fixup<BB><<<dim3(a.pcs.n_pieces, ys), kValThreads, 0, s>>>(a, L.cnt, L.one, L.one_len);
  return launched();
}

}  // namespace

cudaError_t launch_pieces(const SweepArgs& a, bool barrier, const PieceLaunch& L, int num_sms, cudaStream_t s) {
  if (a.pcs.n_pieces == 0 || L.n_split == 0) return cudaSuccess;
  if (a.mode == SYNC_THR_PERLOOP)
    return barrier ? pieces<SYNC_THR_PERLOOP, true>(a, L, num_sms, s) : pieces<SYNC_THR_PERLOOP, false>(a, L, num_sms, s);
  if (a.mode == SYNC_THR_PERENGINE)
    return barrier ? pieces<SYNC_THR_PERENGINE, true>(a, L, num_sms, s)
                   : pieces<SYNC_THR_PERENGINE, false>(a, L, num_sms, s);
  return barrier ? pieces<SYNC_THR_COUNT, true>(a, L, num_sms, s) : pieces<SYNC_THR_COUNT, false>(a, L, num_sms, s);
}

}  // namespace syncgb
