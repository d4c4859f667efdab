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

// One warp per split program: the pieces' start states in order, the
// program's makespan and status; the checksum is zeroed for the fix-up pass
// to accumulate.  State variable v < ne is engine v's cursor, ne + v its
// last retire (stored at x[64 * piece + v] and x[64 * piece + 32 + v]).
template <bool BB>
__global__ void k_piece_resolve(const SweepArgs a, int n_split) {
  const int w = (int)((blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5), lane = threadIdx.x & 31;
  if (w >= n_split) return;
  if (*(volatile int32_t*)(a.pcs.fail + w)) return;
  const SplitProg sp = a.pcs.split[w];
  const int ne = sp.ne;
  if (BB) {
    // after L's statement barrier every engine is at c_barrier; each piece
    // ends with a barrier release, its duration after its start
    int64_t R = a.prm.c_barrier;
    for (int j = 0; j < sp.n_pieces; ++j) {
      const int piece = sp.first_piece + j;
      if (lane < ne) {
        a.pcs.x[(int64_t)piece * 64 + lane] = (int32_t)R;
        a.pcs.x[(int64_t)piece * 64 + 32 + lane] = 0;
      }
      R += __ldg(a.pcs.out + (int64_t)piece * a.pcs.probes * 64);   // probe 0, engine 0: the release
    }
    if (lane == 0) {
      a.makespan[sp.prog] = (int32_t)R;
      a.status[sp.prog] = SYNC_PROG_OK;
      a.checksum[sp.prog] = 0ull;
    }
    return;
  }
  // barrier-free: after L's statement (r-hat := 0, unless the trip register
  // is elided) every cursor is at that cost and nothing has retired
  const bool elide = a.prm.trip_register_elision && __ldg(a.lflag + sp.loop);
  const int nv = 2 * ne;
  // lane holds variables lane and lane + 32 (index v: cursor v < ne, retire v - ne)
  int64_t x0 = lane < nv ? (lane < ne ? (elide ? 0 : a.prm.c_regop) : 0) : 0;
  int64_t x1 = 0;
  for (int j = 0; j < sp.n_pieces; ++j) {
    const int piece = sp.first_piece + j;
    auto slot = [ne](int v) { return v < ne ? v : 32 + v - ne; };
    if (lane < nv) a.pcs.x[(int64_t)piece * 64 + slot(lane)] = (int32_t)x0;
    if (lane + 32 < nv) a.pcs.x[(int64_t)piece * 64 + slot(lane + 32)] = (int32_t)x1;
    int64_t y0 = -1, y1 = -1;                    // -1: no path (times are >= 0)
    for (int q = 0; q < nv; ++q) {
      const int64_t xq = q < 32 ? __shfl_sync(0xffffffffu, x0, q) : __shfl_sync(0xffffffffu, x1, q - 32);
      const int32_t* o = a.pcs.out + ((int64_t)piece * a.pcs.probes + q) * 64;
      if (lane < nv) {
        const int32_t r = __ldg(o + slot(lane));
        if (r >= kProbe) y0 = max(y0, (int64_t)(r - kProbe) + xq);
      }
      if (lane + 32 < nv) {
        const int32_t r = __ldg(o + slot(lane + 32));
        if (r >= kProbe) y1 = max(y1, (int64_t)(r - kProbe) + xq);
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

// Blocks (piece, y): instructions y, y + gridDim.y, ... of the piece's
// program; every instance of the piece gets its true issue and retire times
// from the stored ones (see the top of this file) and adds its checksum
// term; the timelines, if requested, are written here.
template <bool BB>
__global__ void __launch_bounds__(kValThreads) k_piece_fixup(const SweepArgs a, const int32_t* __restrict__ cnt) {
  __shared__ int32_t xs[64];
  __shared__ unsigned long long part[kValThreads / 32];
  const int piece = blockIdx.x;
  const PieceInfo pc = a.pcs.piece[piece];
  if (*(volatile int32_t*)(a.pcs.fail + pc.split)) return;
  const SplitProg sp = a.pcs.split[pc.split];
  const int j = piece - sp.first_piece, ne = sp.ne, nv = BB ? 1 : 2 * ne;
  if (threadIdx.x < 64) xs[threadIdx.x] = a.pcs.x[(int64_t)piece * 64 + threadIdx.x];
  __syncthreads();
  const int32_t* __restrict__ pt = a.pcs.ptimes;
  const int64_t N = a.pcs.plen, tl = pc.tl[BB ? 0 : 1];
  const int64_t ordv = 2 * (int64_t)a.pcs.probes * N;
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
      if (BB) {
        issue = __ldg(pt + i) + xs[0];
        retire = __ldg(pt + N + i) + xs[0];
      } else {
        int64_t bi = -1, br = -1;
        for (int q = 0; q < nv; ++q) {
          const int32_t xq = xs[q < ne ? q : 32 + q - ne];
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
  return cudaGetLastError();
}

template <int MODE, bool BB>
cudaError_t pieces(const SweepArgs& a, const VDep* vdep, const int32_t* cnt, int n_split, int num_sms,
                   cudaStream_t s) {
  const size_t smem = sweep_smem_bytes(a.sem_cap, a.frame_depth, a.ring);
  k_piece_validate<MODE, BB><<<a.pcs.n_pieces, kValThreads, 0, s>>>(a, vdep, cnt);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  // the probe / relative runs, storing every instance's times
  e = launch_items(k_sweep<MODE, BB, true, false, true>, a, (int64_t)a.pcs.n_pieces * a.pcs.probes, smem,
                   num_sms, s);
  if (e != cudaSuccess) return e;
  k_piece_resolve<BB><<<(n_split * 32 + 255) / 256, 256, 0, s>>>(a, n_split);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  // (piece, instruction slice) blocks: about 2048 or more in all
  const int ys = std::max(1, std::min(a.pcs.nx_max, (2048 + a.pcs.n_pieces - 1) / a.pcs.n_pieces));
  k_piece_fixup<BB><<<dim3(a.pcs.n_pieces, ys), kValThreads, 0, s>>>(a, cnt);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_pieces(const SweepArgs& a, bool barrier, const VDep* vdep, const int32_t* cnt, int n_split,
                          int num_sms, cudaStream_t s) {
  if (a.pcs.n_pieces == 0 || n_split == 0) return cudaSuccess;
  if (a.mode == SYNC_THR_PERLOOP)
    return barrier ? pieces<SYNC_THR_PERLOOP, true>(a, vdep, cnt, n_split, num_sms, s)
                   : pieces<SYNC_THR_PERLOOP, false>(a, vdep, cnt, n_split, num_sms, s);
  if (a.mode == SYNC_THR_PERENGINE)
    return barrier ? pieces<SYNC_THR_PERENGINE, true>(a, vdep, cnt, n_split, num_sms, s)
                   : pieces<SYNC_THR_PERENGINE, false>(a, vdep, cnt, n_split, num_sms, s);
  return barrier ? pieces<SYNC_THR_COUNT, true>(a, vdep, cnt, n_split, num_sms, s)
                 : pieces<SYNC_THR_COUNT, false>(a, vdep, cnt, n_split, num_sms, s);
}

}  // namespace syncgb
