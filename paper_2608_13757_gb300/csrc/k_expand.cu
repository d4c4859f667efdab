// Load-time expansion of the trip prefix sums into parent-iteration indices,
// the derived per-iteration arrays of the threshold kernels, and (on first
// per-engine use) the engine-stream positions of producer instances.
//
// For every loop l and every global iteration g of l, pidx_l[g] is the
// parent's global iteration j with rowptr_l[j] <= g < rowptr_l[j+1] (the CSR
// row of g).
#include "enc.h"

namespace syncgb {
namespace {

constexpr int kThreads = 256;

// One warp per 32 consecutive rowptr entries (rows: parent iterations of
// some iteration space, plus each space's closing entry).  The rows' child
// iterations are consecutive in the parent-index pool, so the warp writes
// one contiguous range, each lane finding the row of an entry by a binary
// search over the 32 row starts (shuffles).
__global__ void __launch_bounds__(kThreads)
k_expand(const LoopInfo* __restrict__ loop, const int32_t* __restrict__ tile_rp,
         const int32_t* __restrict__ rowptr, int64_t n_rowptr, int32_t* __restrict__ pidx, int64_t n_iters) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (kThreads / 32);
  for (int64_t w = (int64_t)blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5); w * 32 < n_rowptr; w += warps) {
    const int64_t r = w * 32 + lane;
    int64_t b = n_iters, e = n_iters;             // lanes past the last entry: empty, at the end
    int32_t j = 0;
    if (r < n_rowptr) {
      const int64_t t = r / kTilePairs;
      int lo = tile_rp[t], hi = tile_rp[t + 1];
      while (lo < hi) {                           // largest space with rowptr_off <= r
        const int mid = (lo + hi + 1) >> 1;
        if (loop[mid].rowptr_off <= r) lo = mid; else hi = mid - 1;
      }
      const LoopInfo L = loop[lo];
      j = (int32_t)(r - L.rowptr_off);
      b = L.pidx_off + rowptr[r];
      e = j < L.n_parent ? L.pidx_off + rowptr[r + 1] : b;
    }
    const int64_t wb = __shfl_sync(0xffffffffu, b, 0), we = __shfl_sync(0xffffffffu, e, 31);
    for (int64_t base = wb; base < we; base += 32) {
      const int64_t k = base + lane;
      int lo = 0, hi = 31;                        // largest row with start <= k
      for (int step = 0; step < 5; ++step) {
        const int mid = (lo + hi + 1) >> 1;
        const int64_t bm = __shfl_sync(0xffffffffu, b, mid);
        if (bm <= k) lo = mid; else hi = mid - 1;
      }
      const int32_t v = __shfl_sync(0xffffffffu, j, lo);
      if (k < we) pidx[k] = v;
    }
  }
}

// One thread per (mode, op record or lane): the record's semaphore entry
// copied from its instruction's.
__global__ void __launch_bounds__(kThreads)
k_sem_records(const int4* __restrict__ xsem, int64_t n_instrs, const int4* __restrict__ ops, int64_t n_ops,
              const int4* __restrict__ lrec, int64_t n_lanes, int4* __restrict__ opsem, int4* __restrict__ lsem) {
  const int64_t per = n_ops + n_lanes, n = kModes * per;
  const int64_t stride = (int64_t)gridDim.x * kThreads;
  for (int64_t q = (int64_t)blockIdx.x * kThreads + threadIdx.x; q < n; q += stride) {
    const int64_t m = q / per, r = q - m * per;
    if (r < n_ops) {
      const int32_t x = ops[r].x;
      opsem[m * n_ops + r] = x >= 0 ? xsem[m * n_instrs + x] : make_int4(-1, 0, 0, 0);
    } else {
      const int64_t i = r - n_ops;
      lsem[m * n_lanes + i] = xsem[m * n_instrs + lrec[i].x];
    }
  }
}

// One CTA per tile of kTilePairs derived entries: the jobs that overlap the
// tile (with the path offsets of ancestor jobs) are staged in shared memory,
// then each thread fills entries of the tile.  Tiles overlapping more jobs
// than the stage holds look the jobs up in global memory.
constexpr int kStageJobs = 64;

__device__ __forceinline__ int32_t derive_one(const DeriveJob& J, const int64_t* jpath, int64_t q,
                                              const int32_t* __restrict__ rowptr,
                                              const int32_t* __restrict__ pidx) {
  const int32_t g = (int32_t)(q - J.out);
  if (g >= J.n) return 0;                         // padding entries
  if (J.kind == DERIVE_TSTART) return rowptr[J.b + pidx[J.a + g]];
  int32_t v = g;
  for (int i = 0; i < J.up; ++i) v = pidx[jpath[i] + v];
  return v;
}

__global__ void __launch_bounds__(kThreads)
k_derive(const DeriveJob* __restrict__ jobs, const int32_t* __restrict__ tile_job,
         const int32_t* __restrict__ rowptr, const int32_t* __restrict__ pidx,
         const int64_t* __restrict__ path, int32_t* __restrict__ out, int64_t n) {
  __shared__ DeriveJob sj[kStageJobs];
  __shared__ int64_t sp[kStageJobs][SYNC_MAX_DEPTH];
  const int64_t n_tiles = (n + kTilePairs - 1) / kTilePairs;
  for (int64_t t = blockIdx.x; t < n_tiles; t += gridDim.x) {
    const int j0 = tile_job[t], j1 = tile_job[t + 1];
    const int nj = j1 - j0 + 1;
    const bool staged = nj <= kStageJobs;
    __syncthreads();                              // the previous tile's readers are done
    if (staged) {
      for (int i = threadIdx.x; i < nj; i += kThreads) sj[i] = jobs[j0 + i];
      __syncthreads();
      for (int i = threadIdx.x; i < nj * SYNC_MAX_DEPTH; i += kThreads) {
        const int jj = i / SYNC_MAX_DEPTH, u = i - jj * SYNC_MAX_DEPTH;
        if (sj[jj].kind == DERIVE_ANC && u < sj[jj].up) sp[jj][u] = path[sj[jj].a + u];
      }
      __syncthreads();
    }
    const int64_t q0 = t * kTilePairs, q1 = q0 + kTilePairs < n ? q0 + kTilePairs : n;
    for (int64_t q = q0 + threadIdx.x; q < q1; q += kThreads) {
      int lo = 0, hi = nj - 1;                    // largest job with out <= q
      if (staged) {
        while (lo < hi) {
          const int mid = (lo + hi + 1) >> 1;
          if (sj[mid].out <= q) lo = mid; else hi = mid - 1;
        }
        out[q] = derive_one(sj[lo], sp[lo], q, rowptr, pidx);
      } else {
        lo = j0, hi = j1;
        while (lo < hi) {
          const int mid = (lo + hi + 1) >> 1;
          if (jobs[mid].out <= q) lo = mid; else hi = mid - 1;
        }
        const DeriveJob J = jobs[lo];
        int64_t jp[SYNC_MAX_DEPTH];
        for (int u = 0; J.kind == DERIVE_ANC && u < J.up; ++u) jp[u] = path[J.a + u];
        out[q] = derive_one(J, jp, q, rowptr, pidx);
      }
    }
  }
}

// One thread per (program, engine), programs in descending-work order:
// walk the engine's op rows (its own instructions and the child-loop
// statements of each loop body, in body order) through every iteration,
// counting the engine's instances.
__global__ void __launch_bounds__(kThreads)
k_ordinals(const ProgInfo* __restrict__ prog, const int32_t* __restrict__ order, int32_t n_programs,
           int32_t ne_max, const int32_t* __restrict__ op_ptr, const int4* __restrict__ ops,
           const int32_t* __restrict__ rowptr, const int64_t* __restrict__ ord_off,
           int32_t* __restrict__ ord) {
  struct Frame { int32_t row, pos, g, g_end; };
  const int64_t stride = (int64_t)gridDim.x * kThreads;
  const int64_t n = (int64_t)n_programs * ne_max;
  for (int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x; t < n; t += stride) {
    const int32_t p = order[t / ne_max], e = (int32_t)(t % ne_max);
    const ProgInfo pi = prog[p];
    if (e >= pi.ne) continue;
    Frame st[SYNC_MAX_DEPTH + 1];
    int sp = 0;
    int32_t row = pi.le_base + e, pos = op_ptr[row], g = 0, g_end = 1, count = 0;
    for (;;) {
      const int4 op = ops[pos];
      if (op.x >= 0) {                              // a datapath instance of this engine
        ++count;
        const int64_t o = ord_off[op.x];
        if (o >= 0) ord[o + g] = count;
        ++pos;
      } else if (op.x == OP_LOOP) {                 // a child loop statement
        const int64_t rp = ((int64_t)(uint32_t)op.w << 32) | (uint32_t)op.z;
        const int32_t lo = rowptr[rp + g], hi = rowptr[rp + g + 1];
        ++pos;
        if (lo < hi) {
          st[sp++] = Frame{row, pos, g, g_end};
          row = op.y + e;
          pos = op_ptr[row];
          g = lo;
          g_end = hi;
        }
      } else if (++g < g_end) {                     // end of an iteration: the next one
        pos = op_ptr[row];
      } else if (sp > 0) {                          // end of the loop: back to the parent
        const Frame f = st[--sp];
        row = f.row; pos = f.pos; g = f.g; g_end = f.g_end;
      } else {
        break;                                      // the top-level loop runs once
      }
    }
  }
}

}  // namespace

cudaError_t launch_ordinals(const ProgInfo* prog, const int32_t* order, int32_t n_programs, int32_t ne_max,
                            const int32_t* op_ptr, const int4* ops, const int32_t* rowptr,
                            const int64_t* ord_off, int32_t* ord, int num_sms, cudaStream_t s) {
  const int64_t n = (int64_t)n_programs * ne_max;
  if (n == 0) return cudaSuccess;
  const int64_t want = (n + kThreads - 1) / kThreads;
  const int64_t cap = (int64_t)num_sms * 8;
  const int grid = (int)(want < cap ? want : cap);
  k_ordinals<<<grid, kThreads, 0, s>>>(prog, order, n_programs, ne_max, op_ptr, ops, rowptr, ord_off, ord);
  return launched();
}

cudaError_t launch_derive(const DeriveJob* jobs, const int32_t* tile_job, const int32_t* rowptr,
                          const int32_t* pidx, const int64_t* path, int32_t* derived, int64_t n,
                          int num_sms, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  const int64_t want = (n + kTilePairs - 1) / kTilePairs;
  const int64_t cap = (int64_t)num_sms * 8;
  const int grid = (int)(want < cap ? want : cap);
  k_derive<<<grid, kThreads, 0, s>>>(jobs, tile_job, rowptr, pidx, path, derived, n);
  return launched();
}

cudaError_t launch_sem_records(const int4* xsem, int64_t n_instrs, const int4* ops, int64_t n_ops,
                               const int4* lrec, int64_t n_lanes, int4* opsem, int4* lsem, int num_sms,
                               cudaStream_t s) {
  const int64_t n = kModes * (n_ops + n_lanes);
  if (n == 0) return cudaSuccess;
  const int64_t want = (n + kThreads - 1) / kThreads;
  const int64_t cap = (int64_t)num_sms * 8;
  const int grid = (int)(want < cap ? want : cap);
  k_sem_records<<<grid, kThreads, 0, s>>>(xsem, n_instrs, ops, n_ops, lrec, n_lanes, opsem, lsem);
  return launched();
}

cudaError_t launch_expand(const LoopInfo* loop, const int32_t* tile_rp, const int32_t* rowptr, int64_t n_rowptr,
                          int32_t* pidx, int64_t n_iters, int num_sms, cudaStream_t s) {
  if (n_iters == 0) return cudaSuccess;
  const int64_t want = (n_rowptr + kThreads - 1) / kThreads;
  const int64_t cap = (int64_t)num_sms * 8;
  const int grid = (int)(want < cap ? want : cap);
  k_expand<<<grid, kThreads, 0, s>>>(loop, tile_rp, rowptr, n_rowptr, pidx, n_iters);
  return launched();
}

}  // namespace syncgb
