// Load-time kernels: the derived per-iteration arrays of the threshold
// kernels, the per-mode semaphore records of the simulators, and (on first
// per-engine use) the engine-stream positions of producer instances.
#include <cstdlib>

#include "enc.h"

namespace syncgb {
namespace {

constexpr int kThreads = 256;
constexpr unsigned kFull = 0xffffffffu;

// One thread per op record or lane: the record's semaphore entries of the
// three modes copied from its instruction's.
__global__ void __launch_bounds__(kThreads)
k_sem_records(const int4* __restrict__ xsem, int64_t n_instrs, const int4* __restrict__ ops, int64_t n_ops,
              const int4* __restrict__ lrec, int64_t n_lanes, int4* __restrict__ opsem, int4* __restrict__ lsem) {
  const int64_t n = n_ops + n_lanes;
  const int64_t stride = (int64_t)gridDim.x * kThreads;
  for (int64_t r = (int64_t)blockIdx.x * kThreads + threadIdx.x; r < n; r += stride) {
    const bool op = r < n_ops;
    const int64_t i = op ? r : r - n_ops;
    const int32_t x = op ? ops[i].x : lrec[i].x;
    int4 v[kModes];
#pragma unroll
    for (int m = 0; m < kModes; ++m) v[m] = x >= 0 ? xsem[m * n_instrs + x] : make_int4(-1, 0, 0, 0);
    int4* out = op ? opsem : lsem;
    const int64_t per = op ? n_ops : n_lanes;
#pragma unroll
    for (int m = 0; m < kModes; ++m) out[m * per + i] = v[m];
  }
}

// One warp per 32 consecutive rows of the derive jobs (enc.h: each job's
// rows, then its padding row, jobs in pool order).  The tile table gives
// the job of the warp's first row; the 32 rows lie in that job and at most
// 31 after it, whose first rows the lanes load together, and each lane
// finds its row's job among them by a binary search over the lanes
// (shuffles).  Each lane then reads its row's range of the pool (trip
// prefix sums, composed for ancestors) and its value.  The rows' ranges follow each other, so the warp fills
// one contiguous range of the pool: a window of 32 entries inside one row
// takes that row's value with no search (long rows: a run of whole
// windows), a window across rows finds each entry's row by a binary search
// over the 32 row starts (shuffles).
__global__ void __launch_bounds__(kThreads)
k_derive(const DeriveJob* __restrict__ jobs, const int32_t* __restrict__ tile_job, int64_t n_rows,
         const int32_t* __restrict__ rowptr, const int64_t* __restrict__ path, int32_t* __restrict__ out,
         int64_t n, int wide) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (kThreads / 32);
  for (int64_t w = (int64_t)blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5); w * 32 < n_rows; w += warps) {
    const int64_t r = w * 32 + lane;
    const int32_t j0 = tile_job[w], j_last = tile_job[(w + 1) * 32 < n_rows ? w + 1 : (n_rows + 31) / 32];
    // lane i: the first row of job j0 + i (past the last job: beyond every row)
    const int64_t first = j0 + lane <= j_last ? jobs[j0 + lane].row0 : INT64_MAX;
    int jl = 0;                                   // the last lane whose job starts at or before row r
    for (int o = 16; o > 0; o >>= 1)
      if (__shfl_sync(kFull, first, jl + o) <= r) jl += o;
    int64_t b = n, e = n;                         // lanes past the last row: empty, at the end
    int32_t v = 0;
    if (r < n_rows) {
      const DeriveJob J = jobs[j0 + jl];
      const int64_t j = r - J.row0;
      if (j < J.nrows) {
        int64_t x0 = j, x1 = j + 1;
        if (J.kind == DERIVE_TSTART) {            // a trip of S: its first iteration
          x0 = rowptr[J.path + j];
          x1 = rowptr[J.path + j + 1];
          v = (int32_t)x0;
        } else {                                  // the iterations below S-iteration j
          for (int i = J.up - 1; i >= 0; --i) {
            const int64_t rp = path[J.path + i];
            x0 = rowptr[rp + x0];
            x1 = rowptr[rp + x1];
          }
          v = (int32_t)j;
        }
        b = J.out + x0;
        e = J.out + x1;
      } else {                                    // the padding row: zeros
        b = J.out + J.n;
        e = J.out + J.len;
      }
    }
    const int64_t wb = __shfl_sync(kFull, b, 0), we = __shfl_sync(kFull, e, 31);
    if (!wide && we - wb <= INT32_MAX - 64) {
      // offsets from the warp's first entry fit 32 bits (a job of 2^31
      // entries would not): 32-bit shuffles and compares
      const int32_t rb = (int32_t)(b - wb), re = (int32_t)(e - wb), rend = (int32_t)(we - wb);
      int32_t* o = out + wb;
      for (int32_t base = 0; base < rend;) {
        // the row holding entry `base`: the last lane whose range starts at
        // or before it (ranges ascend; an empty one shares its start with
        // the next)
        const int own = 31 - __clz(__ballot_sync(kFull, rb <= base));
        const int32_t oe = __shfl_sync(kFull, re, own);
        if (oe - base >= 32) {
          const int32_t ov = __shfl_sync(kFull, v, own);
          const int32_t stop = base + ((oe - base) & ~31);
          for (int32_t k = base + lane; k < stop; k += 32) o[k] = ov;
          base = stop;
          continue;
        }
        // the nonempty rows that meet the window, `own` first; an entry's row
        // is the last of them starting at or before it
        const unsigned rows = __ballot_sync(kFull, rb < re && rb < base + 32 && re > base);
        const int32_t k = base + lane;
        int jl = own;
        if (__popc(rows) <= 4) {
          for (unsigned rest = rows & (rows - 1); rest; rest &= rest - 1) {
            const int L = __ffs(rest) - 1;
            if (__shfl_sync(kFull, rb, L) <= k) jl = L;
          }
        } else {
          jl = 0;
          for (int step = 16; step > 0; step >>= 1)
            if (__shfl_sync(kFull, rb, jl + step) <= k) jl += step;
        }
        const int32_t val = __shfl_sync(kFull, v, jl);
        if (k < rend) o[k] = val;
        base += 32;
      }
      continue;
    }
    for (int64_t base = wb; base < we;) {
      const int own = 31 - __clz(__ballot_sync(kFull, b <= base));
      const int64_t oe = __shfl_sync(kFull, e, own);
      if (oe - base >= 32) {
        const int32_t ov = __shfl_sync(kFull, v, own);
        const int64_t stop = base + ((oe - base) & ~int64_t(31));
        for (int64_t k = base + lane; k < stop; k += 32) out[k] = ov;
        base = stop;
        continue;
      }
      const int64_t k = base + lane;
      int jl = 0;                                 // the last lane whose range starts at or before k
      for (int step = 16; step > 0; step >>= 1)
        if (__shfl_sync(kFull, b, jl + step) <= k) jl += step;
      const int32_t val = __shfl_sync(kFull, v, jl);
      if (k < we) out[k] = val;
      base += 32;
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

cudaError_t launch_derive(const DeriveJob* jobs, const int32_t* tile_job, int64_t n_rows, const int32_t* rowptr,
                          const int64_t* path, int32_t* derived, int64_t n, int num_sms, cudaStream_t s) {
  if (n_rows == 0) return cudaSuccess;
  const int64_t want = (n_rows + kThreads - 1) / kThreads;
  const int64_t cap = (int64_t)num_sms * 8;
  const int grid = (int)(want < cap ? want : cap);
  // SYNCGB_WIDE_INDEX=1 takes the 64-bit write path everywhere (tests use
  // it on small batches; otherwise only a warp's range past 2^31 entries does)
  const char* f = std::getenv("SYNCGB_WIDE_INDEX");
  const int wide = f && f[0] == '1' ? 1 : 0;
  k_derive<<<grid, kThreads, 0, s>>>(jobs, tile_job, n_rows, rowptr, path, derived, n, wide);
  return launched();
}

cudaError_t launch_sem_records(const int4* xsem, int64_t n_instrs, const int4* ops, int64_t n_ops,
                               const int4* lrec, int64_t n_lanes, int4* opsem, int4* lsem, int num_sms,
                               cudaStream_t s) {
  const int64_t n = n_ops + n_lanes;
  if (n == 0) return cudaSuccess;
  const int64_t want = (n + kThreads - 1) / kThreads;
  const int64_t cap = (int64_t)num_sms * 8;
  const int grid = (int)(want < cap ? want : cap);
  k_sem_records<<<grid, kThreads, 0, s>>>(xsem, n_instrs, ops, n_ops, lrec, n_lanes, opsem, lsem);
  return launched();
}

}  // namespace syncgb
