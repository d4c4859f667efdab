// Load-time expansion of the trip prefix sums into parent-iteration indices.
//
// For every loop l and every global iteration g of l, pidx_l[g] is the
// parent's global iteration j with rowptr_l[j] <= g < rowptr_l[j+1] (the CSR
// row of g).  One thread per output entry; the loop is found inside the range
// the host's tile table gives, the row by binary search over rowptr_l.
#include "enc.h"

namespace syncgb {
namespace {

constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads)
k_expand(const LoopInfo* __restrict__ loop, const int32_t* __restrict__ tile_loop,
         const int32_t* __restrict__ rowptr, int32_t* __restrict__ pidx, int64_t n_iters) {
  const int64_t stride = (int64_t)gridDim.x * kThreads;
  for (int64_t q = (int64_t)blockIdx.x * kThreads + threadIdx.x; q < n_iters; q += stride) {
    const int64_t t = q / kTilePairs;
    int lo = tile_loop[t], hi = tile_loop[t + 1];
    while (lo < hi) {                 // largest l with pidx_off[l] <= q
      const int mid = (lo + hi + 1) >> 1;
      if (loop[mid].pidx_off <= q) lo = mid; else hi = mid - 1;
    }
    const LoopInfo L = loop[lo];
    const int32_t g = (int32_t)(q - L.pidx_off);
    const int32_t* rp = rowptr + L.rowptr_off;
    int a = 0, b = L.n_parent - 1;    // largest j with rp[j] <= g
    while (a < b) {
      const int mid = (a + b + 1) >> 1;
      if (rp[mid] <= g) a = mid; else b = mid - 1;
    }
    pidx[q] = a;
  }
}

}  // namespace

cudaError_t launch_expand(const LoopInfo* loop, const int32_t* tile_loop, const int32_t* rowptr,
                          int32_t* pidx, int64_t n_iters, int num_sms, cudaStream_t s) {
  if (n_iters == 0) return cudaSuccess;
  const int64_t want = (n_iters + kThreads - 1) / kThreads;
  const int64_t cap = (int64_t)num_sms * 8;
  const int grid = (int)(want < cap ? want : cap);
  k_expand<<<grid, kThreads, 0, s>>>(loop, tile_loop, rowptr, pidx, n_iters);
  return cudaGetLastError();
}

}  // namespace syncgb
