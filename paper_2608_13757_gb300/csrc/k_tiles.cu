// Tile tables of the threshold and derive kernels, built by the loader on
// the device from the tables it copied there.
#include "progbuild.cuh"

namespace syncgb {
namespace {

// table[t] = largest i < n with start(i) <= t * tile (start nondecreasing,
// start(0) = 0), for t < n_tiles; table[n_tiles] = n - 1.  One thread per
// item i writes the tiles whose first entry lies in [start(i), start(i+1))
// (the last item's range is open): the ranges partition the entries, so
// every tile is written once, by the last item starting at or before it
// (items with empty ranges write none).
template <class F>
__global__ void k_tile_table(int32_t* table, int64_t n_tiles, int64_t n, int64_t tile, F start) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t i0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i0 == 0) table[n_tiles] = n > 0 ? (int32_t)(n - 1) : 0;
  if (n == 0) {
    for (int64_t t = i0; t < n_tiles; t += stride) table[t] = 0;
    return;
  }
  for (int64_t i = i0; i < n; i += stride) {
    const int64_t s0 = start(i);
    const int64_t t_end = i + 1 < n ? (start(i + 1) + tile - 1) / tile : n_tiles;   // first tile past the range
    for (int64_t t = (s0 + tile - 1) / tile; t < t_end && t < n_tiles; ++t) table[t] = (int32_t)i;
  }
}

struct SegStart {
  const int64_t* seg;
  __device__ int64_t operator()(int64_t i) const { return seg[i]; }
};
struct JobRowStart {
  const DeriveJob* jobs;
  __device__ int64_t operator()(int64_t i) const { return jobs[i].row0; }
};

int grid_for(int64_t n, int threads, int num_sms) {
  const int64_t want = (n + threads - 1) / threads;
  const int64_t cap = (int64_t)num_sms * 16;
  return (int)(want < 1 ? 1 : want < cap ? want : cap);
}

template <class F>
cudaError_t tile_table(int32_t* table, int64_t n_tiles, int64_t n, int64_t tile, F start, int num_sms,
                       cudaStream_t s) {
  k_tile_table<<<grid_for((n > n_tiles ? n : n_tiles) + 1, 256, num_sms), 256, 0, s>>>(table, n_tiles, n, tile, start);
  return launched();
}

}  // namespace

cudaError_t launch_tile_tables(const int64_t* seg, int64_t n_deps, int32_t* tile_first, int64_t n_first_tiles,
                               const DeriveJob* jobs, int64_t n_jobs, int32_t* tile_job, int64_t n_job_tiles,
                               int num_sms, cudaStream_t s) {
  cudaError_t e = tile_table(tile_first, n_first_tiles, n_deps, kTilePairs, SegStart{seg}, num_sms, s);
  if (e == cudaSuccess) e = tile_table(tile_job, n_job_tiles, n_jobs, kJobTileRows, JobRowStart{jobs}, num_sms, s);
  return e;
}

}  // namespace syncgb
