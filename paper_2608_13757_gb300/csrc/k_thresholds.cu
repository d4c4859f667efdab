// Threshold kernel and minimality checker over the flattened pair space.
//
// A pair is (dependency d, consumer instance g), g the global iteration index
// of the consumer's loop.  Pairs are laid out dependency-major with every
// segment padded to a multiple of 4, so each thread owns one int4 chunk that
// never straddles two dependencies.  Both kernels are HBM-streaming: 4 bytes
// per pair written (thresholds) or read (checker), plus the loop-structure
// reads, which consecutive pairs of one dependency share through L1/L2.
#include "enc.h"

namespace syncgb {
namespace {

constexpr int kThreads = 256;

// Dependency owning pair q: the largest d with seg[d] <= q, searched inside
// the range the tile table gives for q's tile (empty segments share their
// offset with the next dependency, which then wins).
__device__ __forceinline__ int find_dep(const ThrArgs& a, int64_t q) {
  const int64_t t = q / kTilePairs;
  int lo = __ldg(a.tile_first + t), hi = __ldg(a.tile_first + t + 1);
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (__ldg(a.seg + mid) <= q) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Global iteration of S that encloses the consumer's global iteration g:
// follow the expanded parent indices up `up` levels.
__device__ __forceinline__ int32_t up_to_S(const ThrArgs& a, const DepInfo& D, int32_t g) {
  for (int i = 0; i < D.up; ++i) g = __ldg(a.pidx + __ldg(a.path + D.path + i) + g);
  return g;
}

// Global index of the first iteration of S in the trip that holds gs.
__device__ __forceinline__ int32_t trip_start(const ThrArgs& a, const DepInfo& D, int32_t gs) {
  const int64_t pidx_S = __ldg(a.path + D.path + D.up);
  const int64_t rowptr_S = __ldg(a.path + D.path + D.up + 1);
  return __ldg(a.rowptr + rowptr_S + __ldg(a.pidx + pidx_S + gs));
}

// Iterations of P that start inside the first x iterations of S (x may equal
// total(S)): compose the trip prefix sums from S's child down to P.
__device__ __forceinline__ int32_t count_down(const ThrArgs& a, const DepInfo& D, int32_t x) {
  for (int i = 0; i < D.clen; ++i) x = __ldg(a.rowptr + __ldg(a.path + D.path + D.up + 2 + i) + x);
  return x;
}

__device__ __forceinline__ int32_t encode(const DepInfo& D, int32_t c, int mode) {
  // Eq. (5): N*c - (N-K) for the per-(loop, engine) semaphore; 0 stays 0.
  return (mode == SYNC_THR_PERLOOP && c != 0) ? D.N * c - (D.N - D.K) : c;
}

// The paper's register form (Sec. 5.1-5.3): r_S = gs + 1 and r-hat_S = gs -
// trip_start + 1 are the monotone and trip registers of S at the consumer's
// issue; mask = isGT(r-hat_S, k) (Eq. 2); expr = r_S - k when the producer
// sits in S, otherwise r_P, the producer loop's monotone register, which
// counts P's iterations through the current S-iteration (forward) or through
// the previous one (backward, consumer ahead of P in S's body).
__device__ __forceinline__ int32_t wait_value(const ThrArgs& a, const DepInfo& D, int32_t g,
                                              int mode) {
  const int32_t gs = up_to_S(a, D, g);
  const int32_t rhat = gs - trip_start(a, D, gs) + 1;
  if (rhat <= D.k) return 0;
  int32_t expr;
  if (D.kase == CASE_PS) expr = gs + 1 - D.k;
  else expr = count_down(a, D, D.kase == CASE_NEST_FWD ? gs + 1 : gs);
  return encode(D, expr, mode);
}

// Eq. (1) directly, without the case split: the consumer's 1-based position
// v_S in its trip of S, target t_S = v_S - k (outer components equal the
// consumer's, all >= 1), no wait on underflow, else the producer instances
// in every S-iteration up to and including the target (lexicographic order
// of iteration vectors = global iteration order of S).
__device__ __forceinline__ int32_t minimum(const ThrArgs& a, const DepInfo& D, int32_t g,
                                           int mode) {
  const int32_t gs = up_to_S(a, D, g);
  const int32_t start = trip_start(a, D, gs);
  const int32_t tS = gs - start + 1 - D.k;
  if (tS <= 0) return 0;
  const int32_t gt = start + tS - 1;
  return encode(D, count_down(a, D, gt + 1), mode);
}

template <int MODE>
__global__ void __launch_bounds__(kThreads) k_thresholds(const ThrArgs a, int32_t* __restrict__ thr) {
  const int64_t stride = (int64_t)gridDim.x * kThreads;
  for (int64_t c = (int64_t)blockIdx.x * kThreads + threadIdx.x; c < a.n_chunks; c += stride) {
    const int64_t q = c * kChunk;
    const DepInfo D = a.dep[find_dep(a, q)];
    const int32_t g0 = (int32_t)(q - D.seg_off);
    int4 v;
    v.x = g0 + 0 < D.total ? wait_value(a, D, g0 + 0, MODE) : 0;
    v.y = g0 + 1 < D.total ? wait_value(a, D, g0 + 1, MODE) : 0;
    v.z = g0 + 2 < D.total ? wait_value(a, D, g0 + 2, MODE) : 0;
    v.w = g0 + 3 < D.total ? wait_value(a, D, g0 + 3, MODE) : 0;
    __stcs(reinterpret_cast<int4*>(thr + q), v);
  }
}

__device__ __forceinline__ void tally(int32_t got, int32_t want, int64_t idx,
                                      unsigned long long& unsafe, unsigned long long& over,
                                      unsigned long long& first) {
  if (got == want) return;
  if (got < want) ++unsafe; else ++over;
  if ((unsigned long long)idx < first) first = (unsigned long long)idx;
}

template <int MODE>
__global__ void __launch_bounds__(kThreads) k_check(const CheckArgs a) {
  unsigned long long unsafe = 0, over = 0, first = ~0ull;
  const int64_t stride = (int64_t)gridDim.x * kThreads;
  for (int64_t c = (int64_t)blockIdx.x * kThreads + threadIdx.x; c < a.t.n_chunks; c += stride) {
    const int64_t q = c * kChunk;
    const DepInfo D = a.t.dep[find_dep(a.t, q)];
    const int32_t g0 = (int32_t)(q - D.seg_off);
    const int4 v = __ldcs(reinterpret_cast<const int4*>(a.thr + q));
    if (g0 + 0 < D.total) tally(v.x, minimum(a.t, D, g0 + 0, MODE), q + 0, unsafe, over, first);
    if (g0 + 1 < D.total) tally(v.y, minimum(a.t, D, g0 + 1, MODE), q + 1, unsafe, over, first);
    if (g0 + 2 < D.total) tally(v.z, minimum(a.t, D, g0 + 2, MODE), q + 2, unsafe, over, first);
    if (g0 + 3 < D.total) tally(v.w, minimum(a.t, D, g0 + 3, MODE), q + 3, unsafe, over, first);
  }
  for (int o = 16; o > 0; o >>= 1) {
    unsafe += __shfl_xor_sync(0xffffffffu, unsafe, o);
    over += __shfl_xor_sync(0xffffffffu, over, o);
    const unsigned long long f = __shfl_xor_sync(0xffffffffu, first, o);
    first = f < first ? f : first;
  }
  if ((threadIdx.x & 31) == 0) {
    if (unsafe) atomicAdd(a.counts + 0, unsafe);
    if (over) atomicAdd(a.counts + 1, over);
    if (first != ~0ull) atomicMin(a.first_bad, first);
  }
}

int grid_for(int64_t n_chunks, int num_sms) {
  // 8 resident 256-thread CTAs per SM; grid-stride beyond that.
  const int64_t want = (n_chunks + kThreads - 1) / kThreads;
  const int64_t cap = (int64_t)num_sms * 8;
  return (int)(want < cap ? (want > 0 ? want : 1) : cap);
}

}  // namespace

cudaError_t launch_thresholds(const ThrArgs& a, int32_t* thr, int num_sms, cudaStream_t s) {
  if (a.n_chunks == 0) return cudaSuccess;
  const int grid = grid_for(a.n_chunks, num_sms);
  if (a.mode == SYNC_THR_PERLOOP) k_thresholds<SYNC_THR_PERLOOP><<<grid, kThreads, 0, s>>>(a, thr);
  else k_thresholds<SYNC_THR_COUNT><<<grid, kThreads, 0, s>>>(a, thr);
  return cudaGetLastError();
}

cudaError_t launch_check(const CheckArgs& a, int num_sms, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(a.counts, 0, 2 * sizeof(unsigned long long), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(a.first_bad, 0xff, sizeof(unsigned long long), s);
  if (e != cudaSuccess || a.t.n_chunks == 0) return e;
  const int grid = grid_for(a.t.n_chunks, num_sms);
  if (a.t.mode == SYNC_THR_PERLOOP) k_check<SYNC_THR_PERLOOP><<<grid, kThreads, 0, s>>>(a);
  else k_check<SYNC_THR_COUNT><<<grid, kThreads, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace syncgb
