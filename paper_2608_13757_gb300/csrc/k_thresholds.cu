// Threshold kernel and minimality checker over the flattened pair space.
//
// A pair is (dependency d, consumer instance g), g the global iteration index
// of the consumer's loop.  Pairs are laid out dependency-major with every
// segment padded to a multiple of 4, so each thread owns one int4 chunk that
// never straddles two dependencies; consecutive threads own consecutive
// chunks, so a warp's store or load is 512 contiguous bytes.  Both kernels
// are HBM-streaming: 4 bytes per pair written (thresholds) or read
// (checker), plus the derived per-iteration arrays, which consecutive pairs
// of one dependency share through L1/L2.
//
// Both results depend on g only through g_S, the enclosing iteration of the
// dependency's common loop S, and the start of g_S's trip of S (Eq. 1, and
// Sec. 5.1's registers r_S and r-hat_S).  Both come from arrays derived at
// load time (S-ancestor per consumer iteration, trip start per S-iteration),
// so a chunk needs the dependency record, one int4 of ancestors or trip
// starts, and a trip start per distinct g_S: a short chain of dependent
// loads.  A chunk's four consumer iterations usually share g_S, evaluated
// once.
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

// Iterations of P that start inside the first x iterations of S (x may equal
// total(S)): compose the trip prefix sums from S's child down to P.
__device__ __forceinline__ int32_t count_down(const ThrArgs& a, const DepInfo& D, int32_t x) {
  for (int i = 0; i < D.clen; ++i) x = __ldg(a.rowptr + __ldg(a.path + D.path + D.up + 2 + i) + x);
  return x;
}

__device__ __forceinline__ int32_t encode(const ThrArgs& a, const DepInfo& D, int32_t c, int mode) {
  if (c == 0) return 0;
  // Eq. (5): N*c - (N-K) for the per-(loop, engine) semaphore
  if (mode == SYNC_THR_PERLOOP) return D.N * c - (D.N - D.K);
  // Sec. 6.1: the c-th producer instance's position in its engine's stream
  if (mode == SYNC_THR_PERENGINE) return __ldg(a.ord + D.ordp + (c - 1));
  return c;
}

// The paper's register form (Sec. 5.1-5.3): r_S = gs + 1 and r-hat_S = gs -
// start + 1 are the monotone and trip registers of S at the consumer's
// issue; mask = isGT(r-hat_S, k) (Eq. 2); expr = r_S - k when the producer
// sits in S, otherwise r_P, the producer loop's monotone register, which
// counts P's iterations through the current S-iteration (forward) or through
// the previous one (backward, consumer ahead of P in S's body).
__device__ __forceinline__ int32_t wait_value(const ThrArgs& a, const DepInfo& D, int32_t gs,
                                              int32_t start, int mode) {
  if (gs - start + 1 <= D.k) return 0;
  int32_t expr;
  if (D.kase == CASE_PS) expr = gs + 1 - D.k;
  else expr = count_down(a, D, D.kase == CASE_NEST_FWD ? gs + 1 : gs);
  return encode(a, D, expr, mode);
}

// Eq. (1) directly, without the case split: the consumer's 1-based position
// v_S in its trip of S, target t_S = v_S - k (outer components equal the
// consumer's, all >= 1), no wait on underflow, else the producer instances
// in every S-iteration up to and including the target (lexicographic order
// of iteration vectors = global iteration order of S).
__device__ __forceinline__ int32_t minimum(const ThrArgs& a, const DepInfo& D, int32_t gs,
                                           int32_t start, int mode) {
  const int32_t tS = gs - start + 1 - D.k;
  if (tS <= 0) return 0;
  const int32_t gt = start + tS - 1;
  return encode(a, D, count_down(a, D, gt + 1), mode);
}

template <bool CHECK>
__device__ __forceinline__ int32_t eval_at(const ThrArgs& a, const DepInfo& D, int32_t gs, int32_t start,
                                           int mode) {
  return CHECK ? minimum(a, D, gs, start, mode) : wait_value(a, D, gs, start, mode);
}

// Values of the chunk's pairs g0 .. g0+3 (entries at or past `total` are
// padding and get 0).  g0 is a multiple of 4, and so is every derived
// array's start, so the chunk's four trip starts (consumer in S) or
// S-ancestors (consumer below S) come in one int4 load.
template <bool CHECK>
__device__ __forceinline__ int4 chunk_values(const ThrArgs& a, const DepInfo& D, int32_t g0, int mode) {
  const int32_t n = D.total - g0 < kChunk ? D.total - g0 : kChunk;   // >= 1
  int32_t v[kChunk] = {0, 0, 0, 0};
  if (D.up == 0) {
    // consumer directly in S: g_S = g
    const int4 ts = __ldg(reinterpret_cast<const int4*>(a.derived + D.tstart + g0));
    const int32_t st[kChunk] = {ts.x, ts.y, ts.z, ts.w};
#pragma unroll
    for (int i = 0; i < kChunk; ++i)
      if (i < n) v[i] = eval_at<CHECK>(a, D, g0 + i, st[i], mode);
  } else {
    // consumer nested below S: one value per distinct g_S (non-decreasing)
    const int4 an = __ldg(reinterpret_cast<const int4*>(a.derived + D.anc + g0));
    const int32_t gs[kChunk] = {an.x, an.y, an.z, an.w};
    int32_t cur = gs[0];
    int32_t val = eval_at<CHECK>(a, D, cur, __ldg(a.derived + D.tstart + cur), mode);
    v[0] = val;
#pragma unroll
    for (int i = 1; i < kChunk; ++i) {
      if (i < n) {
        if (gs[i] != cur) {
          cur = gs[i];
          val = eval_at<CHECK>(a, D, cur, __ldg(a.derived + D.tstart + cur), mode);
        }
        v[i] = val;
      }
    }
  }
  return make_int4(v[0], v[1], v[2], v[3]);
}

template <int MODE>
__global__ void __launch_bounds__(kThreads, 8) k_thresholds(const ThrArgs a, int32_t* __restrict__ thr) {
  const int64_t stride = (int64_t)gridDim.x * kThreads;
  for (int64_t c = (int64_t)blockIdx.x * kThreads + threadIdx.x; c < a.n_chunks; c += stride) {
    const int64_t q = c * kChunk;
    const DepInfo D = a.dep[find_dep(a, q)];
    __stcs(reinterpret_cast<int4*>(thr + q), chunk_values<false>(a, D, (int32_t)(q - D.seg_off), MODE));
  }
}

__device__ __forceinline__ void tally(int32_t got, int32_t want, int64_t idx, uint32_t& unsafe,
                                      uint32_t& over, unsigned long long& first) {
  if (got == want) return;
  if (got < want) ++unsafe; else ++over;
  if ((unsigned long long)idx < first) first = (unsigned long long)idx;
}

template <int MODE>
__global__ void __launch_bounds__(kThreads, 6) k_check(const CheckArgs a) {
  // a thread's counts fit 32 bits (it sees at most n_chunks / threads chunks)
  uint32_t unsafe = 0, over = 0;
  unsigned long long first = ~0ull;
  const int64_t stride = (int64_t)gridDim.x * kThreads;
  for (int64_t c = (int64_t)blockIdx.x * kThreads + threadIdx.x; c < a.t.n_chunks; c += stride) {
    const int64_t q = c * kChunk;
    const int4 v = __ldcs(reinterpret_cast<const int4*>(a.thr + q));
    const DepInfo D = a.t.dep[find_dep(a.t, q)];
    const int32_t g0 = (int32_t)(q - D.seg_off);
    const int4 m = chunk_values<true>(a.t, D, g0, MODE);
    // padding entries are not pairs: the checker reads only the first n
    const int32_t n = D.total - g0;
    const bool bad = v.x != m.x || (n > 1 && v.y != m.y) || (n > 2 && v.z != m.z) || (n > 3 && v.w != m.w);
    if (bad) {
      tally(v.x, m.x, q + 0, unsafe, over, first);
      if (n > 1) tally(v.y, m.y, q + 1, unsafe, over, first);
      if (n > 2) tally(v.z, m.z, q + 2, unsafe, over, first);
      if (n > 3) tally(v.w, m.w, q + 3, unsafe, over, first);
    }
  }
  unsigned long long u = unsafe, o = over;
  for (int s = 16; s > 0; s >>= 1) {
    u += __shfl_xor_sync(0xffffffffu, u, s);
    o += __shfl_xor_sync(0xffffffffu, o, s);
    const unsigned long long f = __shfl_xor_sync(0xffffffffu, first, s);
    first = f < first ? f : first;
  }
  if ((threadIdx.x & 31) == 0) {
    if (u) atomicAdd(a.counts + 0, u);
    if (o) atomicAdd(a.counts + 1, o);
    if (first != ~0ull) atomicMin(a.first_bad, first);
  }
}

// Resident CTAs of `kern` on every SM, capped by the work; grid-stride
// beyond that.
template <class K>
cudaError_t grid_for(K kern, int64_t n_chunks, int num_sms, int& grid) {
  int per_sm = 0;
  const cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, 0);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) per_sm = 1;
  const int64_t want = (n_chunks + kThreads - 1) / kThreads;
  const int64_t cap = (int64_t)num_sms * per_sm;
  grid = (int)(want < cap ? (want > 0 ? want : 1) : cap);
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_thresholds(const ThrArgs& a, int32_t* thr, int num_sms, cudaStream_t s) {
  if (a.n_chunks == 0) return cudaSuccess;
  auto run = [&](auto kern) -> cudaError_t {
    int grid = 0;
    const cudaError_t e = grid_for(kern, a.n_chunks, num_sms, grid);
    if (e != cudaSuccess) return e;
    kern<<<grid, kThreads, 0, s>>>(a, thr);
    return cudaGetLastError();
  };
  if (a.mode == SYNC_THR_PERLOOP) return run(k_thresholds<SYNC_THR_PERLOOP>);
  if (a.mode == SYNC_THR_PERENGINE) return run(k_thresholds<SYNC_THR_PERENGINE>);
  return run(k_thresholds<SYNC_THR_COUNT>);
}

cudaError_t launch_check(const CheckArgs& a, int num_sms, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(a.counts, 0, 2 * sizeof(unsigned long long), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(a.first_bad, 0xff, sizeof(unsigned long long), s);
  if (e != cudaSuccess || a.t.n_chunks == 0) return e;
  auto run = [&](auto kern) -> cudaError_t {
    int grid = 0;
    const cudaError_t e2 = grid_for(kern, a.t.n_chunks, num_sms, grid);
    if (e2 != cudaSuccess) return e2;
    kern<<<grid, kThreads, 0, s>>>(a);
    return cudaGetLastError();
  };
  if (a.t.mode == SYNC_THR_PERLOOP) return run(k_check<SYNC_THR_PERLOOP>);
  if (a.t.mode == SYNC_THR_PERENGINE) return run(k_check<SYNC_THR_PERENGINE>);
  return run(k_check<SYNC_THR_COUNT>);
}

}  // namespace syncgb
