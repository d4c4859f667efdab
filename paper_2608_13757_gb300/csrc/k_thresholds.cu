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
// starts, and a trip start per distinct g_S (loaded in parallel): a short
// chain of dependent loads.  A nested producer's count (rare) is evaluated
// once per distinct g_S.
#include <cstdlib>

#include "waitval.cuh"

namespace syncgb {
namespace {

constexpr int kThreads = 256;

// Dependency owning pair q: the largest d with seg[d] <= q, searched inside
// the range the tile table gives for q's tile (empty segments share their
// offset with the next dependency, which then wins).
template <typename I>
__device__ __forceinline__ int find_dep(const ThrArgs& a, I q) {
  const I t = q / kTilePairs;
  int lo = __ldg(a.tile_first + t), hi = __ldg(a.tile_first + t + 1);
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (__ldg(a.seg + mid) <= q) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Values of the chunk's pairs g0 .. g0+3 (entries at or past `total` are
// padding and get 0).  g0 is a multiple of 4, and so is every derived
// array's start, so the chunk's four trip starts (consumer in S) or
// S-ancestors (consumer below S) come in one int4 load; below S, the trip
// start of each distinct S-iteration is loaded once (the ancestors are
// non-decreasing), all in parallel.
template <bool CHECK>
__device__ __forceinline__ int4 chunk_values(const ThrArgs& a, const DepInfo& D, int32_t g0, int mode) {
  const int32_t n = D.total - g0 < kChunk ? D.total - g0 : kChunk;   // >= 1
  const int32_t* ts = a.derived + D.tstart;
  int32_t gs[kChunk], st[kChunk];
  if (D.src < 0) {
    // S runs once: every consumer iteration is in S-iteration 0, trip start 0
#pragma unroll
    for (int i = 0; i < kChunk; ++i) gs[i] = st[i] = 0;
  } else if (D.up == 0) {
    const int4 x = __ldg(reinterpret_cast<const int4*>(a.derived + D.src + g0));
    // consumer directly in S: g_S = g
    gs[0] = g0; gs[1] = g0 + 1; gs[2] = g0 + 2; gs[3] = g0 + 3;
    st[0] = x.x; st[1] = x.y; st[2] = x.z; st[3] = x.w;
  } else {
    const int4 x = __ldg(reinterpret_cast<const int4*>(a.derived + D.src + g0));
    gs[0] = x.x; gs[1] = x.y; gs[2] = x.z; gs[3] = x.w;
    st[0] = __ldg(ts + gs[0]);
    st[3] = n > 3 && gs[3] != gs[0] ? __ldg(ts + gs[3]) : st[0];
    st[1] = n > 1 && gs[1] != gs[0] ? (gs[1] == gs[3] ? st[3] : __ldg(ts + gs[1])) : st[0];
    st[2] = n > 2 && gs[2] != gs[0] ? (gs[2] == gs[3] ? st[3] : __ldg(ts + gs[2])) : st[0];
  }
  int32_t v[kChunk];
  if (D.clen == 0) {
    // producer directly in S: the count through the target is its position
#pragma unroll
    for (int i = 0; i < kChunk; ++i) {
      if (CHECK) {
        const int32_t tS = gs[i] - st[i] + 1 - D.k;      // target's position in its trip
        v[i] = i < n && tS > 0 ? encode(a, D, st[i] + tS, mode) : 0;
      } else {
        v[i] = i < n && gs[i] - st[i] + 1 > D.k ? encode(a, D, gs[i] + 1 - D.k, mode) : 0;
      }
    }
  } else {
    // nested producer: one evaluation per distinct g_S
    int32_t val = eval_at<CHECK>(a, D, gs[0], st[0], mode);
    v[0] = val;
#pragma unroll
    for (int i = 1; i < kChunk; ++i) {
      if (i < n && gs[i] != gs[i - 1]) val = eval_at<CHECK>(a, D, gs[i], st[i], mode);
      v[i] = i < n ? val : 0;
    }
  }
  return make_int4(v[0], v[1], v[2], v[3]);
}

// Prefetch hints (no register is held and nothing waits for them).
__device__ __forceinline__ void prefetch_l1(const void* p) { asm volatile("prefetch.global.L1 [%0];" :: "l"(p)); }
__device__ __forceinline__ void prefetch_l2(const void* p) { asm volatile("prefetch.global.L2 [%0];" :: "l"(p)); }

// I is the chunk-index type: 32-bit while every pair index of the launch
// (plus one grid stride) fits, which saves the 64-bit address arithmetic
// of the loop; 64-bit otherwise.
//
// The chunk's chain of dependent loads is latency-bound; the tile-table
// entry of the thread's next chunk is brought into L1 while this one runs,
// which takes the first link out of the next chain.
template <int MODE, typename I>
__global__ void __launch_bounds__(kThreads, 8) k_thresholds(const ThrArgs a, int32_t* __restrict__ thr) {
  const I stride = (I)gridDim.x * kThreads, n_chunks = (I)a.n_chunks;
  for (I c = (I)blockIdx.x * kThreads + threadIdx.x; c < n_chunks; c += stride) {
    const I q = c * kChunk;
    if (c + stride < n_chunks) prefetch_l1(a.tile_first + (q + stride * kChunk) / kTilePairs);
    const DepInfo D = a.dep[find_dep(a, q)];
    __stcs(reinterpret_cast<int4*>(thr + q), chunk_values<false>(a, D, (int32_t)(q - D.seg_off), MODE));
  }
}

// A warp's chunks with a mismatch: tally them warp-wide (unsafe: below the
// minimum, over-synchronised: above it) and record the first offending pair.
__device__ __forceinline__ void report(const CheckArgs& a, const int4 v, const int4 m, int32_t n, int64_t q,
                                       bool bad) {
  const int32_t got[kChunk] = {v.x, v.y, v.z, v.w}, want[kChunk] = {m.x, m.y, m.z, m.w};
  unsigned u = 0, o = 0;
  unsigned long long first = ~0ull;
  if (bad) {
#pragma unroll
    for (int i = kChunk - 1; i >= 0; --i) {
      if (i < n && got[i] != want[i]) {
        if (got[i] < want[i]) ++u; else ++o;
        first = (unsigned long long)(q + i);
      }
    }
  }
  u = __reduce_add_sync(0xffffffffu, u);
  o = __reduce_add_sync(0xffffffffu, o);
  for (int s = 16; s > 0; s >>= 1) {
    const unsigned long long f = __shfl_xor_sync(0xffffffffu, first, s);
    first = f < first ? f : first;
  }
  if ((threadIdx.x & 31) == 0) {
    if (u) atomicAdd(a.counts + 0, (unsigned long long)u);
    if (o) atomicAdd(a.counts + 1, (unsigned long long)o);
    atomicMin(a.first_bad, first);
  }
}

// Warps step through the chunks together (every lane runs every iteration,
// lanes past the end idle), so a mismatch can be tallied warp-wide where it
// occurs and nothing is carried in registers.  The stored thresholds are
// prefetched into L2 when the chunk starts and read after its minimum is
// known, so no register holds them across the chain of lookups.
template <int MODE, typename I>
__global__ void __launch_bounds__(kThreads, 8) k_check(const CheckArgs a) {
  const I stride = (I)gridDim.x * kThreads, n_chunks = (I)a.t.n_chunks;
  const I end = (n_chunks + 31) & ~I(31);
  for (I cf = (I)blockIdx.x * kThreads + threadIdx.x; cf < end; cf += stride) {
    // 32-chunk groups from the last one down (lanes ascending inside a
    // group): the thresholds written last by the threshold kernel, still
    // in L2 when this kernel follows it, are read first
    const I c = end - 32 - (cf & ~I(31)) + (cf & 31);
    const I q = c * kChunk;
    bool bad = false;
    int4 v = make_int4(0, 0, 0, 0), m = v;
    int32_t n = 0;
    if (c < n_chunks) {
      prefetch_l2(a.thr + q);
      const DepInfo D = a.t.dep[find_dep(a.t, q)];
      const int32_t g0 = (int32_t)(q - D.seg_off);
      m = chunk_values<true>(a.t, D, g0, MODE);
      v = __ldcs(reinterpret_cast<const int4*>(a.thr + q));
      // padding entries are not pairs: the checker reads only the first n
      n = D.total - g0;
      bad = v.x != m.x || (n > 1 && v.y != m.y) || (n > 2 && v.z != m.z) || (n > 3 && v.w != m.w);
    }
    if (__ballot_sync(0xffffffffu, bad)) report(a, v, m, n, q, bad);
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


// 64-bit chunk indices when 32 bits could overflow (or when the
// SYNCGB_WIDE_INDEX environment variable is set to 1, which tests use to
// run the 64-bit kernels on small batches).
bool wide_index(int64_t n_chunks, int grid) {
  const char* f = std::getenv("SYNCGB_WIDE_INDEX");
  if (f && f[0] == '1') return true;
  return (n_chunks + (int64_t)grid * kThreads) * kChunk > (int64_t)INT32_MAX;
}

template <int MODE>
cudaError_t launch_thr_mode(const ThrArgs& a, int32_t* thr, int num_sms, cudaStream_t s) {
  int grid = 0;
  cudaError_t e = grid_for(k_thresholds<MODE, int64_t>, a.n_chunks, num_sms, grid);
  if (e != cudaSuccess) return e;
  if (wide_index(a.n_chunks, grid)) k_thresholds<MODE, int64_t><<<grid, kThreads, 0, s>>>(a, thr);
  else k_thresholds<MODE, int32_t><<<grid, kThreads, 0, s>>>(a, thr);
  return launched();
}

template <int MODE>
cudaError_t launch_check_mode(const CheckArgs& a, int num_sms, cudaStream_t s) {
  int grid = 0;
  cudaError_t e = grid_for(k_check<MODE, int64_t>, a.t.n_chunks, num_sms, grid);
  if (e != cudaSuccess) return e;
  if (wide_index(a.t.n_chunks, grid)) k_check<MODE, int64_t><<<grid, kThreads, 0, s>>>(a);
  else k_check<MODE, int32_t><<<grid, kThreads, 0, s>>>(a);
  return launched();
}

}  // namespace

cudaError_t launch_thresholds(const ThrArgs& a, int32_t* thr, int num_sms, cudaStream_t s) {
  if (a.n_chunks == 0) return cudaSuccess;
  if (a.mode == SYNC_THR_PERLOOP) return launch_thr_mode<SYNC_THR_PERLOOP>(a, thr, num_sms, s);
  if (a.mode == SYNC_THR_PERENGINE) return launch_thr_mode<SYNC_THR_PERENGINE>(a, thr, num_sms, s);
  return launch_thr_mode<SYNC_THR_COUNT>(a, thr, num_sms, s);
}

cudaError_t launch_check(const CheckArgs& a, int num_sms, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(a.counts, 0, 2 * sizeof(unsigned long long), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(a.first_bad, 0xff, sizeof(unsigned long long), s);
  if (e != cudaSuccess || a.t.n_chunks == 0) return e;
  if (a.t.mode == SYNC_THR_PERLOOP) return launch_check_mode<SYNC_THR_PERLOOP>(a, num_sms, s);
  if (a.t.mode == SYNC_THR_PERENGINE) return launch_check_mode<SYNC_THR_PERENGINE>(a, num_sms, s);
  return launch_check_mode<SYNC_THR_COUNT>(a, num_sms, s);
}

}  // namespace syncgb
