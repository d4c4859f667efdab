// Wait values of one (dependency, consumer instance) pair, shared by the
// threshold and check kernels and the fused simulators.  The consumer's
// state enters as g_S, its enclosing iteration of the dependency's innermost
// common loop S (global index), and the start of g_S's trip of S; A is any
// argument block with the trip prefix sums (rowptr), the path pool (path)
// and the per-engine ordinal pool (ord).
#pragma once

#include "enc.h"

namespace syncgb {

// Iterations of P that start inside the first x iterations of S (x may equal
// total(S)): compose the trip prefix sums from S's child down to P.
template <class A>
__device__ __forceinline__ int32_t count_down(const A& a, const DepInfo& D, int32_t x) {
  for (int i = 0; i < D.clen; ++i) x = __ldg(a.rowptr + __ldg(a.path + D.path + D.up + i) + x);
  return x;
}

template <class A>
__device__ __forceinline__ int32_t encode(const A& a, const DepInfo& D, int32_t c, int mode) {
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
template <class A>
__device__ __forceinline__ int32_t wait_value(const A& a, const DepInfo& D, int32_t gs,
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
template <class A>
__device__ __forceinline__ int32_t minimum(const A& a, const DepInfo& D, int32_t gs,
                                           int32_t start, int mode) {
  const int32_t tS = gs - start + 1 - D.k;
  if (tS <= 0) return 0;
  const int32_t gt = start + tS - 1;
  return encode(a, D, count_down(a, D, gt + 1), mode);
}

template <bool CHECK, class A>
__device__ __forceinline__ int32_t eval_at(const A& a, const DepInfo& D, int32_t gs, int32_t start,
                                           int mode) {
  return CHECK ? minimum(a, D, gs, start, mode) : wait_value(a, D, gs, start, mode);
}

}  // namespace syncgb
