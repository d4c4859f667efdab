// Costs of the timing model shared by the two simulation kernels: the wait
// ops an instance pays before issue (Table 1, with Sec. 6.2's reductions when
// enabled) and the static time bound that decides SYNC_PROG_OVERFLOW.
#pragma once

#include "enc.h"

namespace syncgb {

__device__ __forceinline__ unsigned long long sat_add(unsigned long long a, unsigned long long b) {
  const unsigned long long r = a + b;
  return r < a ? ~0ull : r;
}
__device__ __forceinline__ unsigned long long sat_mul(unsigned long long a, unsigned long long b) {
  return __umul64hi(a, b) ? ~0ull : a * b;
}

// Barrier-free wait ops of one datapath instance of the record `rec`
// ({instruction, latency, waited dependencies, first dependency}) with
// `levels` (per-engine waits: loops strictly between the top level and the
// producer's loop, summed over the record's dependencies).  Without the
// reductions: c_wait per dependency (3 count, 5 per-loop, Table 1) plus, per
// engine, c_wait_ops_perengine_level per level (Sec. 6.1's path sum).  With
// CSE, only the waits that do not reuse an earlier identical value pay, a
// reused mask saves min(c_regop, c_wait), and a reused outer sum its levels
// term; with LICM (per-engine) the levels term becomes one c_regop read of
// the cached sum per wait with levels.
template <int MODE, class A>
__device__ __forceinline__ int32_t wait_ops(const A& a, const int4 rec, int32_t levels) {
  const sync_sim_params& q = a.prm;
  const int32_t cw = MODE == SYNC_THR_COUNT ? q.c_wait_ops_count : q.c_wait_ops_perloop;
  if (!(q.licm | q.cse))
    return rec.z * cw + (MODE == SYNC_THR_PERENGINE ? q.c_wait_ops_perengine_level * levels : 0);
  if (rec.z == 0) return 0;
  const int4 c = q.cse ? __ldg(a.cost.xcse + rec.x)
                       : make_int4(rec.z, 0, MODE == SYNC_THR_PERENGINE ? __ldg(a.cost.xlvr + rec.x) : 0, levels);
  int32_t w = c.x * cw - c.y * min(q.c_regop, cw);
  if (MODE == SYNC_THR_PERENGINE) w += q.licm ? q.c_regop * c.z : q.c_wait_ops_perengine_level * c.w;
  return w;
}

// LICM's extra cost at each iteration start of the loop whose (loop, engine)
// row is `row`: one cached-sum update per producer engine (per-engine waits,
// barrier-free only).
template <int MODE, bool BB, class A>
__device__ __forceinline__ int32_t hoist_ops(const A& a, int32_t row) {
  if (BB || MODE != SYNC_THR_PERENGINE || !a.prm.licm) return 0;
  return a.prm.c_wait_ops_perengine_level * __ldg(a.cost.hoist + row);
}

// Static time bound of a program under the given costs (saturating): every
// instance's latency, issue interval and wait ops, and every control cost,
// as if nothing overlapped.
template <int MODE, bool BB>
__device__ __forceinline__ unsigned long long time_bound(const ProgInfo& pi, const sync_sim_params& q,
                                                         int32_t cwait) {
  typedef unsigned long long u64;
  u64 b = sat_add((u64)pi.agg_lat, sat_mul((u64)q.ii, (u64)pi.n_inst));
  if (BB) {
    b = sat_add(b, sat_mul(sat_mul((u64)pi.ne, (u64)pi.n_iter), (u64)q.c_branch));
    b = sat_add(b, sat_mul((u64)(pi.n_stmt + pi.n_iter), (u64)q.c_barrier));
  } else {
    b = sat_add(b, sat_mul((u64)cwait, (u64)pi.n_pairs));
    if (MODE == SYNC_THR_PERENGINE) {
      b = sat_add(b, sat_mul((u64)q.c_wait_ops_perengine_level, (u64)pi.pair_levels));
      if (q.licm) {                     // cached-sum updates and reads
        b = sat_add(b, sat_mul((u64)q.c_wait_ops_perengine_level, (u64)pi.licm_upd));
        b = sat_add(b, sat_mul((u64)q.c_regop, (u64)pi.lv_pairs));
      }
    }
    // control operations of every engine (their own trips): r-hat := 0 at
    // statements and the branch, r++ and r-hat++ at iteration starts, minus
    // the r-hat ops of loops without a trip register when that is elided
    const u64 el = q.trip_register_elision ? 1 : 0;
    const u64 rhat_stmts = (u64)pi.eng_stmt - el * (u64)pi.el_stmt;
    const u64 rhat_iters = (u64)pi.eng_iter - el * (u64)pi.el_iter;
    b = sat_add(b, sat_mul(rhat_stmts, (u64)q.c_regop));
    b = sat_add(b, sat_mul((u64)pi.eng_iter, (u64)q.c_branch + (u64)q.c_regop));
    b = sat_add(b, sat_mul(rhat_iters, (u64)q.c_regop));
    b = sat_add(b, sat_mul((u64)pi.fb_iters, (u64)q.c_barrier));   // barrier-fallback barriers
  }
  return b;
}

}  // namespace syncgb
