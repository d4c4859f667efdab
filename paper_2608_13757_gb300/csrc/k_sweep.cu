// Schedule simulator, program-order sweep: the launchers of the sweep kernel
// (its device code, shared with the piece-parallel launches, is sweep.cuh).
#include "sweep.cuh"

namespace syncgb {
namespace {

template <int MODE, bool BB>
cudaError_t launch3(const SweepArgs& a, size_t smem, int num_sms, cudaStream_t s) {
  auto run = [&](auto kern) -> cudaError_t {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kWarps * 32, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    const long long want = ((long long)a.n_programs + kWarps - 1) / kWarps;
    const long long cap = (long long)num_sms * per_sm;
    const int grid = (int)(want < cap ? want : cap);
    e = cudaMemsetAsync(a.next_slot, 0, sizeof(int32_t), s);
    if (e == cudaSuccess) e = cudaMemsetAsync(a.fallback, 0, sizeof(int32_t), s);
    if (e != cudaSuccess) return e;
    kern<<<grid, kWarps * 32, smem, s>>>(a);
    return launched();
  };
  if (a.dep) return a.issue ? run(k_sweep<MODE, BB, true, true>) : run(k_sweep<MODE, BB, false, true>);
  return a.issue ? run(k_sweep<MODE, BB, true, false>) : run(k_sweep<MODE, BB, false, false>);
}

}  // namespace

size_t sweep_smem_bytes(int sem_cap, int frame_depth, int ring) {
  return kWarps * warp_bytes(sem_cap, frame_depth, ring);
}

int sweep_ring_for(int sem_cap, int frame_depth, size_t limit) {
  for (int r = kRingMax; r >= 1; r >>= 1)
    if (sweep_smem_bytes(sem_cap, frame_depth, r) <= limit) return r;
  return 0;
}

cudaError_t launch_sweep(const SweepArgs& a, bool barrier, int num_sms, cudaStream_t s) {
  if (a.n_programs == 0) return cudaSuccess;
  const size_t smem = sweep_smem_bytes(a.sem_cap, a.frame_depth, a.ring);
  if (a.mode == SYNC_THR_PERLOOP)
    return barrier ? launch3<SYNC_THR_PERLOOP, true>(a, smem, num_sms, s)
                   : launch3<SYNC_THR_PERLOOP, false>(a, smem, num_sms, s);
  if (a.mode == SYNC_THR_PERENGINE)
    return barrier ? launch3<SYNC_THR_PERENGINE, true>(a, smem, num_sms, s)
                   : launch3<SYNC_THR_PERENGINE, false>(a, smem, num_sms, s);
  return barrier ? launch3<SYNC_THR_COUNT, true>(a, smem, num_sms, s)
                 : launch3<SYNC_THR_COUNT, false>(a, smem, num_sms, s);
}

}  // namespace syncgb
