// sim_batch kernels: K full placements, one warp per candidate.
#include "gmgsim_sim.cuh"

namespace gsim {
namespace {

// ---------------------------------------------------------------------------
// sim_batch: K full placements.
// ---------------------------------------------------------------------------
template <bool kReg, bool kKey, bool kT32, bool kTypes, bool kBatch>
__global__ void __launch_bounds__(128, 7) sim_full_kernel(const __grid_constant__ SimParams P) {
  extern __shared__ __align__(16) uint8_t smem[];
  const unsigned wib = threadIdx.x >> 5;
  const int64_t slot = (int64_t)blockIdx.x * (blockDim.x >> 5) + wib;
  const int64_t nslots = (int64_t)gridDim.x * (blockDim.x >> 5);
  Sim<kReg, kFull, kKey, kT32, kTypes, kBatch> S(P);
  setup_slot(S, P, wib, slot, smem);
  for (int64_t k = slot; k < P.K; k += nslots) {
    S.row = P.place + k * P.ld;
    if (S.row_has_bad_device(S.row)) {
      S.write_invalid(k, GMG_SIM_BADDEV);
      continue;
    }
    S.reset_common();
    S.run();
    S.finish(k);
  }
}

}  // namespace

// Instances by (accelerator state in registers, accelerator id in the event
// key, 32-bit times, accelerator types, batched sweep).  32-bit times are only
// chosen with the accelerator id in the key; the batched sweep only with
// accelerator state in shared memory and the id in the key.
template <bool R, bool K, bool T32, bool B>
const void* full_ptr5(bool types) {
  return types ? (const void*)sim_full_kernel<R, K, T32, true, B> : (const void*)sim_full_kernel<R, K, T32, false, B>;
}
const void* full_kernel_ptr(bool reg, bool key, bool t32, bool types, bool batch) {
  if (reg) {
    if (!key) return full_ptr5<true, false, false, false>(types);
    return t32 ? full_ptr5<true, true, true, false>(types) : full_ptr5<true, true, false, false>(types);
  }
  if (!key) return full_ptr5<false, false, false, false>(types);
  if (batch) return t32 ? full_ptr5<false, true, true, true>(types) : full_ptr5<false, true, false, true>(types);
  return t32 ? full_ptr5<false, true, true, false>(types) : full_ptr5<false, true, false, false>(types);
}

}  // namespace gsim
