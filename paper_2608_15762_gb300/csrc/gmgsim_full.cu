// sim_batch kernels: K full placements, one warp per candidate.
#include "gmgsim_sim.cuh"

namespace gsim {
namespace {

// ---------------------------------------------------------------------------
// sim_batch: K full placements.
// ---------------------------------------------------------------------------
template <bool kReg, bool kKey, bool kT32, bool kTypes, bool kBatch>
__global__ void __launch_bounds__(128, kBatch ? kBatchBlocksPerSM : 7) sim_full_kernel(const __grid_constant__ SimParams P) {
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

// ---------------------------------------------------------------------------
// sim_batch with the GMG staged in shared memory (sim_opts_t.gmg_staging = 1):
// one CTA per SM of up to kStageMaxWarps warps.  Thread 0 copies the compact
// hot records, the releases and both CSR lists into shared memory with bulk
// copies (cp.async.bulk, completion counted on an mbarrier; plain copies of
// this GPU's own memory, no multicast), once per CTA; every warp then reads
// them from there when it starts ops and tests successors.  The wait for the
// copies is bounded: if it runs out, the CTA waits once more (bounded) for
// its copies in flight and marks its candidates GMG_SIM_LOOP.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void bulk_to_shared(void* dst, const void* src, uint32_t bytes, uint32_t bar) {
  const uint64_t gsrc = (uint64_t)__cvta_generic_to_global(src);
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               :: "r"(smem_addr(dst)), "l"(gsrc), "r"(bytes), "r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile("{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
               " selp.u32 %0, 1, 0, p;\n}"
               : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity) {
  for (int it = 0; it < (1 << 22); ++it)
    if (mbar_try_wait(bar, parity)) return true;
  return false;
}

__global__ void __launch_bounds__(32 * kStageMaxWarps, 1) sim_full_staged_kernel(const __grid_constant__ SimParams P) {
  extern __shared__ __align__(16) uint8_t smem[];
  const DevGmg& g = P.g;
  const uint32_t b_hot = 16u * (uint32_t)g.n;
  const uint32_t b_rel = (4u * (uint32_t)g.n + 15u) / 16u * 16u;
  const uint32_t b_list = (4u * (uint32_t)g.n_edges + 15u) / 16u * 16u;
  uint8_t* s_hot = smem + 16;
  uint8_t* s_rel = s_hot + b_hot;
  uint8_t* s_succ = s_rel + b_rel;
  uint8_t* s_pred = s_succ + b_list;
  const uint32_t bar = smem_addr(smem);
  if (threadIdx.x == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" :: "r"(bar) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    const uint32_t total = b_hot + b_rel + 2u * b_list;
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" :: "r"(bar), "r"(total) : "memory");
    if (b_hot) bulk_to_shared(s_hot, g.st_hot, b_hot, bar);
    if (b_rel) bulk_to_shared(s_rel, g.st_rel, b_rel, bar);
    if (b_list) {
      bulk_to_shared(s_succ, g.succ, b_list, bar);
      bulk_to_shared(s_pred, g.pred, b_list, bar);
    }
  }
  __syncthreads();
  bool done = mbar_wait_bounded(bar, 0);
  if (!__syncthreads_and(done)) {
    done = mbar_wait_bounded(bar, 0);  // let the copies in flight land before leaving
    __syncthreads();
  }
  const bool ok = __syncthreads_and(done) != 0;
  const unsigned wib = threadIdx.x >> 5;
  const int64_t nw = blockDim.x >> 5;
  const int64_t slot = (int64_t)blockIdx.x * nw + wib;
  const int64_t nslots = (int64_t)gridDim.x * nw;
  Sim<true, kFull, true, true, false, false, true> S(P);
  setup_slot(S, P, wib, slot, smem + P.stage_bytes);
  S.sh_hot = reinterpret_cast<const uint4*>(s_hot);
  S.sh_rel = reinterpret_cast<const int32_t*>(s_rel);
  S.sh_succ = reinterpret_cast<const uint32_t*>(s_succ);
  S.sh_pred = reinterpret_cast<const uint32_t*>(s_pred);
  for (int64_t k = slot; k < P.K; k += nslots) {
    S.row = P.place + k * P.ld;
    if (!ok) {
      S.write_invalid(k, GMG_SIM_LOOP);
      continue;
    }
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

const void* full_staged_kernel_ptr() { return (const void*)sim_full_staged_kernel; }

cudaError_t launch_full_staged(const SimParams& P, int grid, int block, size_t smem, cudaStream_t st) {
  void* args[] = {const_cast<SimParams*>(&P)};
  return cudaLaunchKernel((const void*)sim_full_staged_kernel, dim3(grid), dim3(block), args, smem, st);
}

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
