// The base-snapshot kernel, select_best and the launchers of every kernel
// (called from the host translation unit).
#include "gmgsim_sim.cuh"

namespace gsim {
namespace {

// ---------------------------------------------------------------------------
// base_create: simulate the base placement once, recording resume points.
// ---------------------------------------------------------------------------
template <bool kReg, bool kKey, bool kTypes, bool kBatch>
__global__ void __launch_bounds__(32) sim_base_kernel(const __grid_constant__ SimParams P) {
  extern __shared__ __align__(16) uint8_t smem[];
  Sim<kReg, kBase, kKey, false, kTypes, kBatch> S(P);
  setup_slot(S, P, 0, 0, smem);
  const DevBase& B = P.base;
  const unsigned lane = lane_id();
  warp_prefetch_l2(P.g.ws, P.g.ws_bytes);
  // keep a copy of the base placement for the candidates
  for (int c = lane * 16; c < B.ld; c += 512)
    *reinterpret_cast<uint4*>(B.row + c) = *reinterpret_cast<const uint4*>(P.place + c);
  for (int c = lane; c < B.nck; c += 32) B.ck_time[c] = kI64Max;
  S.fbuf = B.fb;
  S.row = P.place;
  __syncwarp();
  if (S.row_has_bad_device(P.place)) {
    if (lane == 0) B.status[0] = GMG_SIM_BADDEV;
    return;
  }
  S.reset_common();
  S.ck = 0;
  S.next_ck = 0;
  // checkpoint 0: the initial state, valid for every resume time >= 0
  S.maybe_checkpoint(S.rq.make(0, 0u, 0u));
  S.run();
  if (lane == 0) B.status[0] = S.status;
  if (S.status != GMG_SIM_OK) return;
  int32_t miss = 0;
  for (int r = lane; r < S.g.R; r += 32) {
    const int64_t c = S.creq[r];
    B.res_creq[r] = c;
    miss += c > __ldg(S.g.deadline + r) ? 1 : 0;
  }
  miss = (int32_t)__reduce_add_sync(kFullMask, (unsigned)miss);
  S.dv.write_peak(B.res_peak);
  if (lane == 0) {
    int64_t* rs = B.res_scalars;
    rs[0] = S.makespan;
    rs[1] = S.vflag ? kI64Max : S.score;
    rs[2] = S.vflag;
    rs[3] = S.vop;
    rs[4] = S.vdev;
    rs[5] = S.vt;
    rs[6] = miss;
    rs[7] = S.ck;
  }
}


// ---------------------------------------------------------------------------
// select_best (Algorithm 1, BestRecordedCandidateResult): block argmin of
// (mode ? sla_miss : 0, score, k) over eligible candidates, then a one-block
// final argmin.
// ---------------------------------------------------------------------------
struct Rank {
  int64_t a;  // sla_miss (mode 1) or 0; INT64_MAX = not eligible
  int64_t s;  // score
  int64_t k;
};

__device__ __forceinline__ bool rank_less(const Rank& x, const Rank& y) {
  if (x.a != y.a) return x.a < y.a;
  if (x.s != y.s) return x.s < y.s;
  return x.k < y.k;
}

__device__ Rank block_argmin(Rank r) {
  __shared__ Rank part[32];
  for (int o = 16; o > 0; o >>= 1) {
    Rank t;
    t.a = __shfl_down_sync(kFullMask, r.a, o);
    t.s = __shfl_down_sync(kFullMask, r.s, o);
    t.k = __shfl_down_sync(kFullMask, r.k, o);
    if (rank_less(t, r)) r = t;
  }
  const unsigned w = threadIdx.x >> 5;
  if (lane_id() == 0) part[w] = r;
  __syncthreads();
  if (w == 0) {
    const unsigned nw = blockDim.x >> 5;
    r = lane_id() < nw ? part[lane_id()] : Rank{kI64Max, kI64Max, kI64Max};
    for (int o = 16; o > 0; o >>= 1) {
      Rank t;
      t.a = __shfl_down_sync(kFullMask, r.a, o);
      t.s = __shfl_down_sync(kFullMask, r.s, o);
      t.k = __shfl_down_sync(kFullMask, r.k, o);
      if (rank_less(t, r)) r = t;
    }
  }
  return r;
}

__global__ void __launch_bounds__(256) select_partial_kernel(const int32_t* status, const int32_t* viol,
                                                             const int64_t* score, const int32_t* miss,
                                                             int32_t K, int32_t mode, Rank* part) {
  Rank r{kI64Max, kI64Max, kI64Max};
  for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < K;
       k += (int64_t)gridDim.x * blockDim.x) {
    if (status[k] != GMG_SIM_OK || viol[k] != 0) continue;
    const Rank c{mode ? (int64_t)miss[k] : 0, score[k], k};
    if (rank_less(c, r)) r = c;
  }
  r = block_argmin(r);
  if (threadIdx.x == 0) part[blockIdx.x] = r;
}

__global__ void __launch_bounds__(256) select_final_kernel(const Rank* part, int32_t nparts, int64_t* best) {
  Rank r{kI64Max, kI64Max, kI64Max};
  for (int i = threadIdx.x; i < nparts; i += blockDim.x)
    if (rank_less(part[i], r)) r = part[i];
  r = block_argmin(r);
  if (threadIdx.x == 0) {
    const bool none = r.k == kI64Max;
    best[0] = none ? -1 : r.k;
    best[1] = none ? kI64Max : r.s;
  }
}

}  // namespace

// ---------------------------------------------------------------------------
// Launchers (called from the host translation unit).
// ---------------------------------------------------------------------------
size_t select_rank_bytes() { return sizeof(Rank); }

const void* full_kernel_ptr(bool reg, bool key, bool t32, bool types, bool batch);  // gmgsim_full.cu
const void* inc_kernel_ptr(bool reg, bool key, bool t32, bool types, bool batch);   // gmgsim_inc.cu

template <bool R, bool K, bool B>
const void* base_ptr4(bool types) {
  return types ? (const void*)sim_base_kernel<R, K, true, B> : (const void*)sim_base_kernel<R, K, false, B>;
}
const void* base_kernel_ptr(bool reg, bool key, bool types, bool batch) {
  if (reg) return key ? base_ptr4<true, true, false>(types) : base_ptr4<true, false, false>(types);
  if (!key) return base_ptr4<false, false, false>(types);
  return batch ? base_ptr4<false, true, true>(types) : base_ptr4<false, true, false>(types);
}

cudaError_t set_smem_limits(int smem) {
  for (int r = 0; r < 2; ++r)
    for (int k = 0; k < 2; ++k)
      for (int t = 0; t < 2; ++t)
        for (int y = 0; y < 2; ++y)
          for (int b = 0; b < 2; ++b) {
            const void* fns[] = {full_kernel_ptr(r, k, t, y, b), inc_kernel_ptr(r, k, t, y, b),
                                 base_kernel_ptr(r, k, y, b)};
            for (const void* f : fns) {
              const cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
              if (e != cudaSuccess) return e;
            }
          }
  return cudaSuccess;
}

// A kernel instance's launch through its pointer (the instance is chosen by
// the graph's flags).
static cudaError_t launch_ptr(const void* fn, const SimParams& P, int grid, int block, size_t smem,
                              cudaStream_t st) {
  void* args[] = {const_cast<SimParams*>(&P)};
  return cudaLaunchKernel(fn, dim3(grid), dim3(block), args, smem, st);
}

cudaError_t launch_full(bool reg, const SimParams& P, int grid, int block, size_t smem, cudaStream_t st) {
  return launch_ptr(full_kernel_ptr(reg, P.g.dev_key != 0, P.g.t32 != 0, P.g.ntypes >= 2, P.g.batch != 0), P, grid,
                    block, smem, st);
}

cudaError_t launch_inc(bool reg, const SimParams& P, int grid, int block, size_t smem, cudaStream_t st) {
  return launch_ptr(inc_kernel_ptr(reg, P.g.dev_key != 0, P.g.t32 != 0, P.g.ntypes >= 2, P.g.batch != 0), P, grid,
                    block, smem, st);
}

cudaError_t launch_base(bool reg, const SimParams& P, size_t smem, cudaStream_t st) {
  return launch_ptr(base_kernel_ptr(reg, P.g.dev_key != 0, P.g.ntypes >= 2, P.g.batch != 0), P, 1, 32, smem, st);
}

cudaError_t launch_select(const int32_t* status, const int32_t* viol, const int64_t* score,
                          const int32_t* miss, int32_t K, int32_t mode, void* tmp, int nparts,
                          int64_t* best, cudaStream_t st) {
  Rank* part = reinterpret_cast<Rank*>(tmp);
  select_partial_kernel<<<nparts, 256, 0, st>>>(status, viol, score, miss, K, mode, part);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  select_final_kernel<<<1, 256, 0, st>>>(part, nparts, best);
  return cudaGetLastError();
}

}  // namespace gsim
