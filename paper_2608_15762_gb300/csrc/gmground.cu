// One scheduling round of Algorithm 1 (Sec. 3.4) on the GPU: frontiers and
// the budget check, the highest-priority unscheduled-frontier op, batch
// collection, candidate rows from pre-defined partitions, and the write-back.
// The C ABI is declared in include/gmground.h.
//
// round_select: a per-op scan (one thread per op) decides frontier
// membership from the op's predecessor / successor states and reduces the
// counts and the (priority, id) argmin per block; one block combines the
// blocks; one warp collects the batch -- a binary min-heap of op ids held by
// lane 0, successor checks spread over the lanes.  Ops already taken or
// waiting carry the round's epoch in a per-op mark array, so nothing is
// cleared between rounds.

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/gmground.h"
#include "gmg_access.h"

namespace ground {
namespace {

using gsim::DevGmg;
using gsim::kIdMask;

constexpr int kScanThreads = 256;
constexpr int64_t kI64Max = 0x7fffffffffffffffll;

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

struct Part {
  int64_t prio, id, n_fu, n_issued, n_fs;
};

struct Layout {
  size_t mark, heap, part, total;
};

Layout layout(int32_t n) {
  Layout L;
  size_t o = 0;
  const int blocks = (n + kScanThreads - 1) / kScanThreads;
  L.mark = o;
  o = align256(o + 4 * (size_t)n + 4);
  L.heap = o;
  o = align256(o + 4 * (size_t)n + 4);
  L.part = o;
  o = align256(o + sizeof(Part) * (size_t)(blocks > 0 ? blocks : 1));
  L.total = o;
  return L;
}

// (succ_off, nsucc, pred_off, npred) from the op record's [release, preds]
// and [xq, succs] pieces.
__device__ __forceinline__ uint4 op_lists(const DevGmg& g, uint32_t i) {
  const uint4 rp = __ldg(reinterpret_cast<const uint4*>(g.ops + i) + 1);
  const uint4 xs = __ldg(reinterpret_cast<const uint4*>(g.ops + i) + 2);
  return make_uint4(xs.z, xs.w, rp.z, rp.w);
}

__device__ __forceinline__ bool key_less(int64_t pa, int64_t ia, int64_t pb, int64_t ib) {
  return pa < pb || (pa == pb && ia < ib);
}

__global__ void __launch_bounds__(kScanThreads) round_scan_kernel(DevGmg g, const uint8_t* __restrict__ state,
                                                                  const int64_t* __restrict__ prio,
                                                                  Part* __restrict__ part) {
  __shared__ int64_t sp[kScanThreads], si[kScanThreads];
  const int t = threadIdx.x;
  const int64_t i = (int64_t)blockIdx.x * kScanThreads + t;
  bool fu = false, fs = false, issued = false;
  if (i < g.n) {
    const uint8_t st = state[i];
    const uint4 ls = op_lists(g, (uint32_t)i);
    issued = st == 1;
    if (st == 0) {
      fu = true;
      for (uint32_t k = 0; k < ls.w && fu; ++k) fu = state[__ldg(g.pred + ls.z + k) & kIdMask] != 0;
    } else {
      for (uint32_t k = 0; k < ls.y && !fs; ++k) fs = state[__ldg(g.succ + ls.x + k)] == 0;
    }
  }
  sp[t] = fu ? prio[i] : kI64Max;
  si[t] = fu ? i : kI64Max;
  const int n_fu = __syncthreads_count(fu);
  const int n_is = __syncthreads_count(issued);
  const int n_fs = __syncthreads_count(fs);
  for (int o = kScanThreads / 2; o > 0; o >>= 1) {
    if (t < o && key_less(sp[t + o], si[t + o], sp[t], si[t])) {
      sp[t] = sp[t + o];
      si[t] = si[t + o];
    }
    __syncthreads();
  }
  if (t == 0) part[blockIdx.x] = Part{sp[0], si[0], n_fu, n_is, n_fs};
}

__global__ void __launch_bounds__(256) round_reduce_kernel(const Part* __restrict__ part, int32_t nparts,
                                                           int64_t* __restrict__ info) {
  __shared__ int64_t sp[256], si[256], c0[256], c1[256], c2[256];
  const int t = threadIdx.x;
  int64_t p = kI64Max, id = kI64Max, a = 0, b = 0, c = 0;
  for (int32_t k = t; k < nparts; k += 256) {  // fixed order per thread
    const Part q = part[k];
    if (key_less(q.prio, q.id, p, id)) {
      p = q.prio;
      id = q.id;
    }
    a += q.n_fu;
    b += q.n_issued;
    c += q.n_fs;
  }
  sp[t] = p, si[t] = id, c0[t] = a, c1[t] = b, c2[t] = c;
  __syncthreads();
  for (int o = 128; o > 0; o >>= 1) {
    if (t < o) {
      if (key_less(sp[t + o], si[t + o], sp[t], si[t])) {
        sp[t] = sp[t + o];
        si[t] = si[t + o];
      }
      c0[t] += c0[t + o];
      c1[t] += c1[t + o];
      c2[t] += c2[t + o];
    }
    __syncthreads();
  }
  if (t == 0) {
    info[0] = 0;
    info[1] = c0[0] > 0 ? si[0] : -1;
    info[2] = c0[0];
    info[3] = c1[0];
    info[4] = c2[0];
    info[5] = 0;
    info[6] = 0;
    info[7] = 0;
  }
}

// Lane 0 owns the heap (op ids, min at the root).
__device__ void heap_push(int32_t* h, int32_t& n, int32_t v) {
  int32_t pos = n++;
  while (pos > 0) {
    const int32_t par = (pos - 1) >> 1;
    if (h[par] <= v) break;
    h[pos] = h[par];
    pos = par;
  }
  h[pos] = v;
}

__device__ int32_t heap_pop(int32_t* h, int32_t& n) {
  const int32_t top = h[0];
  const int32_t v = h[--n];
  int32_t pos = 0;
  while (true) {
    int32_t c = 2 * pos + 1;
    if (c >= n) break;
    if (c + 1 < n && h[c + 1] < h[c]) ++c;
    if (h[c] >= v) break;
    h[pos] = h[c];
    pos = c;
  }
  if (n > 0) h[pos] = v;
  return top;
}

__global__ void __launch_bounds__(32) round_collect_kernel(DevGmg g, const uint8_t* __restrict__ state,
                                                           int32_t budget, int32_t max_batch, uint32_t epoch,
                                                           uint32_t* __restrict__ mark, int32_t* __restrict__ heap,
                                                           int32_t* __restrict__ batch, int64_t* __restrict__ info) {
  const unsigned lane = threadIdx.x;
  const int64_t issued = info[3];
  if (issued >= budget || info[2] == 0) {
    if (lane == 0) {
      info[0] = 0;
      info[5] = issued >= budget ? GMG_ROUND_BUDGET : GMG_ROUND_EMPTY;
    }
    return;
  }
  const int64_t cap = min((int64_t)max_batch, (int64_t)budget - issued);
  const int32_t op0 = (int32_t)info[1];
  int32_t hn = 0, nb = 0;
  if (lane == 0) {
    mark[op0] = epoch;
    heap_push(heap, hn, op0);
  }
  __syncwarp();
  hn = __shfl_sync(0xffffffffu, hn, 0);
  while (hn > 0 && nb < cap) {
    int32_t x = 0;
    if (lane == 0) {
      x = heap_pop(heap, hn);
      batch[nb] = x;
    }
    x = __shfl_sync(0xffffffffu, x, 0);
    ++nb;
    const uint4 ls = op_lists(g, (uint32_t)x);
    for (uint32_t c0 = 0; c0 < ls.y; c0 += 32) {
      const uint32_t u = c0 + lane;
      int32_t j = -1;
      bool take = false;
      if (u < ls.y) {
        j = (int32_t)__ldg(g.succ + ls.x + u);
        take = state[j] == 0 && mark[j] != epoch;
        if (take) {
          const uint4 jl = op_lists(g, (uint32_t)j);
          for (uint32_t k = 0; k < jl.w && take; ++k) {
            const uint32_t p = __ldg(g.pred + jl.z + k) & kIdMask;
            take = state[p] != 0 || mark[p] == epoch;
          }
        }
      }
      uint32_t m = __ballot_sync(0xffffffffu, take);
      while (m) {
        const int src = __ffs(m) - 1;
        m &= m - 1;
        const int32_t v = __shfl_sync(0xffffffffu, j, src);
        if (lane == 0) {
          mark[v] = epoch;
          heap_push(heap, hn, v);
        }
      }
      __syncwarp();
    }
    hn = __shfl_sync(0xffffffffu, hn, 0);
  }
  if (lane == 0) {
    info[0] = nb;
    info[5] = GMG_ROUND_BATCH;
  }
}

__global__ void __launch_bounds__(256) round_rows_kernel(const uint8_t* __restrict__ place, int32_t ld,
                                                         int32_t n_part, uint8_t* __restrict__ rows) {
  const int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t per = ld / 16;
  if (q >= per * n_part) return;
  const int64_t c = q % per;
  reinterpret_cast<uint4*>(rows)[q] = reinterpret_cast<const uint4*>(place)[c];
}

__global__ void __launch_bounds__(256) round_patch_kernel(const int32_t* __restrict__ batch,
                                                          const int64_t* __restrict__ info, int32_t max_batch,
                                                          int32_t ld, int32_t n_part,
                                                          const int32_t* __restrict__ part_off,
                                                          const uint8_t* __restrict__ part_dev,
                                                          const int32_t* __restrict__ tmpl,
                                                          const int32_t* __restrict__ role,
                                                          const int32_t* __restrict__ map, int32_t n_roles,
                                                          uint8_t* __restrict__ rows) {
  const int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (q >= (int64_t)max_batch * n_part) return;
  const int32_t p = (int32_t)(q / max_batch), b = (int32_t)(q % max_batch);
  if (b >= info[0]) return;
  const int32_t x = batch[b];
  const int32_t s = map[((int64_t)tmpl[x] * n_part + p) * n_roles + role[x]];
  const int32_t size = part_off[p + 1] - part_off[p];
  rows[(int64_t)p * ld + x] = (s >= 0 && s < size) ? part_dev[part_off[p] + s] : (uint8_t)255;
}

// One block: the batch is written back by a strided loop, info[5] by
// thread 0 after every thread has read it.
__global__ void __launch_bounds__(1024) round_commit_kernel(const int32_t* __restrict__ batch, int32_t max_batch,
                                                            int64_t* __restrict__ info,
                                                            const int64_t* __restrict__ best,
                                                            const uint8_t* __restrict__ rows, int32_t ld,
                                                            uint8_t* __restrict__ place,
                                                            uint8_t* __restrict__ state) {
  const int64_t k = best[0];
  const int64_t nb = min(info[0], (int64_t)max_batch);
  const bool have = info[5] == GMG_ROUND_BATCH;
  __syncthreads();
  if (!have) return;
  if (k < 0) {
    if (threadIdx.x == 0) info[5] = GMG_ROUND_NO_FEASIBLE;
    return;
  }
  for (int64_t b = threadIdx.x; b < nb; b += blockDim.x) {
    const int32_t x = batch[b];
    place[x] = rows[k * ld + x];
    state[x] = 1;
  }
}

}  // namespace
}  // namespace ground

using namespace ground;

extern "C" {

size_t round_scratch_bytes(const gmg_t* g) {
  const DevGmg* G = gsim::gmg_device_graph(g);
  return G ? layout(G->n).total : 0;
}

int round_select(const gmg_t* g, const uint8_t* d_state, const int64_t* d_prio, int32_t budget,
                 int32_t max_batch, uint32_t epoch, void* d_scratch, size_t scratch_bytes, int32_t* d_batch,
                 int64_t* d_info, gmg_stream_t stream) {
  const DevGmg* G = gsim::gmg_device_graph(g);
  if (!G || max_batch < 1 || budget < 0 || epoch == 0 || !d_info || !d_batch) return GMG_EINVAL;
  if (G->n > 0 && (!d_state || !d_prio)) return GMG_EINVAL;
  const Layout L = layout(G->n);
  if (!d_scratch || (reinterpret_cast<uintptr_t>(d_scratch) & 255) != 0 || scratch_bytes < L.total)
    return GMG_EWS;
  uint8_t* s = static_cast<uint8_t*>(d_scratch);
  Part* part = reinterpret_cast<Part*>(s + L.part);
  const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int blocks = G->n > 0 ? (G->n + kScanThreads - 1) / kScanThreads : 0;
  if (blocks) round_scan_kernel<<<blocks, kScanThreads, 0, st>>>(*G, d_state, d_prio, part);
  round_reduce_kernel<<<1, 256, 0, st>>>(part, blocks, d_info);
  round_collect_kernel<<<1, 32, 0, st>>>(*G, d_state, budget, max_batch, epoch,
                                         reinterpret_cast<uint32_t*>(s + L.mark),
                                         reinterpret_cast<int32_t*>(s + L.heap), d_batch, d_info);
  return cudaGetLastError() == cudaSuccess ? GMG_OK : GMG_ECUDA;
}

int round_candidates(const gmg_t* g, const uint8_t* d_place, int32_t ld, const int32_t* d_batch,
                     int32_t max_batch, const int64_t* d_info, int32_t n_part, const int32_t* d_part_off, const uint8_t* d_part_dev,
                     const int32_t* d_tmpl, const int32_t* d_role, const int32_t* d_map, int32_t n_roles,
                     uint8_t* d_rows, gmg_stream_t stream) {
  const DevGmg* G = gsim::gmg_device_graph(g);
  if (!G || n_part < 1 || n_roles < 1 || max_batch < 1 || ld < G->n || ld % 16 || !d_place || !d_batch || !d_info ||
      !d_part_off || !d_part_dev || !d_tmpl || !d_role || !d_map || !d_rows)
    return GMG_EINVAL;
  if ((reinterpret_cast<uintptr_t>(d_place) | reinterpret_cast<uintptr_t>(d_rows)) & 15) return GMG_EINVAL;
  const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int64_t nrow = (int64_t)(ld / 16) * n_part;
  round_rows_kernel<<<(int)((nrow + 255) / 256), 256, 0, st>>>(d_place, ld, n_part, d_rows);
  // the batch size is on the device: cover the largest possible batch
  const int64_t nq = (int64_t)max_batch * n_part;
  round_patch_kernel<<<(int)((nq + 255) / 256), 256, 0, st>>>(d_batch, d_info, max_batch, ld, n_part, d_part_off,
                                                                 d_part_dev, d_tmpl, d_role, d_map, n_roles,
                                                                 d_rows);
  return cudaGetLastError() == cudaSuccess ? GMG_OK : GMG_ECUDA;
}

int round_commit(const int32_t* d_batch, int32_t max_batch, int64_t* d_info, const int64_t* d_best,
                 const uint8_t* d_rows, int32_t ld, uint8_t* d_place, uint8_t* d_state, gmg_stream_t stream) {
  if (!d_batch || max_batch < 1 || !d_info || !d_best || !d_rows || !d_place || !d_state || ld < 1)
    return GMG_EINVAL;
  round_commit_kernel<<<1, 1024, 0, reinterpret_cast<cudaStream_t>(stream)>>>(d_batch, max_batch, d_info, d_best,
                                                                               d_rows, ld, d_place, d_state);
  return cudaGetLastError() == cudaSuccess ? GMG_OK : GMG_ECUDA;
}

}  // extern "C"
