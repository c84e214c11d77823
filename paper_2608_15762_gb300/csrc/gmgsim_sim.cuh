// Device side of the what-if placement simulator, shared by the kernel
// translation units (gmgsim_full.cu, gmgsim_inc.cu, gmgsim_kernels.cu).
//
// One warp simulates one candidate placement (Algorithm 1 evaluates the
// candidate partitions "in parallel"; here every warp of a persistent grid
// takes candidates k = warp, warp + W, ...).  Inside a warp the simulation
// is the event-driven loop of Sec. 3.3.3 restated as one ordered sweep:
//
//   READY(r_i, i)  op i's last input has arrived (Sec. 3.3.2 ready time).
//                  Taking READY keys in (r, id) order and starting each op
//                  at s_i = max(r_i, accelerator free time) makes every queue
//                  run its ops in (ready time, id) order, one at a time
//                  (Sec. 3.3.2, Sec. 3.5.1) -- exactly "an idle queue starts
//                  the ready op with the earliest ready time".
//   FREE / ALLOC   HBM events of the copies of an op's output: the op's own
//                  buffer at s_i, a receive buffer on every other accelerator
//                  of a successor at f_i (Recv before Send, Sec. 3.5.2), each
//                  released by its last listed consumer there (Sec. 3.3.2).
//
// READY keys live in a warp-cooperative 32-ary min-heap: the 32 children of
// a node are compared by the 32 lanes at once (one coalesced load, two
// redux.sync), so a pop costs log32(size) warp steps.  Ops without
// predecessors never enter it: their keys are pre-sorted on the host.
//
// HBM events are appended to a per-warp log in O(1).  Every event produced
// while handling READY(r, .) happens at a time >= r, so once the next READY
// key has time T, every logged event with time < T is final and no later
// event can precede it.  Such events are drained in batches: extracted into
// shared memory, bitonic-sorted by (time, frees before allocs, op), and
// applied in order to the per-accelerator live bytes, which gives the peaks
// and the first capacity violation (Sec. 3.4.2 OOM discard) exactly.
//
// Lanes also fan out over successor lists (readiness, transfer arrivals,
// distinct receiving accelerators via __match_any_sync) and predecessor
// lists (ready-time maxima, last-consumer releases).  With at most 32
// accelerators, lane d keeps accelerator d's free time, live bytes and peak
// in registers.
//
// No wait in these kernels depends on another warp or block; the only loop
// whose trip count is not bounded by the data is the event loop, capped at
// g.max_iter iterations (status GMG_SIM_LOOP).

#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <type_traits>

#include "gmg_layout.h"

namespace gsim {
namespace {

constexpr unsigned kFullMask = 0xffffffffu;
constexpr uint64_t kKeyMax = ~0ull;
constexpr int64_t kI64Max = 0x7fffffffffffffffll;

__device__ __forceinline__ uint64_t warp_min_u64(uint64_t v) {
  const uint32_t hi = (uint32_t)(v >> 32), lo = (uint32_t)v;
  const uint32_t mh = __reduce_min_sync(kFullMask, hi);
  const uint32_t ml = __reduce_min_sync(kFullMask, hi == mh ? lo : 0xffffffffu);
  return ((uint64_t)mh << 32) | ml;
}

__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
  const uint32_t hi = (uint32_t)(v >> 32), lo = (uint32_t)v;
  const uint32_t mh = __reduce_max_sync(kFullMask, hi);
  const uint32_t ml = __reduce_max_sync(kFullMask, hi == mh ? lo : 0u);
  return ((uint64_t)mh << 32) | ml;
}

__device__ __forceinline__ unsigned lane_id() { return threadIdx.x & 31u; }
__device__ __forceinline__ uint32_t lanes_below() { return (1u << lane_id()) - 1u; }

// Bulk prefetch of [p, p + bytes) into L2 (no completion to wait for), 32 KB
// pieces spread over the warp.  p is 16-byte aligned; a ragged tail below 16
// bytes is left out.  Single-warp kernels that walk the graph serially start
// with it, so that their dependent loads hit L2 instead of DRAM.
__device__ __forceinline__ void warp_prefetch_l2(const void* p, int64_t bytes) {
  const uint64_t a = (uint64_t)__cvta_generic_to_global(p);
  constexpr int64_t kPiece = 1 << 15;
  for (int64_t o = (int64_t)lane_id() * kPiece; o < bytes; o += 32 * kPiece) {
    const int64_t left = bytes - o;
    const uint32_t sz = (uint32_t)((left < kPiece ? left : kPiece) & ~int64_t(15));
    if (sz) asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" :: "l"(a + o), "r"(sz) : "memory");
  }
}

// The next candidate of a launch that hands them out one at a time (uniform).
__device__ __forceinline__ int64_t take_candidate(uint32_t* next_k) {
  uint32_t k = 0;
  if (lane_id() == 0) k = atomicAdd(next_k, 1u);
  return (int64_t)__shfl_sync(kFullMask, k, 0);
}

// Warp copy of `bytes` rounded up to a multiple of 16 between 16-byte
// aligned buffers (both must extend to the rounded size), kDepth 16-byte
// loads in flight per lane (a single-warp kernel takes a deeper pipeline:
// nothing else hides its load latency).
template <int kDepth = 4>
__device__ __forceinline__ void warp_copy16(void* dst, const void* src, int64_t bytes) {
  const int64_t nv = (bytes + 15) >> 4;
  uint4* d = static_cast<uint4*>(dst);
  const uint4* s = static_cast<const uint4*>(src);
  int64_t i = lane_id();
  for (; i + 32 * (kDepth - 1) < nv; i += 32 * kDepth) {
    uint4 v[kDepth];
#pragma unroll
    for (int u = 0; u < kDepth; ++u) v[u] = s[i + 32 * u];
#pragma unroll
    for (int u = 0; u < kDepth; ++u) d[i + 32 * u] = v[u];
  }
  for (; i < nv; i += 32) d[i] = s[i];
}

// 16-byte pieces of an OpRec, loaded through the read-only path.
__device__ __forceinline__ longlong2 op_durbytes(const OpRec* ops, uint32_t i) {
  return __ldg(reinterpret_cast<const longlong2*>(ops + i));
}
struct RelPred {
  int64_t rel;
  uint32_t pred_off, npred;
};
struct XqSucc {
  int64_t xq;
  uint32_t succ_off, nsucc;
};
__device__ __forceinline__ RelPred op_relpred(const OpRec* ops, uint32_t i) {
  const uint4 v = __ldg(reinterpret_cast<const uint4*>(ops + i) + 1);
  return RelPred{(int64_t)(((uint64_t)v.y << 32) | v.x), v.z, v.w};
}
__device__ __forceinline__ XqSucc op_xqsucc(const OpRec* ops, uint32_t i) {
  const uint4 v = __ldg(reinterpret_cast<const uint4*>(ops + i) + 2);
  return XqSucc{(int64_t)(((uint64_t)v.y << 32) | v.x), v.z, v.w};
}
// (succ_off, nsucc, pred_off, npred) from two pieces, for code that needs both lists.
__device__ __forceinline__ uint4 op_lists(const OpRec* ops, uint32_t i) {
  const XqSucc a = op_xqsucc(ops, i);
  const RelPred b = op_relpred(ops, i);
  return make_uint4(a.succ_off, a.nsucc, b.pred_off, b.npred);
}
__device__ __forceinline__ uint4 op_cons(const OpRec* ops, uint32_t i) {
  return __ldg(reinterpret_cast<const uint4*>(ops + i) + 3);  // cons_off, ncons, req, flags
}

struct KeyCodec {
  int ib;
  uint64_t mask;
  template <typename TM>
  __device__ __forceinline__ uint64_t make(TM t, uint32_t cls, uint32_t op) const {
    using U = typename std::make_unsigned<TM>::type;
    return ((uint64_t)(U)t << (ib + 2)) | ((uint64_t)cls << ib) | (uint64_t)op;
  }
  __device__ __forceinline__ int64_t time(uint64_t k) const { return (int64_t)(k >> (ib + 2)); }
  __device__ __forceinline__ uint64_t time_floor(int64_t t) const { return (uint64_t)t << (ib + 2); }
  __device__ __forceinline__ uint32_t cls(uint64_t k) const { return (uint32_t)(k >> ib) & 3u; }
  __device__ __forceinline__ uint32_t op(uint64_t k) const { return (uint32_t)(k & mask); }
};

// READY keys as queued: the KeyCodec key with class READY, shifted up by qb
// bits that hold the op's duration class (floor(log2) of a lower bound of its
// duration) in the batched sweep; qb = 0 otherwise (then equal to the
// KeyCodec key).  The class bits sit below the op id, so they never change
// the order of two keys.
struct ReadyCodec {
  int ib, qb;
  uint64_t mask;
  template <typename TM>
  __device__ __forceinline__ uint64_t make(TM t, uint32_t op, uint32_t q) const {
    using U = typename std::make_unsigned<TM>::type;
    return ((((uint64_t)(U)t << (ib + 2)) | (uint64_t)op) << qb) | (qb ? (uint64_t)q : 0ull);
  }
  __device__ __forceinline__ int64_t time(uint64_t k) const { return (int64_t)(k >> (ib + 2 + qb)); }
  __device__ __forceinline__ uint32_t op(uint64_t k) const { return (uint32_t)((k >> qb) & mask); }
  __device__ __forceinline__ uint32_t q(uint64_t k) const { return (uint32_t)k & ((1u << qb) - 1u); }
};

// floor(log2(dur)) for dur >= 1, at most 31: 2^class is a lower bound of dur.
__device__ __forceinline__ uint32_t dur_class(int64_t dur) {
  const uint32_t c = 63u - (uint32_t)__clzll((unsigned long long)dur);
  return c < 31u ? c : 31u;
}

__device__ __forceinline__ int64_t warp_sum_i64(int64_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFullMask, v, o);
  return v;
}

// ---------------------------------------------------------------------------
// READY keys: warp-cooperative 32-ary min-heap.  Slots [0, qs) are in shared
// memory (qs >= 33, so the root and its children always are), the rest in
// the warp's global scratch.  All lanes call every method with the same
// arguments; lane 0 performs the stores.
// ---------------------------------------------------------------------------
struct ReadyHeap {
  uint64_t* sk;
  uint64_t* gk;
  int qs, cap, size;

  __device__ __forceinline__ uint64_t* kp(int i) const { return i < qs ? sk + i : gk + (i - qs); }
  __device__ __forceinline__ uint64_t top() const { return size > 0 ? sk[0] : kKeyMax; }

  __device__ void sift_down(int pos, uint64_t x) {
    const unsigned lane = lane_id();
    while (true) {
      const int c0 = pos * 32 + 1;
      if (c0 >= size) break;
      const int idx = c0 + (int)lane;
      uint64_t ck = kKeyMax;
      if (idx < size) ck = c0 == 1 ? sk[idx] : *kp(idx);
      const uint64_t m = warp_min_u64(ck);
      if (m >= x) break;
      const int src = __ffs(__ballot_sync(kFullMask, ck == m)) - 1;
      if (lane == 0) *kp(pos) = m;
      pos = c0 + src;
    }
    if (lane == 0) *kp(pos) = x;
    __syncwarp();
  }

  // The same as sift_down while every slot in use is in shared memory.
  __device__ void sift_down_shared(int pos, uint64_t x) {
    const unsigned lane = lane_id();
    while (true) {
      const int c0 = pos * 32 + 1;
      if (c0 >= size) break;
      const int idx = c0 + (int)lane;
      const uint64_t ck = idx < size ? sk[idx] : kKeyMax;
      const uint64_t m = warp_min_u64(ck);
      if (m >= x) break;
      const int src = __ffs(__ballot_sync(kFullMask, ck == m)) - 1;
      if (lane == 0) sk[pos] = m;
      pos = c0 + src;
    }
    if (lane == 0) sk[pos] = x;
    __syncwarp();
  }

  __device__ void pop() {
    const int n = --size;
    if (n == 0) return;
    const uint64_t x = *kp(n);
    sift_down(0, x);
  }

  // pop / push with a branch for a heap held entirely in shared memory (the
  // batched sweep's larger shared part makes that the common case)
  __device__ void pop_fast() {
    const int n = --size;
    if (n == 0) return;
    if (n < qs) {
      sift_down_shared(0, sk[n]);
      return;
    }
    const uint64_t x = *kp(n);
    sift_down(0, x);
  }

  __device__ bool push_fast(uint64_t key) {
    if (size >= cap) return false;
    if (size < qs) {
      int pos = size++;
      while (pos > 0) {
        const int par = (pos - 1) >> 5;
        const uint64_t pk = sk[par];
        if (pk <= key) break;
        if (lane_id() == 0) sk[pos] = pk;
        pos = par;
      }
      if (lane_id() == 0) sk[pos] = key;
      __syncwarp();
      return true;
    }
    return push(key);
  }

  __device__ bool push(uint64_t key) {
    if (size >= cap) return false;
    int pos = size++;
    while (pos > 0) {
      const int par = (pos - 1) >> 5;
      const uint64_t pk = *kp(par);
      if (pk <= key) break;
      if (lane_id() == 0) *kp(pos) = pk;
      pos = par;
    }
    if (lane_id() == 0) *kp(pos) = key;
    __syncwarp();
    return true;
  }

  __device__ void heapify() {
    if (size < 2) return;
    for (int pos = (size - 2) / 32; pos >= 0; --pos) {
      const uint64_t x = *kp(pos);
      __syncwarp();
      sift_down(pos, x);
    }
  }
};

// ---------------------------------------------------------------------------
// HBM event log: unordered 8-byte entries -- (accelerator << ds) | key when
// the accelerator id fits above the key, else the key with the accelerator
// in a side byte array.  Slots [0, ms) are in shared memory, the rest in
// global scratch.
// ---------------------------------------------------------------------------
struct MemLog {
  uint64_t* sk;
  uint8_t* sd;
  uint64_t* gk;
  uint8_t* gd;
  int ms, cap, n;

  __device__ __forceinline__ uint64_t* kp(int i) const { return i < ms ? sk + i : gk + (i - ms); }
  __device__ __forceinline__ uint8_t* dp(int i) const { return i < ms ? sd + i : gd + (i - ms); }
};

// ---------------------------------------------------------------------------
// Per-accelerator state.  Free times: with at most 32 accelerators lane d
// holds accelerator d's in a register, else a shared array of the kernel's
// time type.  Live bytes: a shared array (the drain updates it a batch at a
// time).  Peak bytes: a shared array, or with more than 32 accelerators an
// array in the warp's global scratch (only raised by atomicMax and read at
// the end, so its latency is never waited on).
// ---------------------------------------------------------------------------
template <bool kReg, typename TM>
struct Devices {
  TM fr_reg;
  TM* fr;       // shared [D] (when !kReg)
  int64_t* lv;  // shared [D]
  int64_t* pk;  // [D], shared or global
  int D;
  __device__ void setup(const DevGmg& g, uint8_t* sm, int64_t* pk_global) {
    D = g.D;
    lv = reinterpret_cast<int64_t*>(sm);
    if (kReg) {  // peaks in shared memory (a compile-time fact for these instances)
      pk = lv + D;
      fr = nullptr;
    } else {
      pk = pk_global;
      fr = reinterpret_cast<TM*>(lv + D);
    }
  }
  __device__ void reset(const DevGmg& g) {
    const unsigned l = lane_id();
    for (int d = l; d < D; d += 32) {
      lv[d] = g.base[d];
      pk[d] = g.base[d];
      if (!kReg) fr[d] = (TM)g.avail0[d];
    }
    if (kReg) fr_reg = l < (unsigned)D ? (TM)g.avail0[l] : (TM)0;
    __syncwarp();
  }
  __device__ __forceinline__ TM get_free(int d) const {
    if (kReg) return __shfl_sync(kFullMask, fr_reg, d);
    return fr[d];
  }
  __device__ __forceinline__ void set_free(int d, TM v) {
    if (kReg) {
      if ((int)lane_id() == d) fr_reg = v;
    } else {
      __syncwarp();
      if (lane_id() == 0) fr[d] = v;
    }
  }
  // One event at a time (used when accelerator ids do not fit in the sort key).
  __device__ __forceinline__ bool alloc(int d, int64_t b, int64_t cap) {
    const int64_t v = lv[d] + b;
    const int64_t p = pk[d];
    __syncwarp();
    if (lane_id() == 0) {
      lv[d] = v;
      if (v > p) pk[d] = v;
    }
    __syncwarp();
    return v > cap;
  }
  __device__ __forceinline__ void release(int d, int64_t b) {
    const int64_t v = lv[d] - b;
    __syncwarp();
    if (lane_id() == 0) lv[d] = v;
    __syncwarp();
  }
  __device__ void save(int64_t* dst) const {
    const unsigned l = lane_id();
    for (int d = l; d < D; d += 32) {
      if (!kReg) dst[d] = (int64_t)fr[d];
      dst[D + d] = lv[d];
      dst[2 * D + d] = pk[d];
    }
    if (kReg && l < (unsigned)D) dst[l] = (int64_t)fr_reg;
  }
  __device__ void load(const int64_t* src) {
    const unsigned l = lane_id();
    for (int d = l; d < D; d += 32) {
      if (!kReg) fr[d] = (TM)src[d];
      lv[d] = src[D + d];
      pk[d] = src[2 * D + d];
    }
    if (kReg) fr_reg = l < (unsigned)D ? (TM)src[l] : (TM)0;
    __syncwarp();
  }
  // Largest final free time over the accelerators whose free time moved past
  // their initial availability (0 if none).  Uniform result.
  __device__ int64_t max_busy(const DevGmg& g) const {
    uint64_t m = 0;
    for (int d = lane_id(); d < D; d += 32) {
      const int64_t f = kReg ? (int64_t)fr_reg : (int64_t)fr[d];
      if (f > g.avail0[d]) m = (uint64_t)f > m ? (uint64_t)f : m;
    }
    return (int64_t)warp_max_u64(m);
  }
  __device__ void write_peak(int64_t* dst) const {
    for (int d = lane_id(); d < D; d += 32) dst[d] = pk[d];
  }
};

// Shared-memory carve-up per warp: READY heap head, event-log head, sort
// area, accelerator state.
struct WarpSmem {
  uint32_t* oplog;  // [opcap]
  uint64_t* heap;   // [qs]
  uint64_t* logk;   // [ms]
  uint64_t* sortk;  // [sortcap]
  uint8_t* logd;    // [ms]
  uint8_t* sortd;   // [sortcap]
  uint8_t* dev;     // accelerator state (P.dev_bytes)
};

__device__ __forceinline__ size_t align16(size_t x) { return (x + 15) & ~(size_t)15; }

__device__ __forceinline__ WarpSmem carve_smem(uint8_t* smem, const SimParams& P, unsigned wib) {
  // the side bytes (accelerator of a log entry) are left out where the
  // accelerator is inside the entry and shared memory is tight (P.no_side)
  const size_t side = P.no_side ? 0 : 1;
  const size_t head = align16((size_t)P.qs * 8 + (size_t)P.ms * (8 + side) + (size_t)P.sortcap * (8 + side) +
                              (size_t)P.opcap * 4);
  const size_t per = head + (size_t)P.dev_bytes;
  uint8_t* b = smem + per * wib;
  WarpSmem w;
  w.heap = reinterpret_cast<uint64_t*>(b);
  w.logk = w.heap + P.qs;
  w.sortk = w.logk + P.ms;
  w.logd = reinterpret_cast<uint8_t*>(w.sortk + P.sortcap);
  w.sortd = w.logd + P.ms * side;
  w.oplog = reinterpret_cast<uint32_t*>(w.sortd + P.sortcap * side);
  w.dev = b + head;
  return w;
}

// ---------------------------------------------------------------------------
// One warp's simulator.
// ---------------------------------------------------------------------------
// kT32: every time of the graph is below 2^31 (the host's bound), so ready,
// start, finish, free and arrival times are carried as int32 (bytes, scores
// and outputs stay int64).
// kTypes: the graph has several accelerator types (durations per (type, op)).
// kBatch: the batched sweep (run_batched), for accelerator state in shared
// memory with the accelerator id in the event key.
// kStage: the hot fields of the GMG (durations, transfer sizes, flags, both
// CSR lists, releases) are read from the CTA's shared-memory copy (staged by
// sim_full_staged_kernel) when starting ops and testing successors.
template <bool kReg, int kMode, bool kKey, bool kT32 = false, bool kTypes = false, bool kBatch = false,
          bool kStage = false>
struct Sim {
  static_assert(!(kT32 && kMode == kBase), "the base snapshot keeps 64-bit times");
  static_assert(!kBatch || (!kReg && kKey), "the batched sweep keeps accelerator state in shared memory");
  static_assert(!kStage || (kMode == kFull && kT32 && !kTypes && !kBatch), "staged GMG: 32-bit, one type");
  using tm_t = typename std::conditional<kT32, int32_t, int64_t>::type;
  const SimParams& P;
  const DevGmg& g;
  KeyCodec kc;      // HBM log entries (and READY keys when qb = 0)
  ReadyCodec rq;    // READY keys
  ReadyHeap q;      // READY keys beyond the register tier
  uint64_t rk_reg;  // register tier: one READY key per lane (kKeyMax = empty)
  MemLog log;
  uint64_t* sortk;
  uint8_t* sortd;
  int sortcap;
  uint32_t* oplog;  // ops started since the last HBM-event generation
  int opn;
  int ds;           // accelerator shift of a log entry
  uint64_t lowmask; // key part of a log entry
  Devices<kReg, tm_t> dv;
  const uint8_t* row;
  tm_t* fbuf;       // finish times (scratch; the base's own array in kBase)
  tm_t* holdb;      // latest outgoing arrival of each op's output (scratch)
  uint32_t* bits;
  int64_t* creq;
  // incremental resume
  const int64_t* rb;
  const int64_t* fb;
  tm_t Tc, T0;
  // running results
  int rootptr;
  uint64_t rkey;    // root_keys[rootptr], kKeyMax past the end
  int64_t score, nev, readypops;
  int32_t iters;        // ops started (loop guard; the event count of a full run)
  tm_t makespan, last_t;  // running values, kept in base mode only (checkpoints)
  int32_t vflag, vop, vdev, status;
  int64_t vt;
  // base checkpoints
  int ck, next_ck;
  // staged GMG (kStage): shared copies
  const uint4* sh_hot;      // per op {dur, xq | flags << 29, succ_off | nsucc << 24, pred_off | npred << 24}
  const int32_t* sh_rel;    // per op release
  const uint32_t* sh_succ;  // successor lists
  const uint32_t* sh_pred;  // predecessor lists (hold bits included)

  __device__ Sim(const SimParams& p) : P(p), g(p.g) {
    kc.ib = g.ib;
    kc.mask = (1ull << g.ib) - 1ull;
    rq.ib = g.ib;
    rq.mask = kc.mask;
    rq.qb = kBatch ? kQB : 0;
    ds = g.ib + 2 + g.tb;
    lowmask = kKey ? (1ull << ds) - 1ull : kKeyMax;
  }

  // Started ops are those with a finish time (every finish time is >= 1;
  // the finish array is zeroed per candidate; the batched sweep marks an op
  // whose READY key is queued with -1).
  __device__ __forceinline__ bool popped(uint32_t x) const { return fin(x) > 0; }
  // The low 32 bits of a base-snapshot time (little-endian int64).
  static __device__ __forceinline__ tm_t base_time(const int64_t* a, uint32_t x) {
    if (kT32) return (tm_t)__ldg(reinterpret_cast<const int32_t*>(a) + 2 * (size_t)x);
    return (tm_t)__ldg(a + x);
  }
  // Duration of op i on accelerator d: by the accelerator's type when the
  // graph has several (Sec. 3.3.1 keeps one operator estimate per (type,
  // operator)), else the op record's dur (dflt).
  __device__ __forceinline__ int64_t dur_of(uint32_t i, int d, int64_t dflt) const {
    if (kTypes) return __ldg(g.durt + (size_t)i * g.ntypes + __ldg(g.dtype + d));
    return dflt;
  }
  // Finish time of a simulated op (incremental candidates start from
  // fill_fin: ops started before the resume point keep their base finish).
  __device__ __forceinline__ tm_t fin(uint32_t x) const { return fbuf[x]; }

  // Transfer estimator of one output over link d -> e (d != e), Sec. 3.3.1.
  __device__ __forceinline__ tm_t xfer(int d, int e, int64_t bytes, int64_t xq) const {
    if (g.uniform) return (tm_t)xq + (tm_t)g.lat0;
    const longlong2* L = reinterpret_cast<const longlong2*>(g.links + (d * g.D + e));
    const longlong2 a = __ldg(L), b = __ldg(L + 1);
    LinkRec l;
    l.magic = (uint64_t)a.x;
    l.bw = a.y;
    l.lat = b.x;
    l.shift = (int32_t)(b.y & 0xffffffff);
    return (tm_t)(ceil_div_link(bytes, l) + l.lat);
  }

  // Latest arrival of p's output at another accelerator (or f_p): the
  // earliest its source copy may be released.  Per lane.
  __device__ tm_t lane_hold(uint32_t p, tm_t fp, int dp) const {
    const int64_t pb = op_durbytes(g.ops, p).y;
    const XqSucc ps = op_xqsucc(g.ops, p);
    const int64_t pxq = ps.xq;
    tm_t h = fp;
    for (uint32_t u = 0; u < ps.nsucc; ++u) {
      const int du = row[__ldg(g.succ + ps.succ_off + u)];
      if (du != dp) {
        const tm_t a = fp + xfer(dp, du, pb, pxq);
        h = a > h ? a : h;
      }
    }
    return h;
  }


  __device__ __forceinline__ void load_root() {
    rkey = rootptr < g.nroots ? __ldg((kBatch ? g.root_keys_q : g.root_keys) + rootptr) : kKeyMax;
  }

  // READY keys go to a free lane's register if there is one, else the heap.
  __device__ __forceinline__ void push_ready(uint64_t key) {
    const uint32_t freel = __ballot_sync(kFullMask, rk_reg == kKeyMax);
    if (freel) {
      if ((int)lane_id() == __ffs(freel) - 1) rk_reg = key;
    } else if (!(kBatch ? q.push_fast(key) : q.push(key))) {
      status = GMG_SIM_QUEUE;
    }
  }
  // Every lane with `want` logs (key, dev).  Uniform call.
  __device__ __forceinline__ void log_event(bool want, uint64_t key, int dev) {
    const uint32_t b = __ballot_sync(kFullMask, want);
    const int cnt = __popc(b);
    const int pos = log.n + __popc(b & lanes_below());
    if (kKey && log.n + 32 <= log.ms) {
      // fast path: every lane's slot is in shared memory
      if (want) log.sk[pos] = ((uint64_t)(dev & 0xff) << ds) | key;
      log.n += cnt;
      return;
    }
    if (cnt == 0 || status) return;
    if (log.n + cnt > log.cap) {
      status = GMG_SIM_QUEUE;
      return;
    }
    if (want) {
      *log.kp(pos) = kKey ? (((uint64_t)(dev & 0xff) << ds) | key) : key;
      if (!kKey) *log.dp(pos) = (uint8_t)dev;
    }
    log.n += cnt;
  }

  // Zero this candidate's finish times (16-byte stores; the array is padded).
  __device__ void zero_fin() {
    uint4* v = reinterpret_cast<uint4*>(fbuf);
    const int nv = (int)((sizeof(tm_t) * (size_t)g.n + 15) / 16);
    for (int x = lane_id(); x < nv; x += 32) v[x] = make_uint4(0u, 0u, 0u, 0u);
    __syncwarp();
  }

  // An incremental candidate's finish times at the resume point T_c: the
  // base finish of every op started before it (base ready time < T_c), zero
  // for the others and for the padding.  Four ops in flight per lane.
  __device__ void fill_fin() {
    const int n = g.n;
    const int np = (int)((sizeof(tm_t) * (size_t)n + 15) / 16 * 16 / sizeof(tm_t));
    int x = (int)lane_id();
    for (; x + 96 < np; x += 128) {
      tm_t v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = x + 32 * u;
        const bool in = i < n;
        const tm_t r = in ? base_time(rb, (uint32_t)i) : Tc;
        const tm_t f = in ? base_time(fb, (uint32_t)i) : 0;
        v[u] = r < Tc ? f : 0;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) fbuf[x + 32 * u] = v[u];
    }
    for (; x < np; x += 32) {
      const bool in = x < n;
      const tm_t r = in ? base_time(rb, (uint32_t)x) : Tc;
      fbuf[x] = r < Tc ? base_time(fb, (uint32_t)x) : 0;
    }
    __syncwarp();
  }

  __device__ void reset_common() {
    const unsigned lane = lane_id();
    zero_fin();
    for (int r = lane; r < g.R; r += 32) creq[r] = 0;
    dv.reset(g);
    q.size = 0;
    rk_reg = kKeyMax;
    log.n = 0;
    opn = 0;
    rootptr = 0;
    load_root();
    score = makespan = 0;
    iters = nev = readypops = 0;
    last_t = -1;
    vflag = 0;
    vop = vdev = -1;
    vt = -1;
    status = GMG_SIM_OK;
    __syncwarp();
  }

  // -------------------------------------------------------------------------
  // READY(r, i): start op i (Sec. 3.3.2/3.3.3), record it for HBM-event
  // generation, and push the successors it makes ready.
  // -------------------------------------------------------------------------
  __device__ void start_op(uint32_t i, tm_t r) {
    if constexpr (kStage) {
      start_op_staged(i, r);
      return;
    }
    const unsigned lane = lane_id();
    const longlong2 db = op_durbytes(g.ops, i);
    const XqSucc xs = op_xqsucc(g.ops, i);
    const uint4 cs = op_cons(g.ops, i);
    const int64_t bytes = db.y, xq = xs.xq;
    const uint32_t succ_off = xs.succ_off, nsucc = xs.nsucc;
    const uint32_t flags = cs.w;
    const int d = row[i];
    const tm_t dur = (tm_t)dur_of(i, d, db.x);
    const tm_t fd = dv.get_free(d);
    const tm_t s = r > fd ? r : fd;
    const tm_t f = s + dur;
    dv.set_free(d, f);
    if (lane == 0) {
      fbuf[i] = f;
      if (flags & kReqSink)
        atomicMax(reinterpret_cast<unsigned long long*>(creq + (int32_t)cs.z), (unsigned long long)f);
      if (kMode == kBase) P.base.rb[i] = r;
      oplog[opn] = i;
    }
    ++opn;
    if (flags & kScored) score += (int64_t)f;
    if (kMode == kBase) makespan = f > makespan ? f : makespan;
    if (kMode == kInc && r >= T0) ++nev;
    if (kMode == kBase) ++readypops;
    __syncwarp();

    // Successors: a successor is ready once every predecessor has finished;
    // its ready time is the latest arrival over all of them.
    for (uint32_t c0 = 0; c0 < nsucc; c0 += 32) {
      const uint32_t t = c0 + lane;
      uint32_t j = 0;
      tm_t rj = 0;
      bool rdy = false;
      if (t < nsucc) {
        j = __ldg(g.succ + succ_off + t);
        const int dj = row[j];
        tm_t arr = f;
        if (dj != d) arr = f + xfer(d, dj, bytes, xq);
        const RelPred jp = op_relpred(g.ops, j);
        const tm_t rel = (tm_t)jp.rel;
        rj = rel > arr ? rel : arr;
        rdy = true;
        if (jp.npred > 1) {
          for (uint32_t k = 0; k < jp.npred; ++k) {
            const uint32_t p = __ldg(g.pred + jp.pred_off + k) & kIdMask;
            if (p == i) continue;
            tm_t a = fin(p);
            if (a <= 0) {  // not started yet
              rdy = false;
              break;
            }
            const int dp = row[p];
            if (dp != dj) a += xfer(dp, dj, op_durbytes(g.ops, p).y, op_xqsucc(g.ops, p).xq);
            rj = a > rj ? a : rj;
          }
        }
      }
      uint32_t m = __ballot_sync(kFullMask, rdy);
      while (m) {
        const int src = __ffs(m) - 1;
        m &= m - 1;
        push_ready(__shfl_sync(kFullMask, kc.make(rj, kReady, j), src));
      }
    }
  }

  // start_op with the hot fields from the CTA's staged copy of the GMG (the
  // links are uniform: a transfer takes xq + lat0).
  __device__ void start_op_staged(uint32_t i, tm_t r) {
    const unsigned lane = lane_id();
    const uint4 h = sh_hot[i];
    const uint32_t flags = h.y >> 29;
    const tm_t xq = (tm_t)(h.y & 0x1fffffffu);
    const uint32_t succ_off = h.z & 0xffffffu, nsucc = h.z >> 24;
    const int d = row[i];
    const tm_t fd = dv.get_free(d);
    const tm_t s = r > fd ? r : fd;
    const tm_t f = s + (tm_t)(int32_t)h.x;
    dv.set_free(d, f);
    if (lane == 0) {
      fbuf[i] = f;
      if (flags & kReqSink)
        atomicMax(reinterpret_cast<unsigned long long*>(creq + (int32_t)op_cons(g.ops, i).z), (unsigned long long)f);
      oplog[opn] = i;
    }
    ++opn;
    if (flags & kScored) score += (int64_t)f;
    __syncwarp();
    const tm_t lat = (tm_t)g.lat0;
    for (uint32_t c0 = 0; c0 < nsucc; c0 += 32) {
      const uint32_t t = c0 + lane;
      uint32_t j = 0;
      tm_t rj = 0;
      bool rdy = false;
      if (t < nsucc) {
        j = sh_succ[succ_off + t];
        const int dj = row[j];
        const tm_t arr = dj != d ? f + xq + lat : f;
        const uint32_t po = sh_hot[j].w;
        const uint32_t npred = po >> 24, pred_off = po & 0xffffffu;
        const tm_t rel = (tm_t)sh_rel[j];
        rj = rel > arr ? rel : arr;
        rdy = true;
        if (npred > 1) {
          for (uint32_t k = 0; k < npred; ++k) {
            const uint32_t p = sh_pred[pred_off + k] & kIdMask;
            if (p == i) continue;
            tm_t a = fin(p);
            if (a <= 0) {  // not started yet
              rdy = false;
              break;
            }
            if (row[p] != dj) a += (tm_t)(sh_hot[p].y & 0x1fffffffu) + lat;
            rj = a > rj ? a : rj;
          }
        }
      }
      uint32_t m = __ballot_sync(kFullMask, rdy);
      while (m) {
        const int src = __ffs(m) - 1;
        m &= m - 1;
        push_ready(__shfl_sync(kFullMask, kc.make(rj, kReady, j), src));
      }
    }
  }

  // -------------------------------------------------------------------------
  // HBM events of the ops started since the last generation, one op per lane
  // (Sec. 3.3.2 residency, Recv before Send of Sec. 3.5.2): the op's own
  // output allocated at s; a receive copy on every other accelerator of a
  // successor allocated at f (released on arrival if no listed consumer is
  // there); the own copy released at the latest outgoing arrival if no
  // listed consumer is local; and for every held input whose last local
  // consumer this op is, that copy released at f (an own copy not before its
  // producer's outgoing arrivals).  Ops on one accelerator finish in the
  // order they start, so "last consumer here" compares finish times and can
  // be decided any time after the op started.
  // -------------------------------------------------------------------------
  __device__ void generate() {
    const unsigned lane = lane_id();
    for (int c0 = 0; c0 < opn; c0 += 32) {
      const int idx = c0 + (int)lane;
      const bool v = idx < opn;
      const uint32_t x = v ? oplog[idx] : 0u;
      longlong2 db = make_longlong2(0, 0), rx = make_longlong2(0, 0);
      uint4 ls = make_uint4(0, 0, 0, 0), cs = make_uint4(0, 0, 0, 0);
      int d = 0;
      tm_t f = 0;
      if (v) {
        db = op_durbytes(g.ops, x);
        const XqSucc xs = op_xqsucc(g.ops, x);
        const RelPred rp = op_relpred(g.ops, x);
        rx = make_longlong2(rp.rel, xs.xq);
        ls = make_uint4(xs.succ_off, xs.nsucc, rp.pred_off, rp.npred);
        cs = op_cons(g.ops, x);
        d = row[x];
        f = fbuf[x];
      }
      const int64_t bytes = db.y, xq = rx.y;
      const bool allcons = (cs.w & kAllCons) != 0;
      log_event(v, kc.make(f - (tm_t)dur_of(x, d, db.x), kAlloc, x), d);
      // receive copies, one per distinct remote accelerator
      tm_t hold = f;
      bool localc = false;
      const uint32_t nsx = ls.y;
      const uint32_t maxs = __reduce_max_sync(kFullMask, nsx);
      const bool anyexp = __any_sync(kFullMask, v && !allcons);
      for (uint32_t u = 0; u < maxs; ++u) {
        bool want = false, nocons = false;
        int du = 0;
        tm_t arr = f;
        if (u < nsx) {
          du = row[__ldg(g.succ + ls.x + u)];
          if (du == d) {
            localc = true;
          } else {
            want = true;
            for (uint32_t w = 0; w < u; ++w)
              if (row[__ldg(g.succ + ls.x + w)] == du) {
                want = false;
                break;
              }
          }
          if (want) {
            arr = f + xfer(d, du, bytes, xq);
            hold = arr > hold ? arr : hold;
            if (!allcons) {
              nocons = true;
              for (uint32_t w = 0; w < cs.y; ++w)
                if (row[__ldg(g.cons + cs.x + w)] == du) {
                  nocons = false;
                  break;
                }
            }
          }
        }
        log_event(want, kc.make(f, kAlloc, x), du);
        if (anyexp) log_event(nocons, kc.make(arr, kFree, x), du);
      }
      if (v && !allcons) {
        localc = false;
        for (uint32_t w = 0; w < cs.y; ++w)
          if (row[__ldg(g.cons + cs.x + w)] == d) {
            localc = true;
            break;
          }
      }
      log_event(v && !localc, kc.make(hold, kFree, x), d);
      if (v) holdb[x] = hold;
      __syncwarp();
      // releases of the inputs this op holds
      const uint32_t npx = ls.w;
      const uint32_t maxp = __reduce_max_sync(kFullMask, npx);
      for (uint32_t u = 0; u < maxp; ++u) {
        bool rel = false;
        tm_t T = f;
        uint32_t p = 0;
        if (u < npx) {
          const uint2 ps = __ldg(g.predsib + ls.z + u);
          p = ps.x & kIdMask;
          if (ps.x & kHoldBit) {
            const uint32_t sb = ps.y;
            if (sb == kSibNone) {
              rel = true;
            } else if (sb != kSibMany && (sb & kSibLater)) {
              rel = row[sb & ~kSibLater] != d;  // the other consumer finishes later
            } else if (sb != kSibMany) {
              const tm_t fs = fin(sb);
              rel = !(row[sb] == d && !(fs > 0 && fs < f));
            } else {
              const XqSucc px = op_xqsucc(g.ops, p);
              const uint4 pls = make_uint4(px.succ_off, px.nsucc, 0u, 0u);
              const uint4 pcs = op_cons(g.ops, p);
              const bool all = (pcs.w & kAllCons) != 0;
              const uint32_t* lst = all ? g.succ + pls.x : g.cons + pcs.x;
              const uint32_t nl = all ? pls.y : pcs.y;
              rel = true;
              for (uint32_t w = 0; w < nl; ++w) {
                const uint32_t c = __ldg(lst + w);
                const tm_t fc = c != x ? fin(c) : 0;
                if (c != x && row[c] == d && !(fc > 0 && fc < f)) {
                  rel = false;
                  break;
                }
              }
            }
            if (rel && row[p] == d) {
              // p's own copy: not before its outgoing arrivals (recorded when
              // p's events were generated; p started before this op)
              const tm_t h = (kMode == kInc && base_time(rb, p) < Tc) ? lane_hold(p, fin(p), d) : holdb[p];
              T = h > T ? h : T;
            }
          }
        }
        log_event(rel, kc.make(T, kFree, p), d);
      }
    }
    opn = 0;
    __syncwarp();
  }

  // Apply sorted events one at a time (accelerator ids not in the key).
  __device__ void apply_serial(int m) {
    for (int e = 0; e < m; ++e) {
      const uint64_t k = sortk[e];
      const int dev = sortd[e];
      const uint32_t op = kc.op(k);
      const int64_t b = op_durbytes(g.ops, op).y;
      if (kc.cls(k) == kFree) {
        dv.release(dev, b);
      } else if (dv.alloc(dev, b, __ldg(g.cap + dev))) {
        const int64_t t = kc.time(k);
        if (!vflag || (t == vt && (int32_t)op == vop && dev < vdev)) {
          vflag = 1;
          vt = t;
          vop = (int32_t)op;
          vdev = dev;
        }
      }
    }
    __syncwarp();
  }

  // Apply 32 consecutive events of the (accelerator, time, class, op) order,
  // one per lane (v: lane holds an event).  Each accelerator's events are
  // contiguous, so a segmented warp scan of the byte deltas gives the live
  // bytes after every event; allocations raise the accelerator's peak; the
  // smallest (time, op, accelerator) allocation over capacity is kept in
  // vmin.
  __device__ __forceinline__ void apply_chunk(uint64_t key, bool v, uint64_t& vmin) {
    const unsigned lane = lane_id();
    const uint64_t tmask = (1ull << g.tb) - 1ull;
    const int dev = v ? (int)(key >> ds) : -1 - (int)lane;
    const uint32_t op = (uint32_t)(key & kc.mask);
    const bool isalloc = v && kc.cls(key) == kAlloc;
    int64_t delta = 0;
    if (v) {
      const int64_t b = op_durbytes(g.ops, op).y;
      delta = isalloc ? b : -b;
    }
    int64_t s = delta;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int64_t o = __shfl_up_sync(kFullMask, s, off);
      const int od = __shfl_up_sync(kFullMask, dev, off);
      if ((int)lane >= off && od == dev) s += o;
    }
    const int64_t live = (v ? dv.lv[dev] : 0) + s;
    const int nd = __shfl_down_sync(kFullMask, dev, 1);
    const bool last = v && (lane == 31 || nd != dev);
    const bool over = isalloc && live > __ldg(g.cap + dev);
    const uint64_t vk = over ? ((((key >> (g.ib + 2)) & tmask) << (g.ib + 8)) | ((uint64_t)op << 8) |
                                (uint64_t)dev)
                             : kKeyMax;
    const uint64_t cm = warp_min_u64(vk);
    vmin = cm < vmin ? cm : vmin;
    __syncwarp();
    if (isalloc)  // live bytes are never negative
      atomicMax(reinterpret_cast<unsigned long long*>(dv.pk + dev), (unsigned long long)live);
    if (last) dv.lv[dev] = live;
    __syncwarp();
  }

  // every event of a drain is later than every event already applied, so
  // an earlier violation stands
  __device__ __forceinline__ void settle_violation(uint64_t vmin) {
    if (!vflag && vmin != kKeyMax) {
      vflag = 1;
      vt = (int64_t)(vmin >> (g.ib + 8));
      vop = (int32_t)((vmin >> 8) & kc.mask);
      vdev = (int32_t)(vmin & 0xffu);
    }
  }

  __device__ void apply_segmented(int m) {
    uint64_t vmin = kKeyMax;
    for (int c0 = 0; c0 < m; c0 += 32) {
      const int idx = c0 + (int)lane_id();
      const bool v = idx < m;
      apply_chunk(v ? sortk[idx] : 0ull, v, vmin);
    }
    settle_violation(vmin);
  }

  // Bitonic sort of 32*E keys held in registers: lane l holds elements
  // l + 32 e.  Pairs 32 or more apart meet inside a lane, closer pairs via
  // shfl_xor.  Fully unrolled.
  template <int E>
  static __device__ __forceinline__ void reg_bitonic(uint64_t (&a)[E]) {
    const int lane = (int)lane_id();
#pragma unroll
    for (int k = 2; k <= 32 * E; k <<= 1) {
#pragma unroll
      for (int j = k >> 1; j > 0; j >>= 1) {
        if (j >= 32) {
#pragma unroll
          for (int e = 0; e < E; ++e) {
            const int e2 = e ^ (j >> 5);
            if (e2 > e) {
              const bool asc = ((lane + 32 * e) & k) == 0;
              const uint64_t x = a[e], y = a[e2];
              const bool sw = asc ? (x > y) : (x < y);
              a[e] = sw ? y : x;
              a[e2] = sw ? x : y;
            }
          }
        } else {
#pragma unroll
          for (int e = 0; e < E; ++e) {
            const uint64_t o = __shfl_xor_sync(kFullMask, a[e], j);
            const bool keep_min = ((lane & j) == 0) == (((lane + 32 * e) & k) == 0);
            a[e] = (keep_min == (o < a[e])) ? o : a[e];
          }
        }
      }
    }
  }

  template <int E>
  __device__ __forceinline__ void sort_apply_regs_e(int m) {
    const int lane = (int)lane_id();
    uint64_t a[E];
#pragma unroll
    for (int e = 0; e < E; ++e) a[e] = lane + 32 * e < m ? sortk[lane + 32 * e] : kKeyMax;
    reg_bitonic<E>(a);
    uint64_t vmin = kKeyMax;
#pragma unroll
    for (int e = 0; e < E; ++e) apply_chunk(a[e], lane + 32 * e < m, vmin);
    settle_violation(vmin);
  }

  // Sort and apply m <= 32 extracted events in registers.  (Wider register
  // networks sort faster but their unrolled code -- each inlining its own
  // copies of the segmented apply -- overflowed the instruction cache: larger
  // drains go through the shared-memory sort.)
  __device__ void sort_apply_regs(int m) { sort_apply_regs_e<1>(m); }

  __device__ int count_below(uint64_t kmax) const {
    int c = 0;
    for (int c0 = 0; c0 < log.n; c0 += 32) {
      const int idx = c0 + (int)lane_id();
      const bool take = idx < log.n && (*log.kp(idx) & lowmask) < kmax;
      c += __popc(__ballot_sync(kFullMask, take));
    }
    return c;
  }

  // Move the logged events whose key part is < kmax to the sort area (their
  // number is known to fit) and compact the rest; returns their number.
  __device__ int extract(uint64_t kmax) {
    const unsigned lane = lane_id();
    const bool side = !kKey;
    int m = 0, keep = 0;
    const int n = log.n;
    for (int c0 = 0; c0 < n; c0 += 32) {
      const int idx = c0 + (int)lane;
      const bool v = idx < n;
      uint64_t e = kKeyMax;
      uint8_t dv8 = 0;
      if (v) {
        if (idx < log.ms) {
          e = log.sk[idx];
          if (side) dv8 = log.sd[idx];
        } else {
          e = *log.kp(idx);
          if (side) dv8 = *log.dp(idx);
        }
      }
      const bool take = v && (e & lowmask) < kmax;
      const uint32_t bt = __ballot_sync(kFullMask, take);
      const uint32_t bk = __ballot_sync(kFullMask, v && !take);
      if (take) {
        const int pos = m + __popc(bt & lanes_below());
        sortk[pos] = e;
        if (side) sortd[pos] = dv8;
      } else if (v) {
        const int pos = keep + __popc(bk & lanes_below());  // pos <= idx: in place
        *log.kp(pos) = e;
        if (side) *log.dp(pos) = dv8;
      }
      m += __popc(bt);
      keep += __popc(bk);
      __syncwarp();
    }
    log.n = keep;
    return m;
  }

  // Bitonic sort of sortk[0, m) (and the side bytes alongside), padded to a
  // power of two >= 32.
  __device__ void sort_area(int m) {
    const unsigned lane = lane_id();
    const bool side = !kKey;
    int p2 = 32;
    while (p2 < m) p2 <<= 1;
    for (int x = m + (int)lane; x < p2; x += 32) sortk[x] = kKeyMax;
    __syncwarp();
    for (int k = 2; k <= p2; k <<= 1) {
      for (int j = k >> 1; j > 0; j >>= 1) {
        for (int t = lane; t < (p2 >> 1); t += 32) {
          const int i = ((t & ~(j - 1)) << 1) | (t & (j - 1));
          const int l = i + j;
          const uint64_t a = sortk[i], b = sortk[l];
          const bool asc = (i & k) == 0;
          if ((a > b) == asc) {
            sortk[i] = b;
            sortk[l] = a;
            if (side) {
              const uint8_t da = sortd[i], db = sortd[l];
              sortd[i] = db;
              sortd[l] = da;
            }
          }
        }
        __syncwarp();
      }
    }
  }

  // Apply every logged event that can no longer be preceded (time < t_next).
  __device__ void drain(int64_t t_next) {
    generate();
    const uint64_t lim = t_next == kI64Max ? kKeyMax : kc.time_floor(t_next);
    while (log.n > 0) {
      uint64_t kmax = lim;
      if (log.n > sortcap) {
        const int due = count_below(lim);
        if (due == 0) break;
        if (due > sortcap) {
          // Rare: more due events than the sort area.  Bisect a key bound
          // with at most sortcap events below it (at most n_dev <= sortcap
          // events share a key part).
          uint64_t lo = kKeyMax;
          for (int c0 = 0; c0 < log.n; c0 += 32) {
            const int idx = c0 + (int)lane_id();
            const uint64_t kk = idx < log.n ? (*log.kp(idx) & lowmask) : kKeyMax;
            lo = kk < lo ? kk : lo;
          }
          lo = warp_min_u64(lo) + 1;  // 1 <= count_below(lo) <= sortcap
          uint64_t hi = lim;          // count_below(hi) > sortcap
          while (hi - lo > 1) {
            const uint64_t mid = lo + (hi - lo) / 2;
            if (count_below(mid) <= sortcap) lo = mid;
            else hi = mid;
          }
          kmax = lo;
        }
      }
      const int m = extract(kmax);
      if (m == 0) break;
      if (kKey && m <= 32) {
        sort_apply_regs(m);
      } else {
        sort_area(m);
        if (kKey) apply_segmented(m);
        else apply_serial(m);
      }
      if (kmax == lim) break;
    }
  }

  __device__ void maybe_checkpoint(uint64_t next_key);

  // The event loop (Sec. 3.3.3).
  __device__ void run() {
    if (status) return;
    if constexpr (kBatch) {
      run_batched();
      return;
    }
    while (true) {
      const uint64_t top = q.top();
      const uint64_t rm = warp_min_u64(rk_reg);
      const uint64_t rk = rkey;
      uint64_t nk = rk < top ? rk : top;
      nk = rm < nk ? rm : nk;
      if (kMode == kBase) maybe_checkpoint(nk);
      if (nk == kKeyMax) break;
      if (opn >= P.opcap) drain(kc.time(nk));
      if (nk == rm) {
        if (rk_reg == rm) rk_reg = kKeyMax;  // keys are unique
      } else if (nk == rk) {
        ++rootptr;
        load_root();
      } else {
        __syncwarp();
        q.pop();
      }
      if (++iters > (int32_t)g.max_iter) {
        status = GMG_SIM_LOOP;
        break;
      }
      const tm_t t = (tm_t)kc.time(nk);
      if (kMode == kBase) last_t = t;
      start_op(kc.op(nk), t);
      if (status) break;
    }
    if (!status) drain(kI64Max);
  }

  // -------------------------------------------------------------------------
  // Batched sweep: the keys are taken in the same order as by run(), but
  // consecutive keys are handled together, one op per lane.  Key k_m joins
  // the batch k_1 < ... < k_{m-1} while time(k_m) < min_l (time(k_l) +
  // 2^class(k_l)).  Every key pushed while handling k_l is at least
  // (f_l, READY, .) with f_l >= r_l + dur_l >= r_l + 2^class(k_l) > r_m, so
  // nothing a batch pushes can precede one of its keys: handling them
  // together, each accelerator's ops in key order, gives the starts of
  // handling them one at a time.  (Many tenants on many accelerators keep
  // about a dozen keys per batch; the dependent loads of a batch's ops then
  // overlap instead of following each other.)
  // -------------------------------------------------------------------------
  __device__ __forceinline__ uint64_t peek(uint64_t& rm) const {
    const uint64_t top = q.top();
    rm = warp_min_u64(rk_reg);
    const uint64_t nk = rkey < top ? rkey : top;
    return rm < nk ? rm : nk;
  }
  __device__ __forceinline__ void take(uint64_t nk, uint64_t rm) {
    if (nk == rm) {
      if (rk_reg == rm) rk_reg = kKeyMax;  // keys are unique
    } else if (nk == rkey) {
      ++rootptr;
      load_root();
    } else {
      __syncwarp();
      q.pop_fast();
    }
  }
  // An op whose inputs several ops of one batch complete is queued once: the
  // first lane to mark its (zero) finish time with -1 queues it.
  __device__ __forceinline__ bool claim(uint32_t j) {
    if (kT32) return atomicCAS(reinterpret_cast<int*>(fbuf + j), 0, -1) == 0;
    return atomicCAS(reinterpret_cast<unsigned long long*>(fbuf + j), 0ull, ~0ull) == 0ull;
  }

  __device__ void run_batched() {
    const unsigned lane = lane_id();
    while (true) {
      uint64_t rm;
      uint64_t nk = peek(rm);
      if (kMode == kBase) maybe_checkpoint(nk);
      if (nk == kKeyMax) break;
      if (opn >= P.drain_trigger) drain(rq.time(nk));
      uint64_t mine = kKeyMax;
      int m = 0;
      int64_t lim = 0;
      while (true) {
        const int64_t t = rq.time(nk);
        const bool from_reg = nk == rm;
        take(nk, rm);
        if ((int)lane == m) mine = nk;
        const int64_t e = t + ((int64_t)1 << rq.q(nk));
        lim = (m == 0 || e < lim) ? e : lim;
        if (kMode == kBase) last_t = (tm_t)t;
        if (++m == 32) break;
        // the register tier's minimum only changes when its key was taken
        if (from_reg) rm = warp_min_u64(rk_reg);
        const uint64_t top = q.top();
        nk = rkey < top ? rkey : top;
        nk = rm < nk ? rm : nk;
        if (nk == kKeyMax || rq.time(nk) >= lim) break;
      }
      iters += m;
      if (iters > (int32_t)g.max_iter) {
        status = GMG_SIM_LOOP;
        break;
      }
      start_batch(mine, m);
      if (status) break;
    }
    if (!status) drain(kI64Max);
  }

  // Start the batch's ops (lane b < m holds key b), record them for HBM-event
  // generation, and queue the successors they make ready.
  __device__ void start_batch(uint64_t key, int m) {
    const unsigned lane = lane_id();
    const bool v = (int)lane < m;
    uint32_t i = 0, succ_off = 0, nsucc = 0, flags = 0;
    int32_t req = 0;
    int d = 0;
    tm_t r = 0, f = 0, dur = 0;
    int64_t bytes = 0, xq = 0;
    if (v) {
      i = rq.op(key);
      r = (tm_t)rq.time(key);
      const longlong2 db = op_durbytes(g.ops, i);
      const XqSucc xs = op_xqsucc(g.ops, i);
      const uint4 cs = op_cons(g.ops, i);
      bytes = db.y;
      xq = xs.xq;
      succ_off = xs.succ_off;
      nsucc = xs.nsucc;
      req = (int32_t)cs.z;
      flags = cs.w;
      d = row[i];
      dur = (tm_t)dur_of(i, d, db.x);
    }
    // every accelerator starts its ops of the batch in key (= lane) order
    bool todo = v;
    while (__any_sync(kFullMask, todo)) {
      const uint32_t grp = __match_any_sync(kFullMask, todo ? (uint32_t)d : 256u + lane);
      if (todo && __ffs(grp) - 1 == (int)lane) {
        const tm_t fd = dv.fr[d];
        const tm_t s = r > fd ? r : fd;
        f = s + dur;
        dv.fr[d] = f;
        todo = false;
      }
      __syncwarp();
    }
    if (v) {
      fbuf[i] = f;
      if (flags & kReqSink)
        atomicMax(reinterpret_cast<unsigned long long*>(creq + req), (unsigned long long)f);
      if (kMode == kBase) P.base.rb[i] = r;
      oplog[opn + (int)lane] = i;
    }
    opn += m;
    score += warp_sum_i64((v && (flags & kScored)) ? (int64_t)f : 0);
    if (kMode == kBase) {
      const tm_t mk = (tm_t)warp_max_u64(v ? (uint64_t)f : 0ull);
      makespan = mk > makespan ? mk : makespan;
      readypops += m;
    }
    if (kMode == kInc) nev += __popc(__ballot_sync(kFullMask, v && r >= T0));
    __syncwarp();
    // successors: ready once every predecessor has started; ready time = the
    // latest arrival over all of them (Sec. 3.3.2)
    const uint32_t maxs = __reduce_max_sync(kFullMask, nsucc);
    for (uint32_t u = 0; u < maxs; ++u) {
      uint32_t j = 0, qj = 0;
      tm_t rj = 0;
      bool rdy = false;
      if (u < nsucc) {
        j = __ldg(g.succ + succ_off + u);
        const int dj = row[j];
        tm_t arr = f;
        if (dj != d) arr = f + xfer(d, dj, bytes, xq);
        const RelPred jp = op_relpred(g.ops, j);
        qj = dur_class(dur_of(j, dj, op_durbytes(g.ops, j).x));
        const tm_t rel = (tm_t)jp.rel;
        rj = rel > arr ? rel : arr;
        rdy = true;
        if (jp.npred > 1) {
          for (uint32_t k = 0; k < jp.npred; ++k) {
            const uint32_t p = __ldg(g.pred + jp.pred_off + k) & kIdMask;
            if (p == i) continue;
            tm_t a = fin(p);
            if (a <= 0) {  // not started yet
              rdy = false;
              break;
            }
            const int dp = row[p];
            if (dp != dj) a += xfer(dp, dj, op_durbytes(g.ops, p).y, op_xqsucc(g.ops, p).xq);
            rj = a > rj ? a : rj;
          }
          if (rdy) rdy = claim(j);
        }
      }
      uint32_t bm = __ballot_sync(kFullMask, rdy);
      while (bm) {
        const int src = __ffs(bm) - 1;
        bm &= bm - 1;
        push_ready(__shfl_sync(kFullMask, rq.make(rj, j, qj), src));
      }
    }
  }

  __device__ void write_invalid(int64_t k, int32_t st) {
    const DevOut& o = P.out;
    const unsigned lane = lane_id();
    if (lane == 0) {
      o.makespan[k] = 0;
      o.score[k] = kI64Max;
      o.status[k] = st;
      o.viol_flag[k] = 0;
      o.viol_op[k] = -1;
      o.viol_dev[k] = -1;
      o.viol_time[k] = -1;
      o.sla_miss[k] = 0;
      o.events[k] = 0;
    }
    for (int d = lane; d < g.D; d += 32) o.peak[k * g.D + d] = 0;
    if (o.req_done)
      for (int r = lane; r < g.R; r += 32) o.req_done[k * g.R + r] = 0;
    const int ts = trace_slot(k);
    if (ts >= 0)
      for (int x = lane; x < g.n; x += 32) {
        o.trace_start[(int64_t)ts * g.n + x] = 0;
        o.trace_finish[(int64_t)ts * g.n + x] = 0;
      }
  }

  __device__ int trace_slot(int64_t k) const {
    if (P.n_trace == 0) return -1;
    int ts = -1;
    for (int t = lane_id(); t < P.n_trace; t += 32)
      if (P.trace_k[t] == k) ts = t;
    return __reduce_max_sync(kFullMask, ts);
  }

  __device__ void finish(int64_t k) {
    if (status != GMG_SIM_OK) {
      write_invalid(k, status);
      return;
    }
    const DevOut& o = P.out;
    const unsigned lane = lane_id();
    int32_t miss = 0;
    for (int r = lane; r < g.R; r += 32) {
      const int64_t c = creq[r];
      miss += c > __ldg(g.deadline + r) ? 1 : 0;
      if (o.req_done) o.req_done[k * g.R + r] = c;
    }
    miss = (int32_t)__reduce_add_sync(kFullMask, (unsigned)miss);
    dv.write_peak(o.peak + k * g.D);
    // The makespan is the latest finish, i.e. the largest final free time over
    // the accelerators that ran an op (an op finishes after its accelerator's
    // initial availability).
    const int64_t mk = dv.max_busy(g);
    if (lane == 0) {
      o.makespan[k] = mk;
      o.score[k] = vflag ? kI64Max : score;
      o.status[k] = GMG_SIM_OK;
      o.viol_flag[k] = vflag;
      o.viol_op[k] = vop;
      o.viol_dev[k] = vdev;
      o.viol_time[k] = vt;
      o.sla_miss[k] = miss;
      o.events[k] = kMode == kFull ? (int64_t)iters : nev;
    }
    const int ts = trace_slot(k);
    if (ts >= 0)
      for (int x = lane; x < g.n; x += 32) {
        const int64_t fx = (int64_t)fin((uint32_t)x);
        o.trace_finish[(int64_t)ts * g.n + x] = fx;
        o.trace_start[(int64_t)ts * g.n + x] = fx - dur_of((uint32_t)x, row[x], op_durbytes(g.ops, (uint32_t)x).x);
      }
  }

  // Any placement byte >= D?  (16-byte coalesced loads of the row.)
  __device__ bool row_has_bad_device(const uint8_t* rw) const {
    if (g.D >= 256) return false;
    const unsigned lane = lane_id();
    const uint32_t dd = (uint32_t)g.D * 0x01010101u;
    bool bad = false;
    for (int c = lane * 16; c < g.n; c += 512) {
      const uint4 v = *reinterpret_cast<const uint4*>(rw + c);
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        uint32_t ge = __vcmpgeu4(w[h], dd);
        const int first = c + 4 * h;
        if (first + 4 > g.n) {
          const int keep = g.n - first;  // bytes of this word inside the row
          ge = keep <= 0 ? 0u : (ge & (0xffffffffu >> (8 * (4 - keep))));
        }
        bad |= ge != 0u;
      }
    }
    return __any_sync(kFullMask, bad);
  }
};

// Base-mode checkpoint: at a time boundary T_c (nothing at the next key's
// time handled yet), save the complete simulator state -- accelerator state,
// READY heap, event log, partial results; the ops started by then are those
// with base ready time < T_c.  An incremental candidate whose resume time T0
// is >= T_c restarts there.
template <bool kReg, int kMode, bool kKey, bool kT32, bool kTypes, bool kBatch, bool kStage>
__device__ void Sim<kReg, kMode, kKey, kT32, kTypes, kBatch, kStage>::maybe_checkpoint(uint64_t next_key) {
  if (kMode != kBase) return;
  const DevBase& B = P.base;
  if (next_key == kKeyMax || ck >= B.nck || readypops < next_ck) return;
  const int64_t tn = rq.time(next_key);
  if (tn <= last_t) return;
  const unsigned lane = lane_id();
  generate();
  const bool hasreg = rk_reg != kKeyMax;
  const uint32_t regm = __ballot_sync(kFullMask, hasreg);
  const int nready = q.size + __popc(regm);
  if (nready <= B.ckq && log.n <= B.ckm) {
    int64_t* sc = B.ck_scalars + (int64_t)ck * 8;
    if (hasreg) B.ck_qkey[(int64_t)ck * B.ckq + q.size + __popc(regm & lanes_below())] = rk_reg;
    if (lane == 0) {
      B.ck_time[ck] = tn;
      sc[0] = nready;
      sc[1] = rootptr;
      sc[2] = score;
      sc[3] = makespan;
      sc[4] = vflag;
      sc[5] = vt;
      sc[6] = ((int64_t)vop << 32) | (uint32_t)vdev;
      sc[7] = log.n;
    }
    dv.save(B.ck_dev + (int64_t)ck * 3 * g.D);
    for (int r = lane; r < g.R; r += 32) B.ck_creq[(int64_t)ck * g.R + r] = creq[r];
    for (int x = lane; x < q.size; x += 32) B.ck_qkey[(int64_t)ck * B.ckq + x] = *q.kp(x);
    for (int x = lane; x < log.n; x += 32) {
      B.ck_mkey[(int64_t)ck * B.ckm + x] = *log.kp(x);
      if (!kKey) B.ck_mdev[(int64_t)ck * B.ckm + x] = *log.dp(x);
    }
  } else if (lane == 0) {
    B.ck_time[ck] = kI64Max;
  }
  ++ck;
  next_ck += B.stride_pops;
  __syncwarp();
}

template <bool kReg, int kMode, bool kKey, bool kT32, bool kTypes, bool kBatch, bool kStage>
__device__ void setup_slot(Sim<kReg, kMode, kKey, kT32, kTypes, kBatch, kStage>& S, const SimParams& P, unsigned wib,
                           int64_t slot, uint8_t* smem) {
  uint8_t* sl = P.scratch + slot * P.slot_bytes;
  const WarpSmem w = carve_smem(smem, P, wib);
  S.q.sk = w.heap;
  S.q.gk = reinterpret_cast<uint64_t*>(sl + P.off_qk);
  S.q.qs = P.qs;
  S.q.cap = P.qcap;
  S.q.size = 0;
  S.log.sk = w.logk;
  S.log.sd = w.logd;
  S.log.gk = reinterpret_cast<uint64_t*>(sl + P.off_mk);
  S.log.gd = sl + P.off_md;
  S.log.ms = P.ms;
  S.log.cap = P.mcap;
  S.log.n = 0;
  S.sortk = w.sortk;
  S.sortd = w.sortd;
  S.oplog = w.oplog;
  S.opn = 0;
  S.sortcap = P.sortcap;
  using tm_t = typename Sim<kReg, kMode, kKey, kT32, kTypes, kBatch, kStage>::tm_t;
  S.fbuf = reinterpret_cast<tm_t*>(sl + P.off_f);
  S.holdb = reinterpret_cast<tm_t*>(sl + P.off_hold);
  S.bits = reinterpret_cast<uint32_t*>(sl + P.off_bits);
  S.creq = reinterpret_cast<int64_t*>(sl + P.off_creq);
  S.dv.setup(P.g, w.dev, P.off_pk >= 0 ? reinterpret_cast<int64_t*>(sl + P.off_pk) : nullptr);
  S.T0 = -1;
  S.Tc = 0;
}

}  // namespace
}  // namespace gsim
