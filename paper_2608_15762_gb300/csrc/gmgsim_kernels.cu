// sm_103a kernels of the what-if placement simulator.
//
// One warp simulates one candidate placement (Algorithm 1 evaluates the
// candidate partitions "in parallel"; here every warp of a persistent grid
// takes candidates k = warp, warp + W, ...).  Inside a warp the simulation
// is the event-driven loop of Sec. 3.3.3, restated as one ordered sweep over
// packed 64-bit event keys (time, class, op):
//
//   READY(r_i, i)  op i's last input has arrived (Sec. 3.3.2 ready time);
//                  popping it starts i on its accelerator at
//                  s_i = max(r_i, accelerator free time): every queue runs its
//                  ops in (ready time, id) order, one at a time (Sec. 3.3.2,
//                  Sec. 3.5.1), which is exactly "an idle queue starts the
//                  ready op with the earliest ready time".
//   FREE(t, i)@e   a copy of i's output on accelerator e is released.
//   ALLOC(t, i)@e  a copy of i's output is allocated on e (its own output at
//                  s_i; a receive buffer at f_i, Recv before Send, Sec. 3.5.2).
//
// Every key pushed while handling key k is larger than k (successors are
// ready no earlier than f_i > r_i, memory events happen at >= s_i with a
// larger class), so the queue is monotone and memory events come out in
// (time, frees-before-allocs, op) order: live bytes, per-accelerator peaks and
// the first capacity violation (Sec. 3.3.2 HBM residency, Sec. 3.4.2 OOM
// discard) are tracked online, with no sort.
//
// The queue is a 32-ary min-heap whose 32 children of a node are examined by
// the 32 lanes at once (one coalesced load + two redux.sync), so a pop costs
// log32(size) warp steps.  Its first `qs` entries live in shared memory, the
// rest in the warp's global scratch.  Ops without predecessors never enter
// the heap: their READY keys are pre-sorted on the host and merged in.
//
// Lanes also fan out over successor lists (readiness, transfer arrivals,
// distinct receiving accelerators via __match_any_sync), predecessor lists
// (ready-time maxima) and consumer lists (last-consumer releases).  With at
// most 32 accelerators, lane d keeps accelerator d's free time, live bytes
// and peak in registers.
//
// No wait in these kernels depends on another warp or block; the only loop
// without a data-bounded trip count is the event loop, capped at
// g.max_iter iterations (status GMG_SIM_LOOP).

#include <cuda_runtime.h>
#include <stdint.h>

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

// 16-byte pieces of an OpRec, loaded through the read-only path.
__device__ __forceinline__ longlong2 op_durbytes(const OpRec* ops, uint32_t i) {
  return __ldg(reinterpret_cast<const longlong2*>(ops + i));
}
__device__ __forceinline__ longlong2 op_relxq(const OpRec* ops, uint32_t i) {
  return __ldg(reinterpret_cast<const longlong2*>(ops + i) + 1);
}
__device__ __forceinline__ uint4 op_lists(const OpRec* ops, uint32_t i) {
  return __ldg(reinterpret_cast<const uint4*>(ops + i) + 2);  // succ_off, nsucc, pred_off, npred
}
__device__ __forceinline__ uint4 op_cons(const OpRec* ops, uint32_t i) {
  return __ldg(reinterpret_cast<const uint4*>(ops + i) + 3);  // cons_off, ncons, req, flags
}

struct KeyCodec {
  int ib;
  uint64_t mask;
  __device__ __forceinline__ uint64_t make(int64_t t, uint32_t cls, uint32_t op) const {
    return ((uint64_t)t << (ib + 2)) | ((uint64_t)cls << ib) | (uint64_t)op;
  }
  __device__ __forceinline__ int64_t time(uint64_t k) const { return (int64_t)(k >> (ib + 2)); }
  __device__ __forceinline__ uint32_t cls(uint64_t k) const { return (uint32_t)(k >> ib) & 3u; }
  __device__ __forceinline__ uint32_t op(uint64_t k) const { return (uint32_t)(k & mask); }
};

// ---------------------------------------------------------------------------
// Warp-cooperative 32-ary min-heap.  All lanes call every method with the
// same arguments; lane 0 performs the stores.
// ---------------------------------------------------------------------------
struct WarpHeap {
  uint64_t* sk;  // shared: keys [qs]
  uint32_t* sp;  // shared: payloads [qs]
  uint64_t* gk;  // global spill: keys [cap - qs]
  uint32_t* gp;  // global spill: payloads
  int qs, cap, size;

  __device__ __forceinline__ uint64_t* kp(int i) const { return i < qs ? sk + i : gk + (i - qs); }
  __device__ __forceinline__ uint32_t* pp(int i) const { return i < qs ? sp + i : gp + (i - qs); }

  // Place (x, xp) at `pos` and move it down until its children are >= x.
  __device__ void sift_down(int pos, uint64_t x, uint32_t xp) {
    const unsigned lane = lane_id();
    while (true) {
      const int c0 = pos * 32 + 1;
      if (c0 >= size) break;
      const int idx = c0 + (int)lane;
      const uint64_t ck = idx < size ? *kp(idx) : kKeyMax;
      const uint64_t m = warp_min_u64(ck);
      if (m >= x) break;
      const int src = __ffs(__ballot_sync(kFullMask, ck == m)) - 1;
      uint32_t mp = 0;
      if ((int)lane == src) mp = *pp(idx);
      mp = __shfl_sync(kFullMask, mp, src);
      if (lane == 0) {
        *kp(pos) = m;
        *pp(pos) = mp;
      }
      pos = c0 + src;
    }
    if (lane == 0) {
      *kp(pos) = x;
      *pp(pos) = xp;
    }
    __syncwarp();
  }

  // Remove the minimum (the caller has read it).
  __device__ void pop() {
    const int n = --size;
    if (n == 0) return;
    const uint64_t x = *kp(n);
    const uint32_t xp = *pp(n);
    sift_down(0, x, xp);
  }

  __device__ bool push(uint64_t key, uint32_t pay) {
    if (size >= cap) return false;
    const unsigned lane = lane_id();
    int pos = size++;
    while (pos > 0) {
      const int par = (pos - 1) >> 5;
      const uint64_t pk = *kp(par);
      if (pk <= key) break;
      const uint32_t ppay = *pp(par);
      if (lane == 0) {
        *kp(pos) = pk;
        *pp(pos) = ppay;
      }
      pos = par;
    }
    if (lane == 0) {
      *kp(pos) = key;
      *pp(pos) = pay;
    }
    __syncwarp();
    return true;
  }

  // Append without ordering (followed by heapify()).
  __device__ bool append(uint64_t key, uint32_t pay) {
    if (size >= cap) return false;
    if (lane_id() == 0) {
      *kp(size) = key;
      *pp(size) = pay;
    }
    ++size;
    __syncwarp();
    return true;
  }

  // Floyd's bottom-up construction.
  __device__ void heapify() {
    if (size < 2) return;
    for (int pos = (size - 2) / 32; pos >= 0; --pos) {
      const uint64_t x = *kp(pos);
      const uint32_t xp = *pp(pos);
      __syncwarp();
      sift_down(pos, x, xp);
    }
  }
};

// ---------------------------------------------------------------------------
// Per-accelerator state: free time, live bytes, peak bytes.
// ---------------------------------------------------------------------------
template <bool kReg>
struct Devices;

// D <= 32: lane d holds accelerator d in registers.
template <>
struct Devices<true> {
  int64_t fr, lv, pk, cp;
  int D;
  __device__ void setup(const DevGmg& g, int64_t* /*mem*/) {
    D = g.D;
    cp = lane_id() < (unsigned)D ? g.cap[lane_id()] : kI64Max;
  }
  __device__ void reset(const DevGmg& g) {
    const unsigned l = lane_id();
    fr = l < (unsigned)D ? g.avail0[l] : 0;
    lv = l < (unsigned)D ? g.base[l] : 0;
    pk = lv;
  }
  __device__ __forceinline__ int64_t get_free(int d) const { return __shfl_sync(kFullMask, fr, d); }
  __device__ __forceinline__ void set_free(int d, int64_t v) {
    if ((int)lane_id() == d) fr = v;
  }
  __device__ __forceinline__ bool alloc(int d, int64_t b) {
    bool over = false;
    if ((int)lane_id() == d) {
      lv += b;
      pk = lv > pk ? lv : pk;
      over = lv > cp;
    }
    return __ballot_sync(kFullMask, over) != 0;
  }
  __device__ __forceinline__ void release(int d, int64_t b) {
    if ((int)lane_id() == d) lv -= b;
  }
  __device__ void save(int64_t* dst) const {
    const unsigned l = lane_id();
    if (l < (unsigned)D) {
      dst[l] = fr;
      dst[D + l] = lv;
      dst[2 * D + l] = pk;
    }
  }
  __device__ void load(const int64_t* src) {
    const unsigned l = lane_id();
    if (l < (unsigned)D) {
      fr = src[l];
      lv = src[D + l];
      pk = src[2 * D + l];
    }
  }
  __device__ void write_peak(int64_t* dst) const {
    if (lane_id() < (unsigned)D) dst[lane_id()] = pk;
  }
};

// Any D: arrays in the warp's scratch; all lanes read, lane 0 writes.
template <>
struct Devices<false> {
  int64_t* fr;
  int64_t* lv;
  int64_t* pk;
  const int64_t* cp;
  int D;
  __device__ void setup(const DevGmg& g, int64_t* mem) {
    D = g.D;
    fr = mem;
    lv = mem + D;
    pk = mem + 2 * D;
    cp = g.cap;
  }
  __device__ void reset(const DevGmg& g) {
    for (int d = lane_id(); d < D; d += 32) {
      fr[d] = g.avail0[d];
      lv[d] = g.base[d];
      pk[d] = g.base[d];
    }
    __syncwarp();
  }
  __device__ __forceinline__ int64_t get_free(int d) const { return fr[d]; }
  __device__ __forceinline__ void set_free(int d, int64_t v) {
    if (lane_id() == 0) fr[d] = v;
  }
  __device__ __forceinline__ bool alloc(int d, int64_t b) {
    const int64_t v = lv[d] + b;
    const int64_t p = pk[d];
    if (lane_id() == 0) {
      lv[d] = v;
      if (v > p) pk[d] = v;
    }
    return v > __ldg(cp + d);
  }
  __device__ __forceinline__ void release(int d, int64_t b) {
    const int64_t v = lv[d] - b;
    if (lane_id() == 0) lv[d] = v;
  }
  __device__ void save(int64_t* dst) const {
    for (int d = lane_id(); d < D; d += 32) {
      dst[d] = fr[d];
      dst[D + d] = lv[d];
      dst[2 * D + d] = pk[d];
    }
  }
  __device__ void load(const int64_t* src) {
    for (int d = lane_id(); d < D; d += 32) {
      fr[d] = src[d];
      lv[d] = src[D + d];
      pk[d] = src[2 * D + d];
    }
    __syncwarp();
  }
  __device__ void write_peak(int64_t* dst) const {
    for (int d = lane_id(); d < D; d += 32) dst[d] = pk[d];
  }
};

// ---------------------------------------------------------------------------
// One warp's simulator.
// ---------------------------------------------------------------------------
template <bool kReg, int kMode>
struct Sim {
  const SimParams& P;
  const DevGmg& g;
  KeyCodec kc;
  WarpHeap q;
  Devices<kReg> dv;
  const uint8_t* row;
  int64_t* fbuf;
  uint32_t* bits;
  int64_t* creq;
  // incremental resume
  const int64_t* rb;
  const int64_t* fb;
  const uint8_t* brow;
  int64_t Tc, T0;
  // running results
  int rootptr;
  int64_t score, makespan, iters, nev, readypops, last_t;
  int32_t vflag, vop, vdev, status;
  int64_t vt;
  // base checkpoints
  int ck, next_ck;

  __device__ Sim(const SimParams& p) : P(p), g(p.g) {
    kc.ib = g.ib;
    kc.mask = (1ull << g.ib) - 1ull;
  }

  __device__ __forceinline__ bool bit(uint32_t x) const { return (bits[x >> 5] >> (x & 31u)) & 1u; }

  // Has op x been simulated (is its finish time known)?
  __device__ __forceinline__ bool popped(uint32_t x) const {
    if (kMode == kInc) return bit(x) || rb[x] < Tc;
    return bit(x);
  }
  __device__ __forceinline__ int64_t fin(uint32_t x) const {
    if (kMode == kInc && !bit(x)) return fb[x];
    return fbuf[x];
  }

  // Transfer estimator of one output over link d -> e (d != e), Sec. 3.3.1.
  __device__ __forceinline__ int64_t xfer(int d, int e, int64_t bytes, int64_t xq) const {
    if (g.uniform) return xq + g.lat0;
    const LinkRec* L = g.links + (d * g.D + e);
    LinkRec l;
    const longlong2 a = __ldg(reinterpret_cast<const longlong2*>(L));
    const longlong2 b = __ldg(reinterpret_cast<const longlong2*>(L) + 1);
    l.magic = (uint64_t)a.x;
    l.bw = a.y;
    l.lat = b.x;
    l.shift = (int32_t)(b.y & 0xffffffff);
    return ceil_div_link(bytes, l) + l.lat;
  }

  __device__ __forceinline__ void push(uint64_t key, uint32_t pay) {
    if (status) return;
    if (!q.push(key, pay)) status = GMG_SIM_QUEUE;
  }
  __device__ __forceinline__ void append(uint64_t key, uint32_t pay) {
    if (status) return;
    if (!q.append(key, pay)) status = GMG_SIM_QUEUE;
  }

  // Push (key, pay) of every lane in `mask`, in lane order.
  template <bool kAppend>
  __device__ __forceinline__ void push_lanes(uint32_t mask, uint64_t key, uint32_t pay) {
    while (mask) {
      const int src = __ffs(mask) - 1;
      mask &= mask - 1;
      const uint64_t k = __shfl_sync(kFullMask, key, src);
      const uint32_t p = __shfl_sync(kFullMask, pay, src);
      if (kAppend) append(k, p);
      else push(k, p);
    }
  }

  __device__ void reset_common() {
    const unsigned lane = lane_id();
    const int words = (g.n + 31) >> 5;
    for (int w = lane; w < words; w += 32) bits[w] = 0u;
    for (int r = lane; r < g.R; r += 32) creq[r] = 0;
    dv.reset(g);
    q.size = 0;
    rootptr = 0;
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
  // READY(r, i): start op i (Sec. 3.3.2/3.3.3) and emit what follows from it.
  // -------------------------------------------------------------------------
  __device__ void start_op(uint32_t i, int64_t r) {
    const unsigned lane = lane_id();
    const longlong2 db = op_durbytes(g.ops, i);
    const longlong2 rx = op_relxq(g.ops, i);
    const uint4 ls = op_lists(g.ops, i);
    const uint4 cs = op_cons(g.ops, i);
    const int64_t dur = db.x, bytes = db.y, xq = rx.y;
    const uint32_t succ_off = ls.x, nsucc = ls.y, pred_off = ls.z, npred = ls.w;
    const uint32_t cons_off = cs.x, ncons = cs.y, flags = cs.w;
    const int d = row[i];
    const int64_t fd = dv.get_free(d);
    const int64_t s = r > fd ? r : fd;
    const int64_t f = s + dur;
    dv.set_free(d, f);
    if (lane == 0) {
      fbuf[i] = f;
      atomicOr(&bits[i >> 5], 1u << (i & 31u));
      if (flags & kReqSink)
        atomicMax(reinterpret_cast<unsigned long long*>(creq + (int32_t)cs.z), (unsigned long long)f);
      if (kMode == kBase) P.base.rb[i] = r;
    }
    if (flags & kScored) score += f;
    makespan = f > makespan ? f : makespan;
    if (kMode != kInc || r >= T0) ++nev;
    ++readypops;
    __syncwarp();

    // The op's own output is allocated when it starts.
    push(kc.make(s, kAlloc, i), (uint32_t)d);

    // Successors: transfers, readiness, receive copies.
    int64_t hold = f;   // latest arrival of an outgoing transfer (or f)
    bool local_succ = false;
    for (uint32_t c0 = 0; c0 < nsucc; c0 += 32) {
      const uint32_t t = c0 + lane;
      const bool v = t < nsucc;
      uint32_t j = 0;
      int dj = -1;
      int64_t arr = f, rj = 0;
      bool rdy = false;
      if (v) {
        j = __ldg(g.succ + succ_off + t);
        dj = row[j];
        if (dj != d) arr = f + xfer(d, dj, bytes, xq);
        const longlong2 jrx = op_relxq(g.ops, j);
        const uint4 jls = op_lists(g.ops, j);
        rj = jrx.x > arr ? jrx.x : arr;
        rdy = true;
        if (jls.w > 1) {
          // Ready only when every other predecessor has finished; its ready
          // time is the latest arrival over all of them.
          for (uint32_t k = 0; k < jls.w; ++k) {
            const uint32_t p = __ldg(g.pred + jls.z + k) & kIdMask;
            if (p == i) continue;
            if (!popped(p)) {
              rdy = false;
              break;
            }
            const int dp = row[p];
            int64_t a = fin(p);
            if (dp != dj) {
              const longlong2 pdb = op_durbytes(g.ops, p);
              a += xfer(dp, dj, pdb.y, op_relxq(g.ops, p).y);
            }
            rj = a > rj ? a : rj;
          }
        }
      }
      push_lanes<false>(__ballot_sync(kFullMask, rdy), kc.make(rj, kReady, j), 0u);

      const bool rem = v && dj != d;
      local_succ |= __any_sync(kFullMask, v && dj == d);
      const uint32_t peers = __match_any_sync(kFullMask, rem ? (uint32_t)dj : (256u + lane));
      bool leader = rem && (__ffs(peers) - 1 == (int)lane);
      if (leader && c0 > 0) {
        for (uint32_t u = 0; u < c0; ++u)
          if (row[__ldg(g.succ + succ_off + u)] == dj) {
            leader = false;
            break;
          }
      }
      const uint64_t hm = warp_max_u64(leader ? (uint64_t)arr : 0ull);
      hold = (int64_t)hm > hold ? (int64_t)hm : hold;
      // One receive copy per distinct remote accelerator, allocated when the
      // transfer starts.
      const uint32_t lead_mask = __ballot_sync(kFullMask, leader);
      push_lanes<false>(lead_mask, kc.make(f, kAlloc, i), (uint32_t)dj);
      if (!(flags & kAllCons)) {
        // A receive copy with no listed consumer there is released on arrival.
        bool nocons = false;
        if (leader) {
          nocons = true;
          for (uint32_t u = 0; u < ncons; ++u)
            if (row[__ldg(g.cons + cons_off + u)] == dj) {
              nocons = false;
              break;
            }
        }
        push_lanes<false>(__ballot_sync(kFullMask, nocons), kc.make(arr, kFree, i), (uint32_t)dj);
      }
    }
    // The source copy: released by its last local consumer, or now-known.
    bool local_cons = local_succ;
    if (!(flags & kAllCons)) {
      bool lc = false;
      for (uint32_t c0 = 0; c0 < ncons; c0 += 32) {
        const uint32_t t = c0 + lane;
        if (t < ncons && row[__ldg(g.cons + cons_off + t)] == d) lc = true;
      }
      local_cons = __any_sync(kFullMask, lc);
    }
    if (!local_cons) push(kc.make(hold, kFree, i), (uint32_t)d);

    // Inputs this op holds: if it is the last listed consumer of a
    // predecessor's output on this accelerator, that copy is released at f
    // (the source copy also waits for the predecessor's outgoing arrivals).
    for (uint32_t k = 0; k < npred; ++k) {
      const uint32_t pe = __ldg(g.pred + pred_off + k);
      if (!(pe & kHoldBit)) continue;
      const uint32_t p = pe & kIdMask;
      const uint4 pls = op_lists(g.ops, p);
      const uint4 pcs = op_cons(g.ops, p);
      const bool all = (pcs.w & kAllCons) != 0;
      const uint32_t* lst = all ? g.succ + pls.x : g.cons + pcs.x;
      const uint32_t nl = all ? pls.y : pcs.y;
      bool pending = false;
      for (uint32_t c0 = 0; c0 < nl; c0 += 32) {
        const uint32_t t = c0 + lane;
        if (t < nl) {
          const uint32_t c = __ldg(lst + t);
          if (c != i && row[c] == d && !popped(c)) pending = true;
        }
      }
      if (__any_sync(kFullMask, pending)) continue;
      const int dp = row[p];
      int64_t T = f;
      if (dp == d) {
        const int64_t fp = fin(p);
        const int64_t pb = op_durbytes(g.ops, p).y;
        const int64_t pxq = op_relxq(g.ops, p).y;
        uint64_t mx = 0;
        for (uint32_t c0 = 0; c0 < pls.y; c0 += 32) {
          const uint32_t t = c0 + lane;
          if (t < pls.y) {
            const int du = row[__ldg(g.succ + pls.x + t)];
            if (du != dp) {
              const uint64_t a = (uint64_t)(fp + xfer(dp, du, pb, pxq));
              mx = a > mx ? a : mx;
            }
          }
        }
        const int64_t m = (int64_t)warp_max_u64(mx);
        T = m > T ? m : T;
      }
      push(kc.make(T, kFree, p), (uint32_t)d);
    }
  }

  __device__ __forceinline__ void mem_event(uint32_t cls, uint32_t op, int64_t t, uint32_t pay) {
    const int e = (int)(pay & 0xffu);
    const int64_t b = op_durbytes(g.ops, op).y;
    if (cls == kFree) {
      dv.release(e, b);
    } else if (dv.alloc(e, b)) {
      if (!vflag || (t == vt && (int32_t)op == vop && e < vdev)) {
        vflag = 1;
        vt = t;
        vop = (int32_t)op;
        vdev = e;
      }
    }
  }

  __device__ void maybe_checkpoint(uint64_t next_key);

  // The event loop (Sec. 3.3.3).
  __device__ void run() {
    if (status) return;
    while (true) {
      const uint64_t top = q.size > 0 ? *q.kp(0) : kKeyMax;
      const uint64_t rk = rootptr < g.nroots ? __ldg(g.root_keys + rootptr) : kKeyMax;
      if (kMode == kBase) maybe_checkpoint(rk < top ? rk : top);
      uint64_t key;
      uint32_t pay = 0;
      if (rk < top) {
        key = rk;
        ++rootptr;
      } else if (top != kKeyMax) {
        key = top;
        pay = *q.pp(0);
        __syncwarp();
        q.pop();
      } else {
        break;
      }
      if (++iters > g.max_iter) {
        status = GMG_SIM_LOOP;
        break;
      }
      const uint32_t cls = kc.cls(key), op = kc.op(key);
      const int64_t t = kc.time(key);
      last_t = t;
      if (cls == kReady) start_op(op, t);
      else mem_event(cls, op, t, pay);
      __syncwarp();
      if (status) break;
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
    if (lane == 0) {
      o.makespan[k] = makespan;
      o.score[k] = vflag ? kI64Max : score;
      o.status[k] = GMG_SIM_OK;
      o.viol_flag[k] = vflag;
      o.viol_op[k] = vop;
      o.viol_dev[k] = vdev;
      o.viol_time[k] = vt;
      o.sla_miss[k] = miss;
      o.events[k] = nev;
    }
    const int ts = trace_slot(k);
    if (ts >= 0)
      for (int x = lane; x < g.n; x += 32) {
        const int64_t fx = fin((uint32_t)x);
        o.trace_finish[(int64_t)ts * g.n + x] = fx;
        o.trace_start[(int64_t)ts * g.n + x] = fx - op_durbytes(g.ops, (uint32_t)x).x;
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

// Base-mode checkpoint: at a time boundary (nothing at the next key's time
// processed yet), save the complete simulator state; an incremental
// candidate whose resume time T0 is >= that time may restart from it.
template <bool kReg, int kMode>
__device__ void Sim<kReg, kMode>::maybe_checkpoint(uint64_t next_key) {
  if (kMode != kBase) return;
  const DevBase& B = P.base;
  if (next_key == kKeyMax || ck >= B.nck || readypops < next_ck) return;
  const int64_t tn = kc.time(next_key);
  if (tn <= last_t) return;
  const unsigned lane = lane_id();
  if (q.size <= B.ckq) {
    int64_t* sc = B.ck_scalars + (int64_t)ck * 8;
    if (lane == 0) {
      B.ck_time[ck] = tn;
      sc[0] = q.size;
      sc[1] = rootptr;
      sc[2] = score;
      sc[3] = makespan;
      sc[4] = vflag;
      sc[5] = vt;
      sc[6] = vop;
      sc[7] = vdev;
    }
    dv.save(B.ck_dev + (int64_t)ck * 3 * g.D);
    for (int r = lane; r < g.R; r += 32) B.ck_creq[(int64_t)ck * g.R + r] = creq[r];
    for (int x = lane; x < q.size; x += 32) {
      B.ck_qkey[(int64_t)ck * B.ckq + x] = *q.kp(x);
      B.ck_qpay[(int64_t)ck * B.ckq + x] = *q.pp(x);
    }
  } else if (lane == 0) {
    B.ck_time[ck] = kI64Max;
  }
  ++ck;
  next_ck += B.stride_pops;
  __syncwarp();
}

template <bool kReg, int kMode>
__device__ void setup_slot(Sim<kReg, kMode>& S, const SimParams& P, unsigned warp_in_block,
                           int64_t slot, uint8_t* smem) {
  uint8_t* sl = P.scratch + slot * P.slot_bytes;
  S.q.sk = reinterpret_cast<uint64_t*>(smem) + (int64_t)warp_in_block * P.qs;
  S.q.sp = reinterpret_cast<uint32_t*>(smem + (size_t)blockDim.x / 32 * P.qs * 8) +
           (int64_t)warp_in_block * P.qs;
  S.q.gk = reinterpret_cast<uint64_t*>(sl + P.off_qk);
  S.q.gp = reinterpret_cast<uint32_t*>(sl + P.off_qp);
  S.q.qs = P.qs;
  S.q.cap = P.qcap;
  S.q.size = 0;
  S.fbuf = reinterpret_cast<int64_t*>(sl + P.off_f);
  S.bits = reinterpret_cast<uint32_t*>(sl + P.off_bits);
  S.creq = reinterpret_cast<int64_t*>(sl + P.off_creq);
  S.dv.setup(P.g, reinterpret_cast<int64_t*>(sl + P.off_dev));
  S.T0 = -1;
  S.Tc = 0;
}

// ---------------------------------------------------------------------------
// sim_batch: K full placements.
// ---------------------------------------------------------------------------
template <bool kReg>
__global__ void __launch_bounds__(128) sim_full_kernel(const __grid_constant__ SimParams P) {
  extern __shared__ __align__(16) uint8_t smem[];
  const unsigned wib = threadIdx.x >> 5;
  const int64_t slot = (int64_t)blockIdx.x * (blockDim.x >> 5) + wib;
  const int64_t nslots = (int64_t)gridDim.x * (blockDim.x >> 5);
  Sim<kReg, kFull> S(P);
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
// base_create: simulate the base placement once, recording resume points.
// ---------------------------------------------------------------------------
template <bool kReg>
__global__ void __launch_bounds__(32) sim_base_kernel(const __grid_constant__ SimParams P) {
  extern __shared__ __align__(16) uint8_t smem[];
  Sim<kReg, kBase> S(P);
  setup_slot(S, P, 0, 0, smem);
  const DevBase& B = P.base;
  const unsigned lane = lane_id();
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
  S.last_t = -1;
  // checkpoint 0: the initial state, valid for every resume time >= 0
  S.maybe_checkpoint(S.kc.make(0, kReady, 0));
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
// sim_incremental: K move lists against the base.
// ---------------------------------------------------------------------------
template <bool kReg>
__device__ void regen(Sim<kReg, kInc>& S, uint32_t p);

template <bool kReg>
__device__ void inc_candidate(Sim<kReg, kInc>& S, const SimParams& P, int64_t k, uint8_t* crow) {
  const DevGmg& g = S.g;
  const DevBase& B = P.base;
  const unsigned lane = lane_id();
  const int32_t m0 = P.move_off[k], m1 = P.move_off[k + 1];
  const int32_t nm = m1 - m0;
  const int words = (g.n + 31) >> 5;
  for (int w = lane; w < words; w += 32) S.bits[w] = 0u;
  __syncwarp();
  // Validate the move list; duplicates are found with the (zeroed) bitmap.
  bool bad_range = false, dup = false;
  for (int t = lane; t < nm; t += 32) {
    const int32_t op = P.move_op[m0 + t];
    const int dvc = P.move_dev[m0 + t];
    if (op < 0 || op >= g.n || dvc >= g.D) {
      bad_range = true;
    } else {
      const uint32_t b = 1u << (op & 31);
      if (atomicOr(&S.bits[op >> 5], b) & b) dup = true;
    }
  }
  bad_range = __any_sync(kFullMask, bad_range);
  dup = __any_sync(kFullMask, dup);
  __syncwarp();
  for (int t = lane; t < nm; t += 32) {
    const int32_t op = P.move_op[m0 + t];
    if (op >= 0 && op < g.n) atomicAnd(&S.bits[op >> 5], ~(1u << (op & 31)));
  }
  __syncwarp();
  if (B.status[0] != GMG_SIM_OK) {
    S.write_invalid(k, GMG_SIM_BADBASE);
    return;
  }
  if (bad_range || dup) {
    S.write_invalid(k, bad_range ? GMG_SIM_MOVE_RANGE : GMG_SIM_MOVE_DUP);
    return;
  }
  // The candidate's placement = base + moves.
  for (int c = lane * 16; c < B.ld; c += 512)
    *reinterpret_cast<uint4*>(crow + c) = *reinterpret_cast<const uint4*>(B.row + c);
  __syncwarp();
  uint64_t t0 = kKeyMax;
  for (int t = lane; t < nm; t += 32) {
    const int32_t op = P.move_op[m0 + t];
    const uint8_t dvc = P.move_dev[m0 + t];
    crow[op] = dvc;
    if (dvc != B.row[op]) {
      const uint4 ls = op_lists(g.ops, (uint32_t)op);
      uint64_t tx;
      if (ls.w == 0) {
        tx = (uint64_t)op_relxq(g.ops, (uint32_t)op).x;
      } else {
        tx = kKeyMax;
        for (uint32_t u = 0; u < ls.w; ++u) {
          const uint64_t fp = (uint64_t)S.fb[__ldg(g.pred + ls.z + u) & kIdMask];
          tx = fp < tx ? fp : tx;
        }
      }
      t0 = tx < t0 ? tx : t0;
    }
  }
  t0 = warp_min_u64(t0);
  __syncwarp();
  S.row = crow;
  const DevOut& o = P.out;
  if (t0 == kKeyMax) {
    // No effective move: the base results.
    const int64_t* rs = B.res_scalars;
    if (lane == 0) {
      o.makespan[k] = rs[0];
      o.score[k] = rs[1];
      o.status[k] = GMG_SIM_OK;
      o.viol_flag[k] = (int32_t)rs[2];
      o.viol_op[k] = (int32_t)rs[3];
      o.viol_dev[k] = (int32_t)rs[4];
      o.viol_time[k] = rs[5];
      o.sla_miss[k] = (int32_t)rs[6];
      o.events[k] = 0;
    }
    for (int d = lane; d < g.D; d += 32) o.peak[k * g.D + d] = B.res_peak[d];
    if (o.req_done)
      for (int r = lane; r < g.R; r += 32) o.req_done[k * g.R + r] = B.res_creq[r];
    const int ts = S.trace_slot(k);
    if (ts >= 0)
      for (int x = lane; x < g.n; x += 32) {
        o.trace_finish[(int64_t)ts * g.n + x] = B.fb[x];
        o.trace_start[(int64_t)ts * g.n + x] = B.fb[x] - op_durbytes(g.ops, (uint32_t)x).x;
      }
    return;
  }
  S.T0 = (int64_t)t0;
  // Latest recorded resume point at or before T0.
  int best = -1;
  for (int c = lane; c < B.nck; c += 32)
    if (B.ck_time[c] <= S.T0) best = c;
  const int c = __reduce_max_sync(kFullMask, best);
  // Restore the simulator state of checkpoint c.
  const int64_t* sc = B.ck_scalars + (int64_t)c * 8;
  S.Tc = B.ck_time[c];
  const int qsz = (int)sc[0];
  if (qsz > S.q.cap) {
    S.write_invalid(k, GMG_SIM_QUEUE);
    return;
  }
  S.rootptr = (int)sc[1];
  S.score = sc[2];
  S.makespan = sc[3];
  S.vflag = (int32_t)sc[4];
  S.vt = sc[5];
  S.vop = (int32_t)sc[6];
  S.vdev = (int32_t)sc[7];
  S.iters = 0;
  S.nev = 0;
  S.readypops = 0;
  S.last_t = -1;
  S.status = GMG_SIM_OK;
  S.dv.load(B.ck_dev + (int64_t)c * 3 * g.D);
  for (int r = lane; r < g.R; r += 32) S.creq[r] = B.ck_creq[(int64_t)c * g.R + r];
  // Copy the checkpoint queue, dropping events that the moves invalidate and
  // re-keying moved ops that were ready at T_c:
  //  * READY(x) of a moved x: its inputs' transfer times change;
  //  * FREE / remote ALLOC events of an op p with a moved successor: the set
  //    of receiving accelerators and last consumers of p's output changed
  //    (they are all at times >= f_p >= T0 and are regenerated below).
  int outn = 0;
  for (int c0 = 0; c0 < qsz; c0 += 32) {
    const int idx = c0 + (int)lane;
    const bool v = idx < qsz;
    uint64_t key = 0;
    uint32_t pay = 0;
    bool keep = false;
    if (v) {
      key = B.ck_qkey[(int64_t)c * B.ckq + idx];
      pay = B.ck_qpay[(int64_t)c * B.ckq + idx];
      keep = true;
      const uint32_t cls = S.kc.cls(key), op = S.kc.op(key);
      if (cls == kReady) {
        if (crow[op] != B.row[op]) {
          const int dx = crow[op];
          const uint4 ls = op_lists(g.ops, op);
          int64_t rx = op_relxq(g.ops, op).x;
          for (uint32_t u = 0; u < ls.w; ++u) {
            const uint32_t p = __ldg(g.pred + ls.z + u) & kIdMask;
            const int dp = crow[p];
            int64_t a = S.fb[p];
            if (dp != dx) a += S.xfer(dp, dx, op_durbytes(g.ops, p).y, op_relxq(g.ops, p).y);
            rx = a > rx ? a : rx;
          }
          key = S.kc.make(rx, kReady, op);
        }
      } else {
        const uint4 ls = op_lists(g.ops, op);
        bool moved_succ = false;
        for (uint32_t u = 0; u < ls.y && !moved_succ; ++u) {
          const uint32_t j = __ldg(g.succ + ls.x + u);
          moved_succ = crow[j] != B.row[j];
        }
        if (moved_succ && (cls == kFree || (int)(pay & 0xffu) != B.row[op])) keep = false;
      }
    }
    __syncwarp();
    const uint32_t bal = __ballot_sync(kFullMask, keep);
    const int pos = outn + __popc(bal & ((1u << lane) - 1u));
    if (keep) {
      *S.q.kp(pos) = key;
      *S.q.pp(pos) = pay;
    }
    outn += __popc(bal);
    __syncwarp();
  }
  S.q.size = outn;
  // Regenerate the memory events of every predecessor p (simulated before
  // T_c) of a moved op under the candidate placement.  Each p is handled by
  // its smallest-id moved successor.
  for (int c0 = 0; c0 < nm; c0 += 32) {
    const int t = c0 + (int)lane;
    int32_t x = -1;
    uint4 xls = make_uint4(0, 0, 0, 0);
    if (t < nm) {
      const int32_t op = P.move_op[m0 + t];
      if (crow[op] != B.row[op]) {
        x = op;
        xls = op_lists(g.ops, (uint32_t)op);
      }
    }
    const uint32_t maxp = __reduce_max_sync(kFullMask, x >= 0 ? xls.w : 0u);
    for (uint32_t u = 0; u < maxp; ++u) {
      uint32_t p = 0;
      bool want = false;
      if (x >= 0 && u < xls.w) {
        p = __ldg(g.pred + xls.z + u) & kIdMask;
        want = S.rb[p] < S.Tc;
        if (want) {
          const uint4 pls = op_lists(g.ops, p);
          for (uint32_t w = 0; w < pls.y; ++w) {
            const uint32_t j = __ldg(g.succ + pls.x + w);
            if ((int32_t)j >= x) break;  // successors are ascending
            if (crow[j] != B.row[j]) {
              want = false;
              break;
            }
          }
        }
      }
      uint32_t m = __ballot_sync(kFullMask, want);
      while (m) {
        const int src = __ffs(m) - 1;
        m &= m - 1;
        regen(S, __shfl_sync(kFullMask, p, src));
      }
    }
  }
  S.q.heapify();
  S.run();
  S.finish(k);
}

// Memory events of op p (finished before the resume point) under the
// candidate placement: receive copies on every remote accelerator of its
// successors (allocated at f_p), and the releases that are already
// determined because every listed consumer on that accelerator has finished.
template <bool kReg>
__device__ void regen(Sim<kReg, kInc>& S, uint32_t p) {
  const DevGmg& g = S.g;
  const unsigned lane = lane_id();
  const int64_t fp = S.fb[p];
  const int dp = S.row[p];
  const int64_t pb = op_durbytes(g.ops, p).y, pxq = op_relxq(g.ops, p).y;
  const uint4 pls = op_lists(g.ops, p);
  const uint4 pcs = op_cons(g.ops, p);
  const bool all = (pcs.w & kAllCons) != 0;
  const uint32_t* lst = all ? g.succ + pls.x : g.cons + pcs.x;
  const uint32_t nl = all ? pls.y : pcs.y;
  int64_t hold = fp;
  for (uint32_t c0 = 0; c0 < pls.y; c0 += 32) {
    const uint32_t t = c0 + lane;
    const bool v = t < pls.y;
    int du = -1;
    int64_t arr = fp;
    if (v) {
      du = S.row[__ldg(g.succ + pls.x + t)];
      if (du != dp) arr = fp + S.xfer(dp, du, pb, pxq);
    }
    const bool rem = v && du != dp;
    const uint32_t peers = __match_any_sync(kFullMask, rem ? (uint32_t)du : (256u + lane));
    bool leader = rem && (__ffs(peers) - 1 == (int)lane);
    if (leader && c0 > 0)
      for (uint32_t u = 0; u < c0; ++u)
        if (S.row[__ldg(g.succ + pls.x + u)] == du) {
          leader = false;
          break;
        }
    const uint64_t hm = warp_max_u64(leader ? (uint64_t)arr : 0ull);
    hold = (int64_t)hm > hold ? (int64_t)hm : hold;
    S.template push_lanes<true>(__ballot_sync(kFullMask, leader), S.kc.make(fp, kAlloc, p), (uint32_t)du);
    bool rel = false;
    int64_t tr = arr;
    if (leader) {
      rel = true;
      for (uint32_t u = 0; u < nl; ++u) {
        const uint32_t c = __ldg(lst + u);
        if (S.row[c] != du) continue;
        if (!S.popped(c)) {
          rel = false;
          break;
        }
        const int64_t fc = S.fin(c);
        tr = fc > tr ? fc : tr;
      }
    }
    S.template push_lanes<true>(__ballot_sync(kFullMask, rel), S.kc.make(tr, kFree, p), (uint32_t)du);
  }
  // source copy
  bool pending = false;
  uint64_t mx = 0;
  for (uint32_t c0 = 0; c0 < nl; c0 += 32) {
    const uint32_t t = c0 + lane;
    if (t < nl) {
      const uint32_t c = __ldg(lst + t);
      if (S.row[c] == dp) {
        if (!S.popped(c)) pending = true;
        else {
          const uint64_t fc = (uint64_t)S.fin(c);
          mx = fc > mx ? fc : mx;
        }
      }
    }
  }
  if (__any_sync(kFullMask, pending)) return;
  const int64_t m = (int64_t)warp_max_u64(mx);
  S.append(S.kc.make(m > hold ? m : hold, kFree, p), (uint32_t)dp);
}

template <bool kReg>
__global__ void __launch_bounds__(128) sim_inc_kernel(const __grid_constant__ SimParams P) {
  extern __shared__ __align__(16) uint8_t smem[];
  const unsigned wib = threadIdx.x >> 5;
  const int64_t slot = (int64_t)blockIdx.x * (blockDim.x >> 5) + wib;
  const int64_t nslots = (int64_t)gridDim.x * (blockDim.x >> 5);
  Sim<kReg, kInc> S(P);
  setup_slot(S, P, wib, slot, smem);
  S.rb = P.base.rb;
  S.fb = P.base.fb;
  S.brow = P.base.row;
  uint8_t* crow = P.scratch + slot * P.slot_bytes + P.off_row;
  for (int64_t k = slot; k < P.K; k += nslots) inc_candidate(S, P, k, crow);
}

// ---------------------------------------------------------------------------
// select_best (Algorithm 1, BestRecordedCandidateResult): block argmin of
// the packed rank, then a one-block final argmin.
// rank = (status != 0 || infeasible) ? none : (mode ? sla_miss : 0, score, k)
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

const void* full_kernel_ptr(bool reg) {
  return reg ? (const void*)sim_full_kernel<true> : (const void*)sim_full_kernel<false>;
}
const void* inc_kernel_ptr(bool reg) {
  return reg ? (const void*)sim_inc_kernel<true> : (const void*)sim_inc_kernel<false>;
}

cudaError_t launch_full(bool reg, const SimParams& P, int grid, int block, size_t smem, cudaStream_t st) {
  if (reg) sim_full_kernel<true><<<grid, block, smem, st>>>(P);
  else sim_full_kernel<false><<<grid, block, smem, st>>>(P);
  return cudaGetLastError();
}

cudaError_t launch_inc(bool reg, const SimParams& P, int grid, int block, size_t smem, cudaStream_t st) {
  if (reg) sim_inc_kernel<true><<<grid, block, smem, st>>>(P);
  else sim_inc_kernel<false><<<grid, block, smem, st>>>(P);
  return cudaGetLastError();
}

cudaError_t launch_base(bool reg, const SimParams& P, size_t smem, cudaStream_t st) {
  if (reg) sim_base_kernel<true><<<1, 32, smem, st>>>(P);
  else sim_base_kernel<false><<<1, 32, smem, st>>>(P);
  return cudaGetLastError();
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
