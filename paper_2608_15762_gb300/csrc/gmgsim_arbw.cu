// sim_batch / sim_incremental with arbitrated transfers (Sec. 3.5.2,
// "Tensor Transfer Arbitration") for 33 to 256 accelerators.  The same
// simulation as gmgsim_arb.cu (same events, same arbitration order, same
// HBM accounting); what differs is where an accelerator's transfer state
// lives.  With more accelerators than lanes, the state of accelerator a --
// the completion time, producer and destination of the transfer it is
// sending, the head, tail and head finish time of its FIFO of coming intents
// (started ops with remote successors, in finish order), and the set of
// destinations it has pending intents for -- sits in per-warp tables that the
// lanes stride over (a = lane, lane + 32, ...).  Busy sending and receiving
// endpoints and the sources with pending intents are W = ceil(D/32)-word bit
// sets in shared memory; busy links a bit set over the D*D link ids.
//
// The next DONE and the next INTENT are warp minima over the tables, kept
// current as they change.  The arbiter scans, per lane, the free sources with
// pending intents and their pending destinations whose receiver (and link)
// is free, takes the smallest queue number over the warp, starts it, and
// repeats.  Intents are numbered as they arrive, in (time, producer) order
// and destination order within a producer, so the smallest head number is
// the (intent time, producer, destination) order of the paper's FIFO-greedy
// reading.  An op's remote destinations are recomputed from its successor
// list (one bit per accelerator) when needed instead of being stored.
//
// The HBM-event generation and the input counting are the narrow kernel's
// (gmg_arb_events.h).  Every loop is bounded by the graph: DONEs by the
// number of transfers, INTENTs by the number of ops.
#include <algorithm>

#include "gmg_arbw.h"
#include "gmg_arb_events.h"

namespace gsim {
namespace {

template <bool kT32, bool kTypes>
struct ArbWSim : ArbEvents<ArbWSim<kT32, kTypes>, Sim<false, kFull, true, kT32, kTypes>> {
  using Base = ArbEvents<ArbWSim<kT32, kTypes>, Sim<false, kFull, true, kT32, kTypes>>;
  using tm_t = typename Base::tm_t;
  using U = typename std::make_unsigned<tm_t>::type;
  using Base::g;
  using Base::P;
  using Base::row;
  using Base::status;
  using Base::add_input;
  using Base::drain;
  using Base::drop_hold;
  using Base::generate;
  using Base::push_readies;
  static constexpr tm_t kNever = (tm_t)(~(U)0 >> 1);
  const ArbWParams& A;
  uint8_t* sl;       // the warp's scratch slot
  uint32_t* sb;      // shared [W] busy senders
  uint32_t* rb;      // shared [W] busy receivers
  uint32_t* ps;      // shared [W] sources with a pending intent
  uint32_t* rs;      // shared [W] work set: an op's remote accelerators
  int32_t nx;        // intents arrived so far
  int32_t xev;       // transfer events handled (loop guard)
  bool arb_due;
  tm_t t_arb;
  tm_t td_c;         // next DONE time, kept current
  int td_src;        // the lowest accelerator whose transfer completes at td_c
  uint64_t ik_c;     // next INTENT key (time << ib | op), kept current

  __device__ ArbWSim(const ArbWParams& a) : Base(a.P), A(a) {}

  template <typename T>
  __device__ __forceinline__ T* at(int64_t off) const { return reinterpret_cast<T*>(sl + off); }
  __device__ __forceinline__ int32_t* cnt() const { return at<int32_t>(A.off_cnt); }
  __device__ __forceinline__ tm_t* rmax() const { return at<tm_t>(A.off_rmax); }
  __device__ __forceinline__ int32_t* refs() const { return at<int32_t>(A.off_refs); }
  __device__ __forceinline__ int32_t* nextop() const { return at<int32_t>(A.off_nextop); }
  __device__ __forceinline__ uint32_t* xent() const { return at<uint32_t>(A.off_xent); }
  __device__ __forceinline__ int32_t* xnext() const { return at<int32_t>(A.off_xnext); }
  __device__ __forceinline__ int32_t* qhead() const { return at<int32_t>(A.off_qhead); }
  __device__ __forceinline__ int32_t* qtail() const { return at<int32_t>(A.off_qtail); }
  __device__ __forceinline__ tm_t* xd() const { return at<tm_t>(A.off_xd); }
  __device__ __forceinline__ uint32_t* xp() const { return at<uint32_t>(A.off_xp); }
  __device__ __forceinline__ int32_t* xe() const { return at<int32_t>(A.off_xe); }
  __device__ __forceinline__ int32_t* fh() const { return at<int32_t>(A.off_fh); }
  __device__ __forceinline__ int32_t* ft() const { return at<int32_t>(A.off_ft); }
  __device__ __forceinline__ tm_t* fa() const { return at<tm_t>(A.off_fa); }
  __device__ __forceinline__ uint32_t* pm() const { return at<uint32_t>(A.off_pm); }
  __device__ __forceinline__ uint32_t* lb() const { return at<uint32_t>(A.off_lb); }

  __device__ __forceinline__ tm_t warp_min_t(tm_t v) const {
    if (kT32) return (tm_t)__reduce_min_sync(kFullMask, (int)v);
    return (tm_t)warp_min_u64((uint64_t)v);  // times are >= 0
  }
  static __device__ __forceinline__ bool bit(const uint32_t* s, int i) { return (s[i >> 5] >> (i & 31)) & 1u; }

  // The tables hold at most 256 accelerators, eight per lane: each lane loads
  // its eight entries together, then reduces.
  static constexpr int kPerLane = 8;

  // The next completion and the lowest accelerator completing then.
  __device__ void refresh_done() {
    const int lane = (int)lane_id();
    tm_t v[kPerLane];
#pragma unroll
    for (int u = 0; u < kPerLane; ++u) {
      const int a = lane + 32 * u;
      v[u] = a < g.D ? xd()[a] : kNever;
    }
    tm_t m = kNever;
    int am = 0x7fffffff;
#pragma unroll
    for (int u = 0; u < kPerLane; ++u)
      if (v[u] < m) {
        m = v[u];
        am = lane + 32 * u;
      }
    td_c = warp_min_t(m);
    td_src = (int)__reduce_min_sync(kFullMask, (unsigned)(m == td_c ? am : 0x7fffffff));
  }
  __device__ void refresh_intent() {
    const int lane = (int)lane_id();
    int32_t h[kPerLane];
    tm_t f[kPerLane];
#pragma unroll
    for (int u = 0; u < kPerLane; ++u) {
      const int a = lane + 32 * u;
      const bool in = a < g.D;
      h[u] = in ? fh()[a] : -1;
      f[u] = in ? fa()[a] : kNever;
    }
    uint64_t k = kKeyMax;
#pragma unroll
    for (int u = 0; u < kPerLane; ++u)
      if (h[u] >= 0) {
        const uint64_t v = ((uint64_t)(U)f[u] << g.ib) | (uint32_t)h[u];
        k = v < k ? v : k;
      }
    ik_c = warp_min_u64(k);
  }

  __device__ void setup_arb(int64_t slot, uint8_t* smem_warp) {
    sl = P.scratch + slot * P.slot_bytes;
    uint32_t* w = reinterpret_cast<uint32_t*>(smem_warp);
    sb = w;
    rb = w + 8;
    ps = w + 16;
    rs = w + 24;
  }

  __device__ void reset_arb() {
    const unsigned lane = lane_id();
    const int D = g.D, W = A.words;
    this->reset_common();
    uint4* c4 = reinterpret_cast<uint4*>(cnt());
    const int nv = (int)((4 * (size_t)g.n + 15) / 16);
    for (int x = lane; x < nv; x += 32) c4[x] = make_uint4(0u, 0u, 0u, 0u);
    int32_t* qh = qhead();
    int32_t* qt = qtail();
    for (int x = lane; x < D * D; x += 32) {
      qh[x] = -1;
      qt[x] = -1;
    }
    for (int a = lane; a < D; a += 32) {
      xd()[a] = kNever;
      fh()[a] = -1;
      ft()[a] = -1;
      fa()[a] = kNever;
    }
    for (int x = lane; x < D * W; x += 32) pm()[x] = 0u;
    for (int x = lane; x < (D * D + 31) / 32; x += 32) lb()[x] = 0u;
    if (lane < 8) {
      sb[lane] = 0u;
      rb[lane] = 0u;
      ps[lane] = 0u;
      rs[lane] = 0u;
    }
    nx = 0;
    xev = 0;
    arb_due = false;
    t_arb = 0;
    td_c = kNever;
    td_src = 0;
    ik_c = kKeyMax;
    __syncwarp();
  }

  // rs := the accelerators other than dp that run a successor of p; returns
  // their number (uniform).
  __device__ int remote_set(uint32_t p, int dp) {
    const unsigned lane = lane_id();
    if (lane < 8) rs[lane] = 0u;
    __syncwarp();
    const XqSucc xs = op_xqsucc(g.ops, p);
    for (uint32_t u = lane; u < xs.nsucc; u += 32) {
      const int dj = row[__ldg(g.succ + xs.succ_off + u)];
      if (dj != dp) atomicOr(rs + (dj >> 5), 1u << (dj & 31));
    }
    __syncwarp();
    const int c = lane < (unsigned)A.words ? __popc(rs[lane]) : 0;
    return (int)__reduce_add_sync(kFullMask, (unsigned)c);
  }

  // READY(r, i): start op i; local successors get this input; if some
  // successor is remote, i joins its accelerator's FIFO of coming intents.
  __device__ void start_op(uint32_t i, tm_t r) {
    const unsigned lane = lane_id();
    const longlong2 db = op_durbytes(g.ops, i);
    const XqSucc xs = op_xqsucc(g.ops, i);
    const uint4 cs = op_cons(g.ops, i);
    const int d = row[i];
    const tm_t dur = (tm_t)this->dur_of(i, d, db.x);
    const tm_t fd = this->dv.get_free(d);
    const tm_t s = r > fd ? r : fd;
    const tm_t f = s + dur;
    this->dv.set_free(d, f);
    if (lane == 0) {
      this->fbuf[i] = f;
      if (cs.w & kReqSink)
        atomicMax(reinterpret_cast<unsigned long long*>(this->creq + (int32_t)cs.z), (unsigned long long)f);
      this->oplog[this->opn] = i;
    }
    ++this->opn;
    if (cs.w & kScored) this->score += (int64_t)f;
    __syncwarp();
    for (uint32_t c0 = 0; c0 < xs.nsucc; c0 += 32) {
      const uint32_t t = c0 + lane;
      uint32_t j = 0;
      tm_t rj = 0;
      bool rdy = false;
      if (t < xs.nsucc) {
        j = __ldg(g.succ + xs.succ_off + t);
        if (row[j] == d) rdy = add_input(j, f, rj);
      }
      push_readies(rdy, rj, j);
    }
    __syncwarp();
    const int nrem = remote_set(i, d);
    if (lane == 0) {
      refs()[i] = 1 + nrem;
      this->holdb[i] = f;
      if (nrem) {
        if (fh()[d] < 0) {
          fh()[d] = (int32_t)i;
          fa()[d] = f;
        } else {
          nextop()[ft()[d]] = (int32_t)i;
        }
        ft()[d] = (int32_t)i;
      }
    }
    __syncwarp();
    if (nrem) refresh_intent();
  }

  // The intents of the earliest FIFO head p arrive: one per remote
  // accelerator, numbered in destination order.
  __device__ void intents_arrive(uint32_t p) {
    const unsigned lane = lane_id();
    const int a = row[p];
    const int W = A.words;
    const int nrem = remote_set(p, a);
    if (nx + nrem > A.xcap) {
      status = GMG_SIM_QUEUE;
      return;
    }
    if (lane == 0) {
      uint32_t* xe_ = xent();
      int32_t* xn = xnext();
      int32_t* qh = qhead();
      int32_t* qt = qtail();
      uint32_t* pmr = pm() + (size_t)a * W;
      for (int w = 0; w < W; ++w) {
        uint32_t r = rs[w];
        pmr[w] |= r;
        while (r) {
          const int e = 32 * w + __ffs(r) - 1;
          r &= r - 1;
          const int32_t x = nx++;
          const int pair = a * g.D + e;
          xe_[x] = (p << 8) | (uint32_t)e;
          xn[x] = -1;
          const int32_t tl = qt[pair];
          if (tl >= 0) xn[tl] = x;
          else qh[pair] = x;
          qt[pair] = x;
        }
      }
      ps[a >> 5] |= 1u << (a & 31);
      // advance a's FIFO
      const int32_t h = fh()[a];
      if (h == ft()[a]) {
        fh()[a] = -1;
        ft()[a] = -1;
        fa()[a] = kNever;
      } else {
        const int32_t nh = nextop()[h];
        fh()[a] = nh;
        fa()[a] = this->fbuf[nh];
      }
    } else {
      nx += nrem;
    }
    __syncwarp();
    refresh_intent();
  }

  // The transfer sent by accelerator src completes at time t.
  __device__ void transfer_done(int src, tm_t t) {
    const unsigned lane = lane_id();
    const uint32_t p = xp()[src];
    const int e = xe()[src];
    __syncwarp();
    if (lane == 0) {
      xd()[src] = kNever;
      sb[src >> 5] &= ~(1u << (src & 31));
      rb[e >> 5] &= ~(1u << (e & 31));
      if (A.shared_links) {
        const uint32_t lid = __ldg(A.link + src * g.D + e);
        lb()[lid >> 5] &= ~(1u << (lid & 31u));
      }
    }
    __syncwarp();
    refresh_done();
    // p's successors on e have this input now
    const XqSucc xs = op_xqsucc(g.ops, p);
    for (uint32_t c0 = 0; c0 < xs.nsucc; c0 += 32) {
      const uint32_t u = c0 + lane;
      uint32_t j = 0;
      tm_t rj = 0;
      bool rdy = false;
      if (u < xs.nsucc) {
        j = __ldg(g.succ + xs.succ_off + u);
        if (row[j] == e) rdy = add_input(j, t, rj);
      }
      push_readies(rdy, rj, j);
    }
    __syncwarp();
    // the receive copy: released on arrival if no listed consumer is on e
    const uint4 cs = op_cons(g.ops, p);
    bool here = (cs.w & kAllCons) != 0;
    if (!here) {
      bool f = false;
      for (uint32_t u = lane; u < cs.y; u += 32) f |= row[__ldg(g.cons + cs.x + u)] == e;
      here = __any_sync(kFullMask, f);
    }
    this->log_event(lane == 0 && !here, this->kc.make(t, kFree, p), e);
    drop_hold(lane == 0, p, t, src);
  }

  __device__ __forceinline__ tm_t xfer_of(int src, int e, uint32_t p) const {
    return this->xfer(src, e, op_durbytes(g.ops, p).y, op_xqsucc(g.ops, p).xq);
  }

  // Start every pending intent whose endpoints and link are free, in order.
  __device__ void arbitrate(tm_t t) {
    const unsigned lane = lane_id();
    const int D = g.D, W = A.words;
    const bool links = A.shared_links != 0;
    bool started = false;
    while (true) {
      uint32_t best = 0xffffffffu;
      int bs = 0, be = 0;
      for (int a = lane; a < D; a += 32) {
        if (!bit(ps, a) || bit(sb, a)) continue;
        const uint32_t* pmr = pm() + (size_t)a * W;
        for (int w = 0; w < W; ++w) {
          uint32_t c = pmr[w] & ~rb[w];
          while (c) {
            const int e = 32 * w + __ffs(c) - 1;
            c &= c - 1;
            if (links) {
              const uint32_t lid = __ldg(A.link + a * D + e);
              if ((lb()[lid >> 5] >> (lid & 31u)) & 1u) continue;
            }
            const uint32_t h = (uint32_t)qhead()[a * D + e];
            if (h < best) {
              best = h;
              bs = a;
              be = e;
            }
          }
        }
      }
      const uint32_t m = __reduce_min_sync(kFullMask, best);
      if (m == 0xffffffffu) break;
      started = true;
      const int sel = __ffs(__ballot_sync(kFullMask, best == m)) - 1;
      const int src = __shfl_sync(kFullMask, bs, sel);
      const int e = __shfl_sync(kFullMask, be, sel);
      const uint32_t p = xent()[m] >> 8;
      const int32_t nxt = xnext()[m];
      const int pair = src * D + e;
      const tm_t done = t + xfer_of(src, e, p);
      __syncwarp();
      if (lane == 0) {
        qhead()[pair] = nxt;
        if (nxt < 0) {
          qtail()[pair] = -1;
          uint32_t* pmr = pm() + (size_t)src * W;
          pmr[e >> 5] &= ~(1u << (e & 31));
          uint32_t any = 0u;
          for (int w = 0; w < W; ++w) any |= pmr[w];
          if (!any) ps[src >> 5] &= ~(1u << (src & 31));
        }
        sb[src >> 5] |= 1u << (src & 31);
        rb[e >> 5] |= 1u << (e & 31);
        if (links) {
          const uint32_t lid = __ldg(A.link + pair);
          lb()[lid >> 5] |= 1u << (lid & 31u);
        }
        xd()[src] = done;
        xp()[src] = p;
        xe()[src] = e;
      }
      __syncwarp();
      this->log_event(lane == 0, this->kc.make(t, kAlloc, p), e);
    }
    if (started) refresh_done();
  }

  // The event loop: transfer events, then the arbiter once the last event of
  // a time is handled, then READY keys.
  __device__ void run() {
    if (status) return;
    const int32_t xlim = A.xcap + g.n + 2;
    while (true) {
      const tm_t td = td_c;
      const uint64_t ik = ik_c;
      const tm_t ti = ik == kKeyMax ? kNever : (tm_t)(ik >> g.ib);
      const tm_t tx = td < ti ? td : ti;
      if (arb_due && tx > t_arb) {
        arbitrate(t_arb);
        arb_due = false;
        if (status) break;
        continue;
      }
      const uint64_t top = this->q.top();
      const uint64_t rm = warp_min_u64(this->rk_reg);
      const uint64_t rk = this->rkey;
      uint64_t nk = rk < top ? rk : top;
      nk = rm < nk ? rm : nk;
      if (tx != kNever && (nk == kKeyMax || (int64_t)tx <= this->kc.time(nk))) {
        if (++xev > xlim) {
          status = GMG_SIM_LOOP;
          break;
        }
        if (td == tx) {
          transfer_done(td_src, td);
        } else {
          intents_arrive((uint32_t)(ik & this->kc.mask));
        }
        arb_due = true;
        t_arb = tx;
        if (status) break;
        continue;
      }
      if (nk == kKeyMax) break;
      if (this->opn >= P.opcap) drain(this->kc.time(nk));
      if (nk == rm) {
        if (this->rk_reg == rm) this->rk_reg = kKeyMax;
      } else if (nk == rk) {
        ++this->rootptr;
        this->load_root();
      } else {
        __syncwarp();
        this->q.pop();
      }
      if (++this->iters > (int32_t)g.max_iter) {
        status = GMG_SIM_LOOP;
        break;
      }
      start_op(this->kc.op(nk), (tm_t)this->kc.time(nk));
      if (status) break;
    }
    if (!status) drain(kI64Max);
  }
};

template <bool kT32, bool kTypes>
__global__ void __launch_bounds__(128, 6) sim_arbw_kernel(const __grid_constant__ ArbWParams A) {
  extern __shared__ __align__(16) uint8_t smem[];
  const unsigned wib = threadIdx.x >> 5;
  const int64_t slot = (int64_t)blockIdx.x * (blockDim.x >> 5) + wib;
  const int64_t nslots = (int64_t)gridDim.x * (blockDim.x >> 5);
  ArbWSim<kT32, kTypes> S(A);
  setup_slot(S, A.P, wib, slot, smem);
  S.setup_arb(slot, smem + A.smem_std + (size_t)wib * A.smem_arb);
  for (int64_t k = slot; k < A.P.K; k += nslots) {
    S.row = A.P.place + k * A.P.ld;
    if (A.pre_status) {
      const int32_t st = A.pre_status[k];
      if (st != GMG_SIM_OK) {
        S.write_invalid(k, st);
        continue;
      }
    }
    if (S.row_has_bad_device(S.row)) {
      S.write_invalid(k, GMG_SIM_BADDEV);
      continue;
    }
    S.reset_arb();
    S.run();
    S.finish(k);
  }
}

}  // namespace

const void* arbw_kernel_ptr(bool t32, bool types) {
  if (t32) return types ? (const void*)sim_arbw_kernel<true, true> : (const void*)sim_arbw_kernel<true, false>;
  return types ? (const void*)sim_arbw_kernel<false, true> : (const void*)sim_arbw_kernel<false, false>;
}

cudaError_t launch_arbw(bool t32, bool types, const ArbWParams& A, int grid, int block, size_t smem,
                        cudaStream_t st) {
  void* args[] = {const_cast<ArbWParams*>(&A)};
  return cudaLaunchKernel(arbw_kernel_ptr(t32, types), dim3(grid), dim3(block), args, smem, st);
}

}  // namespace gsim
