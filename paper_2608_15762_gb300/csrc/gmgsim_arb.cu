// sim_batch with arbitrated transfers (Sec. 3.5.2, "Tensor Transfer
// Arbitration"): one warp per candidate, as in the pure-latency simulation,
// with two more kinds of event.
//
//   INTENT(f_p, p)     producer p finished; its output is wanted on every
//                      distinct remote accelerator e of p's successors: one
//                      intent per e joins the FIFO queue of the pair (dev p, e).
//   DONE(c, p, e)      the transfer arrived: the sender's endpoint, e's
//                      receiving endpoint and the pair's link are free again;
//                      p's successors on e have one more input present.
//
// Lane a keeps accelerator a's side of both in registers.  An accelerator
// sends one transfer at a time, so lane a holds the completion time of the
// transfer it is sending, if any; and its ops finish in the order they start,
// so the ops with remote successors that it has started but whose intents
// have not arrived form a FIFO in finish order: lane a holds its head.  The
// next DONE and the next INTENT are warp minima over the lanes (intents by
// (time, producer)).
//
// After every INTENT / DONE at time t the arbiter starts, in (intent time,
// producer, destination) order, every pending intent whose sending endpoint,
// receiving endpoint and link are all free (the communication graph of Sec.
// 3.5.2; the selection rule among conflicting intents is this FIFO greedy
// one).  Intents are numbered as they arrive, which is that order, and only
// the head of a pair's queue can start (the rest share its endpoints), so the
// arbiter repeatedly takes the smallest head number over the pairs whose
// endpoints and link are free: lane a scans the pairs out of accelerator a, a
// warp minimum picks the winner.  A started transfer allocates its receive
// buffer and lasts the transfer estimate.  When no two ordered pairs share a
// link id, a busy link implies a busy sender and the link state is not kept.
//
// Readiness: an op's inputs are counted as they become present -- a local
// predecessor's output when that predecessor starts (its finish time is then
// known), a remote one when its transfer is DONE -- and the op becomes READY
// at the latest arrival once all are there.  Transfer events at a time are
// handled before READY keys at that time (a DONE can make an op ready then).
//
// HBM events: an op's own copy is released once two holds are gone -- its
// last local listed consumer has finished (or the op itself, if none) and
// every outgoing transfer has arrived -- at the later of those times; a
// receive copy is allocated when its transfer starts and released by its last
// listed consumer there (or on arrival if none).  Every such event is logged
// at a time no earlier than the sweep's, so the batched drain of the
// pure-latency simulation applies unchanged.
//
// Requires at most 32 accelerators (endpoint sets are warp bit masks) and an
// accelerator id that fits beside the packed key.  Every loop is bounded by
// the graph: DONEs by the number of transfers, INTENTs by the number of ops.
#include <algorithm>

#include "gmg_arb.h"
#include "gmg_arb_events.h"

namespace gsim {
namespace {

// kMode: kFull (sim_batch), kBase (the arbitrated base snapshot: records
// ready and finish times and checkpoints), kInc (candidates resumed from it).
template <bool kT32, bool kTypes, int kMode = kFull>
struct ArbSim : ArbEvents<ArbSim<kT32, kTypes, kMode>, Sim<true, kMode, true, kT32, kTypes>> {
  using Base = ArbEvents<ArbSim<kT32, kTypes, kMode>, Sim<true, kMode, true, kT32, kTypes>>;
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
  const ArbParams& A;
  // The warp's scratch slot and shared area; the arrays in them are found
  // from the launch parameters' offsets when used (registers are scarce).
  uint8_t* sl;
  uint8_t* sm;       // [0, 128): busy links (32 words); then the queue heads if shared
  int32_t nx;        // intents arrived so far
  int32_t xev;       // transfer events handled (loop guard)
  uint32_t sendm, recvm;  // accelerators whose sending / receiving endpoint is busy
  // lane a: accelerator a's transfer state
  uint32_t pm;       // destinations with a pending intent from a
  tm_t xd;           // completion of the transfer a is sending (kNever: none)
  uint32_t xdp;      // its producer
  int xde;           // its destination
  int32_t fh, ft;    // FIFO of started ops with remote successors (-1: empty)
  tm_t fa;           // finish time of the FIFO head (kNever: empty)
  bool arb_due;
  tm_t t_arb;
  tm_t td_c;         // next DONE time (warp minimum of xd), kept current
  uint64_t ik_c;     // next INTENT key (time << ib | op), kept current

  __device__ ArbSim(const ArbParams& a) : Base(a.P), A(a) {}

  template <typename T>
  __device__ __forceinline__ T* at(int64_t off) const { return reinterpret_cast<T*>(sl + off); }
  __device__ __forceinline__ int32_t* cnt() const { return at<int32_t>(A.off_cnt); }      // [N] inputs present
  __device__ __forceinline__ tm_t* rmax() const { return at<tm_t>(A.off_rmax); }          // [N] latest arrival
  __device__ __forceinline__ int32_t* refs() const { return at<int32_t>(A.off_refs); }    // [N] holds left
  __device__ __forceinline__ uint32_t* rmask() const { return at<uint32_t>(A.off_rmask); }  // [N] remote accs
  __device__ __forceinline__ int32_t* nextop() const { return at<int32_t>(A.off_nextop); }  // [N] FIFO link
  __device__ __forceinline__ uint32_t* xent() const { return at<uint32_t>(A.off_xent); }  // [xcap] p << 5 | e
  __device__ __forceinline__ int32_t* xnext() const { return at<int32_t>(A.off_xnext); }  // [xcap]
  __device__ __forceinline__ int32_t* qtail() const { return at<int32_t>(A.off_qtail); }  // [D*D]
  __device__ __forceinline__ int32_t* qhead() const {                                      // [D*D]
    return A.heads_shared ? reinterpret_cast<int32_t*>(sm + 128) : at<int32_t>(A.off_qhead);
  }
  __device__ __forceinline__ uint32_t* lbits() const { return reinterpret_cast<uint32_t*>(sm); }

  __device__ __forceinline__ tm_t warp_min_t(tm_t v) const {
    if (kT32) return (tm_t)__reduce_min_sync(kFullMask, (int)v);
    return (tm_t)warp_min_u64((uint64_t)v);  // times are >= 0
  }

  __device__ __forceinline__ void refresh_done() { td_c = warp_min_t(xd); }
  __device__ __forceinline__ void refresh_intent() {
    ik_c = warp_min_u64(fh >= 0 ? (((uint64_t)(U)fa << g.ib) | (uint32_t)fh) : kKeyMax);
  }

  __device__ void setup_arb(int64_t slot, uint8_t* smem_warp) {
    sl = P.scratch + slot * P.slot_bytes;
    sm = smem_warp;
  }

  __device__ void reset_arb() {
    const unsigned lane = lane_id();
    this->reset_common();
    uint4* c4 = reinterpret_cast<uint4*>(cnt());
    int32_t* qh = qhead();
    int32_t* qt = qtail();
    const int nv = (int)((4 * (size_t)g.n + 15) / 16);
    for (int x = lane; x < nv; x += 32) c4[x] = make_uint4(0u, 0u, 0u, 0u);
    for (int x = lane; x < g.D * g.D; x += 32) {
      qh[x] = -1;
      qt[x] = -1;
    }
    lbits()[lane] = 0u;
    nx = 0;
    xev = 0;
    sendm = recvm = pm = 0u;
    xd = kNever;
    xdp = 0u;
    xde = 0;
    fh = ft = -1;
    fa = kNever;
    arb_due = false;
    t_arb = 0;
    td_c = kNever;
    ik_c = kKeyMax;
    __syncwarp();
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
      if (kMode == kBase) P.base.rb[i] = r;
      this->oplog[this->opn] = i;
    }
    ++this->opn;
    if (cs.w & kScored) this->score += (int64_t)f;
    if (kMode == kBase) {
      this->makespan = f > this->makespan ? f : this->makespan;
      ++this->readypops;
    }
    if (kMode == kInc && r >= this->T0) ++this->nev;
    __syncwarp();
    uint32_t remote = 0u;
    for (uint32_t c0 = 0; c0 < xs.nsucc; c0 += 32) {
      const uint32_t t = c0 + lane;
      uint32_t j = 0;
      tm_t rj = 0;
      bool rdy = false;
      if (t < xs.nsucc) {
        j = __ldg(g.succ + xs.succ_off + t);
        const int dj = row[j];
        if (dj == d) rdy = add_input(j, f, rj);
        else remote |= 1u << dj;
      }
      push_readies(rdy, rj, j);
    }
    remote = __reduce_or_sync(kFullMask, remote);
    if (lane == 0) {
      refs()[i] = 1 + __popc(remote);
      this->holdb[i] = f;
      if (remote) rmask()[i] = remote;
    }
    if (remote && (int)lane == d) {
      if (fh < 0) {
        fh = (int32_t)i;
        fa = f;
      } else {
        nextop()[ft] = (int32_t)i;
      }
      ft = (int32_t)i;
    }
    __syncwarp();
    if (remote) refresh_intent();
  }

  // The intents of the earliest FIFO head arrive: one per remote
  // accelerator, numbered in destination order.
  __device__ void intents_arrive(uint32_t p) {
    const unsigned lane = lane_id();
    const int a = row[p];
    const uint32_t R = rmask()[p];
    if (nx + __popc(R) > A.xcap) {
      status = GMG_SIM_QUEUE;
      return;
    }
    if (lane == 0) {
      uint32_t* xe = xent();
      int32_t* xn = xnext();
      int32_t* qh = qhead();
      int32_t* qt = qtail();
      uint32_t r = R;
      while (r) {
        const int e = __ffs(r) - 1;
        r &= r - 1;
        const int32_t x = nx++;
        const int pair = a * g.D + e;
        xe[x] = (p << 5) | (uint32_t)e;
        xn[x] = -1;
        const int32_t tl = qt[pair];
        if (tl >= 0) xn[tl] = x;
        else qh[pair] = x;
        qt[pair] = x;
      }
    } else {
      nx += __popc(R);
    }
    if ((int)lane == a) {
      pm |= R;
      if (fh == ft) {
        fh = ft = -1;
        fa = kNever;
      } else {
        fh = nextop()[fh];
        fa = this->fin((uint32_t)fh);
      }
    }
    __syncwarp();
    refresh_intent();
  }

  // The transfer sent by lane src completes at time t.
  __device__ void transfer_done(int src, tm_t t) {
    const unsigned lane = lane_id();
    const uint32_t p = __shfl_sync(kFullMask, xdp, src);
    const int e = __shfl_sync(kFullMask, xde, src);
    if ((int)lane == src) xd = kNever;
    refresh_done();
    sendm &= ~(1u << src);
    recvm &= ~(1u << e);
    if (A.shared_links) {
      const uint32_t lid = __ldg(A.link + src * g.D + e);
      if (lane == 0) lbits()[lid >> 5] &= ~(1u << (lid & 31u));
      __syncwarp();
    }
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
    bool here = (cs.w & kAllCons) != 0;  // the successors there are consumers
    if (!here) {
      bool f = false;
      for (uint32_t u = lane; u < cs.y; u += 32) f |= row[__ldg(g.cons + cs.x + u)] == e;
      here = __any_sync(kFullMask, f);
    }
    this->log_event(lane == 0 && !here, this->kc.make(t, kFree, p), e);
    // the sender's copy: one hold fewer
    drop_hold(lane == 0, p, t, src);
  }

  // Start every pending intent whose endpoints and link are free, in order.
  __device__ void arbitrate(tm_t t) {
    const int lane = (int)lane_id();
    const int D = g.D;
    const bool links = A.shared_links != 0;
    bool started = false;
    while (true) {
      uint32_t best = 0xffffffffu;
      int be = 0;
      if (lane < D && !((sendm >> lane) & 1u)) {
        uint32_t c = pm & ~recvm;
        while (c) {
          const int e = __ffs(c) - 1;
          c &= c - 1;
          if (links) {
            const uint32_t lid = __ldg(A.link + lane * D + e);
            if ((lbits()[lid >> 5] >> (lid & 31u)) & 1u) continue;
          }
          const uint32_t h = (uint32_t)qhead()[lane * D + e];
          if (h < best) {
            best = h;
            be = e;
          }
        }
      }
      const uint32_t m = __reduce_min_sync(kFullMask, best);
      if (m == 0xffffffffu) break;
      started = true;
      const int src = __ffs(__ballot_sync(kFullMask, best == m)) - 1;
      const int e = __shfl_sync(kFullMask, be, src);
      const uint32_t p = xent()[m] >> 5;
      const int32_t nxt = xnext()[m];
      const int pair = src * D + e;
      __syncwarp();
      if (lane == 0) {
        qhead()[pair] = nxt;
        if (nxt < 0) qtail()[pair] = -1;
        if (links) {
          const uint32_t lid = __ldg(A.link + pair);
          lbits()[lid >> 5] |= 1u << (lid & 31u);
        }
      }
      if (nxt < 0 && lane == src) pm &= ~(1u << e);
      sendm |= 1u << src;
      recvm |= 1u << e;
      const tm_t done = t + this->xfer(src, e, op_durbytes(g.ops, p).y, op_xqsucc(g.ops, p).xq);
      if (lane == src) {
        xd = done;
        xdp = p;
        xde = e;
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
        if (td == tx) transfer_done(__ffs(__ballot_sync(kFullMask, xd == td)) - 1, td);
        else intents_arrive((uint32_t)(ik & this->kc.mask));
        if (kMode == kBase) this->last_t = tx;
        arb_due = true;
        t_arb = tx;
        if (status) break;
        continue;
      }
      if (nk == kKeyMax) break;
      if (kMode == kBase) arb_checkpoint(nk);
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
      if (kMode == kBase) this->last_t = (tm_t)this->kc.time(nk);
      start_op(this->kc.op(nk), (tm_t)this->kc.time(nk));
      if (status) break;
    }
    if (!status) drain(kI64Max);
  }

  // -------------------------------------------------------------------------
  // Arbitrated base snapshot.  A checkpoint is taken right before a READY key
  // whose time T_c is past every event handled so far: every transfer event
  // and arbitration before T_c is done (transfer events at a time come before
  // READY keys at that time, and the arbiter runs before the next later
  // event), nothing at T_c or later is.  The simulation part is the base
  // snapshot's (Sim::maybe_checkpoint, after this simulator's own event
  // generation); the arbiter's part goes to the checkpoint's arena.
  // -------------------------------------------------------------------------
  __device__ void arb_checkpoint(uint64_t next_key) {
    const DevBase& B = P.base;
    if (this->ck >= B.nck || this->readypops < this->next_ck) return;
    if (this->kc.time(next_key) <= (int64_t)this->last_t) return;
    generate();  // the simulation checkpoint then finds no started op left to generate
    const int c = this->ck;
    this->maybe_checkpoint(next_key);
    if (this->ck > c && B.ck_time[c] != kI64Max) save_arb(c);
  }

  __device__ uint8_t* arena(int c) const { return A.ck.arena + (int64_t)c * A.ck.bytes; }

  // The base runs with 64-bit times, so every per-op array has the arena's
  // element size and is copied as bytes (each region of the slot and of the
  // arena is padded to 256 bytes).
  __device__ void save_arb(int c) {
    static_assert(kMode != kBase || !kT32, "the base snapshot keeps 64-bit times");
    const unsigned lane = lane_id();
    uint8_t* a = arena(c);
    const ArbCk& K = A.ck;
    const int64_t n = g.n;
    warp_copy16<16>(a + K.off_cnt, cnt(), 4 * n);
    warp_copy16<16>(a + K.off_rmax, rmax(), 8 * n);
    warp_copy16<16>(a + K.off_refs, refs(), 4 * n);
    warp_copy16<16>(a + K.off_rmask, rmask(), 4 * n);
    warp_copy16<16>(a + K.off_nextop, nextop(), 4 * n);
    warp_copy16<16>(a + K.off_hold, this->holdb, 8 * n);
    warp_copy16<16>(a + K.off_xent, xent(), 4 * (int64_t)nx);
    warp_copy16<16>(a + K.off_xnext, xnext(), 4 * (int64_t)nx);
    for (int x = lane; x < g.D * g.D; x += 32) {
      reinterpret_cast<int32_t*>(a + K.off_qhead)[x] = qhead()[x];
      reinterpret_cast<int32_t*>(a + K.off_qtail)[x] = qtail()[x];
    }
    int64_t* ls = reinterpret_cast<int64_t*>(a + K.off_lanes) + 7 * lane;
    ls[0] = pm;
    ls[1] = (int64_t)xd;
    ls[2] = xdp;
    ls[3] = xde;
    ls[4] = fh;
    ls[5] = ft;
    ls[6] = (int64_t)fa;
    int64_t* w = reinterpret_cast<int64_t*>(a + K.off_warp);
    if (lane == 0) {
      w[0] = nx;
      w[1] = xev;
      w[2] = sendm;
      w[3] = recvm;
    }
    reinterpret_cast<uint32_t*>(w + 4)[lane] = lbits()[lane];
    __syncwarp();
  }

  // A base time (int64) in this kernel's time type; the base's "never" maps
  // to this kernel's.
  static __device__ __forceinline__ tm_t narrow_time(int64_t v) {
    return v >= (int64_t)kNever ? kNever : (tm_t)v;
  }

  // An arena's 64-bit times into this kernel's time type, four loads in
  // flight per lane.
  static __device__ void narrow_times(tm_t* dst, const int64_t* src, int n) {
    int x = (int)lane_id();
    for (; x + 96 < n; x += 128) {
      const int64_t a = src[x], b = src[x + 32], c = src[x + 64], e = src[x + 96];
      dst[x] = narrow_time(a);
      dst[x + 32] = narrow_time(b);
      dst[x + 64] = narrow_time(c);
      dst[x + 96] = narrow_time(e);
    }
    for (; x < n; x += 32) dst[x] = narrow_time(src[x]);
  }

  __device__ void restore_arb(int c) {
    const unsigned lane = lane_id();
    const uint8_t* a = arena(c);
    const ArbCk& K = A.ck;
    const int64_t n = g.n;
    warp_copy16(cnt(), a + K.off_cnt, 4 * n);
    warp_copy16(refs(), a + K.off_refs, 4 * n);
    warp_copy16(rmask(), a + K.off_rmask, 4 * n);
    warp_copy16(nextop(), a + K.off_nextop, 4 * n);
    if (kT32) {
      narrow_times(rmax(), reinterpret_cast<const int64_t*>(a + K.off_rmax), g.n);
      narrow_times(this->holdb, reinterpret_cast<const int64_t*>(a + K.off_hold), g.n);
    } else {
      warp_copy16(rmax(), a + K.off_rmax, 8 * n);
      warp_copy16(this->holdb, a + K.off_hold, 8 * n);
    }
    const int64_t* w = reinterpret_cast<const int64_t*>(a + K.off_warp);
    nx = (int32_t)w[0];
    xev = (int32_t)w[1];
    sendm = (uint32_t)w[2];
    recvm = (uint32_t)w[3];
    lbits()[lane] = reinterpret_cast<const uint32_t*>(w + 4)[lane];
    warp_copy16(xent(), a + K.off_xent, 4 * (int64_t)nx);
    warp_copy16(xnext(), a + K.off_xnext, 4 * (int64_t)nx);
    for (int x = lane; x < g.D * g.D; x += 32) {
      qhead()[x] = reinterpret_cast<const int32_t*>(a + K.off_qhead)[x];
      qtail()[x] = reinterpret_cast<const int32_t*>(a + K.off_qtail)[x];
    }
    const int64_t* ls = reinterpret_cast<const int64_t*>(a + K.off_lanes) + 7 * lane;
    pm = (uint32_t)ls[0];
    xd = narrow_time(ls[1]);
    xdp = (uint32_t)ls[2];
    xde = (int)ls[3];
    fh = (int32_t)ls[4];
    ft = (int32_t)ls[5];
    fa = narrow_time(ls[6]);
    arb_due = false;
    t_arb = 0;
    __syncwarp();
  }

  // Remote accelerators of p's successors under placement rw (uniform).
  __device__ uint32_t remote_set(uint32_t p, const uint8_t* rw) const {
    const XqSucc xs = op_xqsucc(g.ops, p);
    const int dp = rw[p];
    uint32_t m = 0u;
    for (uint32_t u = lane_id(); u < xs.nsucc; u += 32) {
      const int dj = rw[__ldg(g.succ + xs.succ_off + u)];
      if (dj != dp) m |= 1u << dj;
    }
    return __reduce_or_sync(kFullMask, m);
  }

  // A listed consumer of p on p's accelerator under placement rw (uniform).
  __device__ bool local_consumer(uint32_t p, const uint8_t* rw) const {
    const uint4 cs = op_cons(g.ops, p);
    const XqSucc xs = op_xqsucc(g.ops, p);
    const bool all = (cs.w & kAllCons) != 0;
    const uint32_t* lst = all ? g.succ + xs.succ_off : g.cons + cs.x;
    const uint32_t nl = all ? xs.nsucc : cs.y;
    const int dp = rw[p];
    bool f = false;
    for (uint32_t u = lane_id(); u < nl; u += 32) f |= rw[__ldg(lst + u)] == dp;
    return __any_sync(kFullMask, f);
  }

  // Op p (started before the resume point, finishing at or after it) in the
  // FIFO of coming intents of its accelerator d, kept in finish order: insert
  // (want) or remove.  The list runs from the head to the tail through
  // nextop (the tail's link is not kept).  Uniform call; lane d owns the head
  // and tail.
  __device__ void fifo_set(uint32_t p, int d, bool want) {
    const unsigned lane = lane_id();
    int32_t h = __shfl_sync(kFullMask, fh, d);
    int32_t t = __shfl_sync(kFullMask, ft, d);
    int32_t* nxp = nextop();
    const tm_t fp = this->fin(p);
    int32_t prev = -1, cur = h;
    bool found = false;
    for (int guard = 0; cur >= 0 && guard <= g.n; ++guard) {
      if (cur == (int32_t)p) {
        found = true;
        break;
      }
      if (this->fin((uint32_t)cur) > fp) break;
      prev = cur;
      cur = cur == t ? -1 : nxp[cur];
    }
    if (want == found) return;
    if (want) {  // link p between prev and cur
      if (lane == 0) {
        nxp[p] = cur;
        if (prev >= 0) nxp[prev] = (int32_t)p;
      }
      if (prev < 0) h = (int32_t)p;
      if (cur < 0) t = (int32_t)p;
    } else {  // unlink p (cur == p)
      const int32_t after = (int32_t)p == t ? -1 : nxp[p];
      if (lane == 0 && prev >= 0) nxp[prev] = after;
      if (prev < 0) h = after;
      if (t == (int32_t)p) t = prev;
    }
    __syncwarp();
    if ((int)lane == d) {
      fh = h;
      ft = h < 0 ? -1 : t;
      fa = h < 0 ? kNever : this->fin((uint32_t)h);
    }
    __syncwarp();
  }

  // One incremental candidate resumed from the arbitrated base snapshot.
  // Results equal the full arbitrated simulation of the moved placement
  // (Sec. 3.5.2); the fix-ups below are what the moves change in the state
  // at the checkpoint T_c <= T0: a moved op's inputs counted so far (only
  // predecessors local under the new placement and already started count; no
  // remote one has finished) and its READY key; and for every predecessor p
  // of a moved op that started before T_c (it finishes at or after T0, so
  // none of its intents, transfers or receive buffers exist yet): its remote
  // set, the holds on its copy, its place in its accelerator's FIFO of coming
  // intents, and whether its copy's release is already logged.
  __device__ void inc_candidate(int64_t k, uint8_t* crow) {
    const DevBase& B = P.base;
    const unsigned lane = lane_id();
    const int32_t m0 = P.move_off[k], m1 = P.move_off[k + 1];
    const int32_t nm = m1 - m0;
    // validate the move list (range, then an op moved twice)
    bool bad = false, dup = false;
    for (int32_t m = m0 + (int32_t)lane; m < m1; m += 32)
      bad |= P.move_op[m] < 0 || P.move_op[m] >= g.n || P.move_dev[m] >= g.D;
    bad = __any_sync(kFullMask, bad);
    if (!bad)
      for (int32_t m = m0 + (int32_t)lane; m < m1; m += 32)
        for (int32_t m2 = m + 1; m2 < m1 && !dup; ++m2) dup = P.move_op[m2] == P.move_op[m];
    dup = __any_sync(kFullMask, dup);
    if (B.status[0] != GMG_SIM_OK) {
      this->write_invalid(k, GMG_SIM_BADBASE);
      return;
    }
    if (bad || dup) {
      this->write_invalid(k, bad ? GMG_SIM_MOVE_RANGE : GMG_SIM_MOVE_DUP);
      return;
    }
    warp_copy16(crow, B.row, B.ld);
    __syncwarp();
    uint64_t t0 = kKeyMax;
    for (int t = lane; t < nm; t += 32) {
      const int32_t op = P.move_op[m0 + t];
      const uint8_t dvc = P.move_dev[m0 + t];
      crow[op] = dvc;
      if (dvc != B.row[op]) {
        const RelPred rp = op_relpred(g.ops, (uint32_t)op);
        uint64_t tx = (uint64_t)rp.rel;
        if (rp.npred) {
          tx = kKeyMax;
          for (uint32_t u = 0; u < rp.npred; ++u) {
            const uint64_t fp = (uint64_t)B.fb[__ldg(g.pred + rp.pred_off + u) & kIdMask];
            tx = fp < tx ? fp : tx;
          }
        }
        t0 = tx < t0 ? tx : t0;
      }
    }
    t0 = warp_min_u64(t0);
    __syncwarp();
    row = crow;
    const DevOut& o = P.out;
    if (t0 == kKeyMax) {  // no effective move: the base results
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
      const int ts = this->trace_slot(k);
      if (ts >= 0)
        for (int x = lane; x < g.n; x += 32) {
          o.trace_finish[(int64_t)ts * g.n + x] = B.fb[x];
          o.trace_start[(int64_t)ts * g.n + x] =
              B.fb[x] - this->dur_of((uint32_t)x, B.row[x], op_durbytes(g.ops, (uint32_t)x).x);
        }
      return;
    }
    this->T0 = (tm_t)t0;
    int best = -1;
    for (int c = lane; c < B.nck; c += 32)
      if (B.ck_time[c] <= (int64_t)t0) best = c;
    const int c = __reduce_max_sync(kFullMask, best);
    const int64_t* sc = B.ck_scalars + (int64_t)c * 8;
    const int qsz = (int)sc[0];
    const int msz = (int)sc[7];
    if (qsz + nm > this->q.cap || msz + nm > this->log.cap) {
      this->write_invalid(k, GMG_SIM_QUEUE);
      return;
    }
    // the simulation state of checkpoint c
    this->Tc = (tm_t)B.ck_time[c];
    this->rootptr = (int)sc[1];
    this->load_root();
    this->score = sc[2];
    this->makespan = (tm_t)sc[3];
    this->vflag = (int32_t)sc[4];
    this->vt = sc[5];
    this->vop = (int32_t)(sc[6] >> 32);
    this->vdev = (int32_t)(sc[6] & 0xffffffff);
    this->iters = 0;
    this->nev = 0;
    this->readypops = 0;
    this->last_t = -1;
    status = GMG_SIM_OK;
    this->rk_reg = kKeyMax;
    this->opn = 0;
    this->dv.load(B.ck_dev + (int64_t)c * 3 * g.D);
    for (int r = lane; r < g.R; r += 32) this->creq[r] = B.ck_creq[(int64_t)c * g.R + r];
    this->fill_fin();
    restore_arb(c);
    // READY keys, except those of moved ops (recomputed below)
    int nq = 0;
    for (int c0 = 0; c0 < qsz; c0 += 32) {
      const int x = c0 + (int)lane;
      const bool v = x < qsz;
      const uint64_t key = v ? B.ck_qkey[(int64_t)c * B.ckq + x] : 0ull;
      const uint32_t op = this->kc.op(key);
      const bool keep = v && crow[op] == B.row[op];
      const uint32_t bal = __ballot_sync(kFullMask, keep);
      if (keep) *this->q.kp(nq + __popc(bal & lanes_below())) = key;
      nq += __popc(bal);
    }
    // logged HBM events, except the release of a moved op's predecessor's own
    // copy (regenerated below if it is due)
    int outn = 0;
    for (int c0 = 0; c0 < msz; c0 += 32) {
      const int x = c0 + (int)lane;
      const bool v = x < msz;
      const uint64_t e = v ? B.ck_mkey[(int64_t)c * B.ckm + x] : 0ull;
      bool keep = v;
      if (v && this->kc.cls(e) == kFree) {
        const uint32_t op = this->kc.op(e);
        const int dev = (int)(e >> this->ds);
        if (dev == B.row[op]) {
          const XqSucc xs = op_xqsucc(g.ops, op);
          for (uint32_t u = 0; u < xs.nsucc && keep; ++u) {
            const uint32_t j = __ldg(g.succ + xs.succ_off + u);
            keep = crow[j] == B.row[j];
          }
        }
      }
      const uint32_t bal = __ballot_sync(kFullMask, keep);
      if (keep) *this->log.kp(outn + __popc(bal & lanes_below())) = e;
      outn += __popc(bal);
    }
    this->log.n = outn;
    __syncwarp();
    // every effective move: the moved op's inputs, its predecessors' state
    for (int32_t t = 0; t < nm; ++t) {
      const uint32_t x = (uint32_t)P.move_op[m0 + t];
      if (crow[x] == B.row[x]) continue;
      const RelPred rp = op_relpred(g.ops, x);
      // inputs of x present so far: started predecessors local under crow
      int32_t cx = 0;
      uint64_t rx = 0;
      for (uint32_t u = lane; u < rp.npred; u += 32) {
        const uint32_t p = __ldg(g.pred + rp.pred_off + u) & kIdMask;
        if (this->base_time(this->rb, p) < this->Tc && crow[p] == crow[x]) {
          ++cx;
          const uint64_t fp = (uint64_t)this->base_time(this->fb, p);
          rx = fp > rx ? fp : rx;
        }
      }
      cx = (int32_t)__reduce_add_sync(kFullMask, (uint32_t)cx);
      rx = warp_max_u64(rx);
      if (lane == 0) {
        cnt()[x] = cx;
        rmax()[x] = (tm_t)rx;
      }
      if (rp.npred > 0 && (uint32_t)cx == rp.npred) {
        const tm_t rel = (tm_t)rp.rel;
        const tm_t rj = rel > (tm_t)rx ? rel : (tm_t)rx;
        if (lane == 0) *this->q.kp(nq) = this->kc.make(rj, kReady, x);
        ++nq;
      }
      // started predecessors: remote set, holds, FIFO, own copy's release;
      // each predecessor once, by its first moved successor in this list
      for (uint32_t u = 0; u < rp.npred; ++u) {
        const uint32_t p = __ldg(g.pred + rp.pred_off + u) & kIdMask;
        if (this->base_time(this->rb, p) >= this->Tc) continue;
        bool first = true;
        for (int32_t t2 = 0; t2 < t && first; ++t2) {
          const uint32_t x2 = (uint32_t)P.move_op[m0 + t2];
          if (crow[x2] == B.row[x2]) continue;
          const RelPred r2 = op_relpred(g.ops, x2);
          for (uint32_t u2 = 0; u2 < r2.npred; ++u2)
            if ((__ldg(g.pred + r2.pred_off + u2) & kIdMask) == p) {
              first = false;
              break;
            }
        }
        if (!first) continue;
        const uint32_t rc = remote_set(p, crow);
        const bool lc = local_consumer(p, crow);
        const int dp = crow[p];
        const int32_t holds = 1 + __popc(rc) - (lc ? 0 : 1);
        const tm_t fp = this->fin(p);
        if (lane == 0) {
          rmask()[p] = rc;
          refs()[p] = holds;
          this->holdb[p] = fp;
        }
        __syncwarp();
        fifo_set(p, dp, rc != 0u);
        this->log_event(lane == 0 && holds == 0, this->kc.make(fp, kFree, p), dp);
      }
    }
    this->q.size = nq;
    this->q.heapify();
    refresh_done();
    refresh_intent();
    run();
    this->finish(k);
  }
};

template <bool kT32, bool kTypes>
__global__ void __launch_bounds__(128, 7) sim_arb_kernel(const __grid_constant__ ArbParams A) {
  extern __shared__ __align__(16) uint8_t smem[];
  const unsigned wib = threadIdx.x >> 5;
  const int64_t slot = (int64_t)blockIdx.x * (blockDim.x >> 5) + wib;
  const int64_t nslots = (int64_t)gridDim.x * (blockDim.x >> 5);
  ArbSim<kT32, kTypes> S(A);
  setup_slot(S, A.P, wib, slot, smem);
  S.setup_arb(slot, smem + A.smem_std + (size_t)wib * A.smem_arb);
  for (int64_t k = slot; k < A.P.K; k += nslots) {
    S.row = A.P.place + k * A.P.ld;
    if (A.pre_status) {
      const int32_t ps = A.pre_status[k];
      if (ps != GMG_SIM_OK) {
        S.write_invalid(k, ps);
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

// The arbitrated base snapshot: the base placement simulated once (64-bit
// times) with checkpoints of the simulation and the arbiter.
template <bool kTypes>
__global__ void __launch_bounds__(32) sim_arb_base_kernel(const __grid_constant__ ArbParams A) {
  extern __shared__ __align__(16) uint8_t smem[];
  ArbSim<false, kTypes, kBase> S(A);
  setup_slot(S, A.P, 0, 0, smem);
  S.setup_arb(0, smem + A.smem_std);
  const DevBase& B = A.P.base;
  const unsigned lane = lane_id();
  warp_prefetch_l2(A.P.g.ws, A.P.g.ws_bytes);
  for (int c = lane * 16; c < B.ld; c += 512)
    *reinterpret_cast<uint4*>(B.row + c) = *reinterpret_cast<const uint4*>(A.P.place + c);
  for (int c = lane; c < B.nck; c += 32) B.ck_time[c] = kI64Max;
  S.fbuf = B.fb;
  S.row = A.P.place;
  __syncwarp();
  if (S.row_has_bad_device(A.P.place)) {
    if (lane == 0) B.status[0] = GMG_SIM_BADDEV;
    return;
  }
  S.reset_arb();
  S.ck = 0;
  S.next_ck = 0;
  S.arb_checkpoint(S.kc.make(0, kReady, 0));  // checkpoint 0: the initial state
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

// Incremental candidates resumed from the arbitrated base snapshot.
template <bool kT32, bool kTypes>
__global__ void __launch_bounds__(128, 7) sim_arb_inc_kernel(const __grid_constant__ ArbParams A) {
  extern __shared__ __align__(16) uint8_t smem[];
  const unsigned wib = threadIdx.x >> 5;
  const int64_t slot = (int64_t)blockIdx.x * (blockDim.x >> 5) + wib;
  ArbSim<kT32, kTypes, kInc> S(A);
  setup_slot(S, A.P, wib, slot, smem);
  S.setup_arb(slot, smem + A.smem_std + (size_t)wib * A.smem_arb);
  S.rb = A.P.base.rb;
  S.fb = A.P.base.fb;
  uint8_t* crow = A.P.scratch + slot * A.P.slot_bytes + A.P.off_row;
  for (int64_t k = take_candidate(A.P.next_k); k < A.P.K; k = take_candidate(A.P.next_k)) S.inc_candidate(k, crow);
}

// One warp per incremental candidate: check the move list (an op or device
// out of range, then an op moved twice), copy the base row, apply the moves.
// A base row with a device out of range makes every candidate BADBASE.
__global__ void __launch_bounds__(128) expand_moves_kernel(const uint8_t* base_row, const int32_t* base_status,
                                                           int32_t ld, int32_t n, int32_t D, const int32_t* off,
                                                           const int32_t* op, const uint8_t* dev, int32_t K,
                                                           uint8_t* rows, int32_t* status) {
  const unsigned lane = lane_id();
  const int64_t w0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  // Only a base row with a device out of range invalidates the moved rows;
  // the base's own (pure-latency) simulation status -- a queue or loop limit
  // of that run -- says nothing about the arbitrated simulations of the
  // moved placements, which run in full.
  const bool base_ok = *base_status != GMG_SIM_BADDEV;
  for (int64_t k = w0; k < K; k += nw) {
    const int32_t a = off[k], b = off[k + 1];
    int32_t st = base_ok ? GMG_SIM_OK : GMG_SIM_BADBASE;
    if (st == GMG_SIM_OK) {
      bool bad = false;
      for (int32_t m = a + (int32_t)lane; m < b; m += 32) bad |= op[m] < 0 || op[m] >= n || dev[m] >= D;
      if (__any_sync(kFullMask, bad)) st = GMG_SIM_MOVE_RANGE;
    }
    if (st == GMG_SIM_OK) {
      bool dup = false;
      for (int32_t m = a + (int32_t)lane; m < b; m += 32)
        for (int32_t m2 = m + 1; m2 < b && !dup; ++m2) dup = op[m2] == op[m];
      if (__any_sync(kFullMask, dup)) st = GMG_SIM_MOVE_DUP;
    }
    uint8_t* rw = rows + k * (int64_t)ld;
    warp_copy16(rw, base_row, ld);
    __syncwarp();
    if (st == GMG_SIM_OK)
      for (int32_t m = a + (int32_t)lane; m < b; m += 32) rw[op[m]] = dev[m];
    if (lane == 0) status[k] = st;
    __syncwarp();
  }
}

}  // namespace

cudaError_t launch_expand_moves(const uint8_t* base_row, const int32_t* base_status, int32_t ld, int32_t n,
                                int32_t D, const int32_t* off, const int32_t* op, const uint8_t* dev, int32_t K,
                                uint8_t* rows, int32_t* status, cudaStream_t st) {
  const int blocks = (int)std::min<int64_t>(((int64_t)K + 3) / 4, 152 * 16);
  expand_moves_kernel<<<std::max(blocks, 1), 128, 0, st>>>(base_row, base_status, ld, n, D, off, op, dev, K,
                                                           rows, status);
  return cudaGetLastError();
}

const void* arb_kernel_ptr(bool t32, bool types) {
  if (t32) return types ? (const void*)sim_arb_kernel<true, true> : (const void*)sim_arb_kernel<true, false>;
  return types ? (const void*)sim_arb_kernel<false, true> : (const void*)sim_arb_kernel<false, false>;
}

cudaError_t launch_arb(bool t32, bool types, const ArbParams& A, int grid, int block, size_t smem,
                       cudaStream_t st) {
  void* args[] = {const_cast<ArbParams*>(&A)};
  return cudaLaunchKernel(arb_kernel_ptr(t32, types), dim3(grid), dim3(block), args, smem, st);
}

const void* arb_base_kernel_ptr(bool types) {
  return types ? (const void*)sim_arb_base_kernel<true> : (const void*)sim_arb_base_kernel<false>;
}

const void* arb_inc_kernel_ptr(bool t32, bool types) {
  if (t32) return types ? (const void*)sim_arb_inc_kernel<true, true> : (const void*)sim_arb_inc_kernel<true, false>;
  return types ? (const void*)sim_arb_inc_kernel<false, true> : (const void*)sim_arb_inc_kernel<false, false>;
}

cudaError_t launch_arb_base(bool types, const ArbParams& A, size_t smem, cudaStream_t st) {
  void* args[] = {const_cast<ArbParams*>(&A)};
  return cudaLaunchKernel(arb_base_kernel_ptr(types), dim3(1), dim3(32), args, smem, st);
}

cudaError_t launch_arb_inc(bool t32, bool types, const ArbParams& A, int grid, int block, size_t smem,
                           cudaStream_t st) {
  void* args[] = {const_cast<ArbParams*>(&A)};
  return cudaLaunchKernel(arb_inc_kernel_ptr(t32, types), dim3(grid), dim3(block), args, smem, st);
}

}  // namespace gsim
