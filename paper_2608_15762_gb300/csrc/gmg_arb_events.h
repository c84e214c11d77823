// Parts shared by the two arbitrated-transfer simulators (gmgsim_arb.cu, at
// most 32 accelerators with transfer state in lane registers; gmgsim_arbw.cu,
// 33 to 256 accelerators with it in per-warp tables): counting an op's inputs
// as they arrive, the holds on a producer's own copy, and the HBM events of
// the ops started since the last generation (Sec. 3.5.2: a receive buffer is
// allocated when its transfer starts, a producer's copy is released once its
// last local consumer has finished and every outgoing transfer has arrived).
//
// ArbEvents<Self, SimBase> sits between the pure-latency simulator SimBase and
// the kernel's own simulator Self, which provides the per-op scratch arrays
// cnt() (inputs present), rmax() (latest arrival so far) and refs() (holds
// left on the op's own copy).
#pragma once

#include "gmgsim_sim.cuh"

namespace gsim {
namespace {

template <class Self, class SimBase>
struct ArbEvents : SimBase {
  using tm_t = typename SimBase::tm_t;
  __device__ explicit ArbEvents(const SimParams& p) : SimBase(p) {}
  __device__ __forceinline__ const Self& self() const { return *static_cast<const Self*>(this); }

  // One more input of op j present at time a (per lane); true if it was the
  // last, with its ready time in rj.
  __device__ __forceinline__ bool add_input(uint32_t j, tm_t a, tm_t& rj) const {
    int32_t* cp = self().cnt() + j;
    tm_t* mp = self().rmax() + j;
    const int32_t c = *cp + 1;
    *cp = c;
    const tm_t m = c == 1 ? a : (*mp > a ? *mp : a);
    *mp = m;
    const RelPred jp = op_relpred(this->g.ops, j);
    if ((uint32_t)c != jp.npred) return false;
    const tm_t rel = (tm_t)jp.rel;
    rj = rel > m ? rel : m;
    return true;
  }

  __device__ __forceinline__ void push_readies(bool rdy, tm_t rj, uint32_t j) {
    uint32_t m = __ballot_sync(kFullMask, rdy);
    while (m) {
      const int src = __ffs(m) - 1;
      m &= m - 1;
      this->push_ready(__shfl_sync(kFullMask, this->kc.make(rj, kReady, j), src));
    }
  }

  // One hold on op p's own copy (on accelerator dp) ends at time v (per
  // lane; `want`: this lane releases one).  Logs the copy's release when it
  // was the last hold.
  __device__ __forceinline__ void drop_hold(bool want, uint32_t p, tm_t v, int dp) {
    bool last = false;
    tm_t h = v;
    if (want) {
      int32_t* rp = self().refs() + p;
      const int32_t left = *rp - 1;
      *rp = left;
      const tm_t o = this->holdb[p];
      h = o > v ? o : v;
      this->holdb[p] = h;
      last = left == 0;
    }
    this->log_event(last, this->kc.make(h, kFree, p), dp);
  }

  // HBM events of the ops started since the last generation, one op per
  // lane: the own copy allocated at s; the op's local hold on its own copy
  // ends at f if no listed consumer is local; every held input whose last
  // local listed consumer this op is gets released at f (a receive copy) or
  // loses its local hold (the producer's own copy).
  __device__ void generate() {
    const unsigned lane = lane_id();
    for (int c0 = 0; c0 < this->opn; c0 += 32) {
      const int idx = c0 + (int)lane;
      const bool v = idx < this->opn;
      const uint32_t x = v ? this->oplog[idx] : 0u;
      longlong2 db = make_longlong2(0, 0);
      uint4 ls = make_uint4(0, 0, 0, 0), cs = make_uint4(0, 0, 0, 0);
      int d = 0;
      tm_t f = 0;
      if (v) {
        db = op_durbytes(this->g.ops, x);
        ls = op_lists(this->g.ops, x);
        cs = op_cons(this->g.ops, x);
        d = this->row[x];
        f = this->fbuf[x];
      }
      this->log_event(v, this->kc.make(f - (tm_t)this->dur_of(x, d, db.x), kAlloc, x), d);
      bool localc = false;
      if (v) {
        const bool all = (cs.w & kAllCons) != 0;
        const uint32_t* lst = all ? this->g.succ + ls.x : this->g.cons + cs.x;
        const uint32_t nl = all ? ls.y : cs.y;
        for (uint32_t w = 0; w < nl; ++w)
          if (this->row[__ldg(lst + w)] == d) {
            localc = true;
            break;
          }
      }
      drop_hold(v && !localc, x, f, d);
      __syncwarp();
      const uint32_t npx = ls.w;
      const uint32_t maxp = __reduce_max_sync(kFullMask, npx);
      for (uint32_t u = 0; u < maxp; ++u) {
        bool rel = false;
        uint32_t p = 0;
        if (u < npx) {
          const uint2 ps = __ldg(this->g.predsib + ls.z + u);
          p = ps.x & kIdMask;
          if (ps.x & kHoldBit) {
            const uint32_t sb = ps.y;
            if (sb == kSibNone) {
              rel = true;
            } else if (sb != kSibMany && (sb & kSibLater)) {
              rel = this->row[sb & ~kSibLater] != d;  // the other consumer finishes later
            } else if (sb != kSibMany) {
              const tm_t fs = this->fin(sb);
              rel = !(this->row[sb] == d && !(fs > 0 && fs < f));
            } else {
              const XqSucc px = op_xqsucc(this->g.ops, p);
              const uint4 pcs = op_cons(this->g.ops, p);
              const bool all = (pcs.w & kAllCons) != 0;
              const uint32_t* lst = all ? this->g.succ + px.succ_off : this->g.cons + pcs.x;
              const uint32_t nl = all ? px.nsucc : pcs.y;
              rel = true;
              for (uint32_t w = 0; w < nl; ++w) {
                const uint32_t c = __ldg(lst + w);
                const tm_t fc = c != x ? this->fin(c) : 0;
                if (c != x && this->row[c] == d && !(fc > 0 && fc < f)) {
                  rel = false;
                  break;
                }
              }
            }
          }
        }
        const bool own = rel && this->row[p] == d;
        this->log_event(rel && !own, this->kc.make(f, kFree, p), d);
        drop_hold(own, p, f, d);
      }
    }
    this->opn = 0;
    __syncwarp();
  }

  __device__ void drain(int64_t t_next) {
    generate();
    this->opn = 0;  // generate() emptied the op log; the base drain's own call is then a no-op
    SimBase::drain(t_next);
  }
};

}  // namespace
}  // namespace gsim
