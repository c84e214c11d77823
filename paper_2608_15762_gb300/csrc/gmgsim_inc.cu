// sim_incremental kernels: K move lists against a base snapshot, one warp per
// candidate.
#include "gmgsim_sim.cuh"

namespace gsim {
namespace {

// ---------------------------------------------------------------------------
// sim_incremental: K move lists against the base.
// ---------------------------------------------------------------------------
template <bool kReg, bool kKey, bool kT32, bool kTypes, bool kBatch>
__device__ void regen(Sim<kReg, kInc, kKey, kT32, kTypes, kBatch>& S, uint32_t p);

template <bool kReg, bool kKey, bool kT32, bool kTypes, bool kBatch>
__device__ void inc_candidate(Sim<kReg, kInc, kKey, kT32, kTypes, kBatch>& S, const SimParams& P, int64_t k, uint8_t* crow) {
  using tm_t = typename Sim<kReg, kInc, kKey, kT32, kTypes, kBatch>::tm_t;
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
  if (B.status[0] != GMG_SIM_OK) {
    S.write_invalid(k, GMG_SIM_BADBASE);
    return;
  }
  if (bad_range || dup) {
    S.write_invalid(k, bad_range ? GMG_SIM_MOVE_RANGE : GMG_SIM_MOVE_DUP);
    return;
  }
  // The candidate's placement = base + moves.
  warp_copy16(crow, B.row, B.ld);
  __syncwarp();
  uint64_t t0 = kKeyMax;
  for (int t = lane; t < nm; t += 32) {
    const int32_t op = P.move_op[m0 + t];
    const uint8_t dvc = P.move_dev[m0 + t];
    crow[op] = dvc;
    if (dvc != B.row[op]) {
      const RelPred rp = op_relpred(g.ops, (uint32_t)op);
      const uint4 ls = make_uint4(0u, 0u, rp.pred_off, rp.npred);
      uint64_t tx;
      if (ls.w == 0) {
        tx = (uint64_t)rp.rel;
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
        o.trace_start[(int64_t)ts * g.n + x] =
            B.fb[x] - S.dur_of((uint32_t)x, B.row[x], op_durbytes(g.ops, (uint32_t)x).x);
      }
    return;
  }
  S.T0 = (tm_t)t0;
  // Latest recorded resume point at or before T0.
  int best = -1;
  for (int c = lane; c < B.nck; c += 32)
    if (B.ck_time[c] <= S.T0) best = c;
  const int c = __reduce_max_sync(kFullMask, best);
  const int64_t* sc = B.ck_scalars + (int64_t)c * 8;
  const int qsz = (int)sc[0];
  const int msz = (int)sc[7];
  if (qsz > S.q.cap || msz > S.log.cap) {
    S.write_invalid(k, GMG_SIM_QUEUE);
    return;
  }
  // Restore the simulator state of checkpoint c.
  S.Tc = (tm_t)B.ck_time[c];
  S.rootptr = (int)sc[1];
  S.load_root();
  S.score = sc[2];
  S.makespan = (tm_t)sc[3];
  S.vflag = (int32_t)sc[4];
  S.vt = sc[5];
  S.vop = (int32_t)(sc[6] >> 32);
  S.vdev = (int32_t)(sc[6] & 0xffffffff);
  S.iters = 0;
  S.nev = 0;
  S.readypops = 0;
  S.last_t = -1;
  S.status = GMG_SIM_OK;
  S.rk_reg = kKeyMax;
  S.opn = 0;
  S.dv.load(B.ck_dev + (int64_t)c * 3 * g.D);
  for (int r = lane; r < g.R; r += 32) S.creq[r] = B.ck_creq[(int64_t)c * g.R + r];
  // ops started before T_c are those with base ready time < T_c: they keep
  // their base finish; the others start with no finish time
  S.fill_fin();
  // READY keys at T_c; a moved op's key is recomputed (its inputs' transfer
  // times change; its predecessors all finished before T_c).
  for (int x = lane; x < qsz; x += 32) {
    uint64_t key = B.ck_qkey[(int64_t)c * B.ckq + x];
    const uint32_t op = S.rq.op(key);
    if (crow[op] != B.row[op]) {
      const int dx = crow[op];
      const RelPred rp = op_relpred(g.ops, op);
      const uint4 ls = make_uint4(0u, 0u, rp.pred_off, rp.npred);
      int64_t rx = rp.rel;
      for (uint32_t u = 0; u < ls.w; ++u) {
        const uint32_t p = __ldg(g.pred + ls.z + u) & kIdMask;
        const int dp = crow[p];
        int64_t a = S.fb[p];
        if (dp != dx) a += S.xfer(dp, dx, op_durbytes(g.ops, p).y, op_xqsucc(g.ops, p).xq);
        rx = a > rx ? a : rx;
      }
      key = S.rq.make(rx, op, kBatch ? dur_class(S.dur_of(op, dx, op_durbytes(g.ops, op).x)) : 0u);
    }
    *S.q.kp(x) = key;
  }
  S.q.size = qsz;
  // Logged HBM events at T_c, except those of an op p with a moved
  // successor: the receiving accelerators and last consumers of p's output
  // changed (its receive allocations and releases all happen at times
  // >= f_p >= T0), so they are regenerated below.
  int outn = 0;
  for (int c0 = 0; c0 < msz; c0 += 32) {
    const int idx = c0 + (int)lane;
    const bool v = idx < msz;
    uint64_t e = 0;
    uint8_t dv8 = 0;
    bool keep = false;
    if (v) {
      e = B.ck_mkey[(int64_t)c * B.ckm + idx];
      if (!kKey) dv8 = B.ck_mdev[(int64_t)c * B.ckm + idx];
      keep = true;
      const uint32_t cls = S.kc.cls(e), op = S.kc.op(e);
      const int dev = kKey ? (int)(e >> S.ds) : (int)dv8;
      const uint4 ls = op_lists(g.ops, op);
      bool moved_succ = false;
      for (uint32_t u = 0; u < ls.y && !moved_succ; ++u) {
        const uint32_t j = __ldg(g.succ + ls.x + u);
        moved_succ = crow[j] != B.row[j];
      }
      if (moved_succ && (cls == kFree || dev != B.row[op])) keep = false;
    }
    const uint32_t bal = __ballot_sync(kFullMask, keep);
    if (keep) {
      const int pos = outn + __popc(bal & lanes_below());
      *S.log.kp(pos) = e;
      if (!kKey) *S.log.dp(pos) = dv8;
    }
    outn += __popc(bal);
  }
  S.log.n = outn;
  __syncwarp();
  // Regenerate the HBM events of every predecessor p (finished before T_c)
  // of a moved op under the candidate placement; each p once, by its
  // smallest-id moved successor.
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

// HBM events of op p (finished before the resume point) under the candidate
// placement: receive copies on every remote accelerator of its successors
// (allocated at f_p), and the releases that are already determined because
// every listed consumer on that accelerator has finished.
template <bool kReg, bool kKey, bool kT32, bool kTypes, bool kBatch>
__device__ void regen(Sim<kReg, kInc, kKey, kT32, kTypes, kBatch>& S, uint32_t p) {
  const DevGmg& g = S.g;
  const unsigned lane = lane_id();
  const int64_t fp = S.fb[p];
  const int dp = S.row[p];
  const int64_t pb = op_durbytes(g.ops, p).y, pxq = op_xqsucc(g.ops, p).xq;
  const uint4 pls = op_lists(g.ops, p);
  const uint4 pcs = op_cons(g.ops, p);
  const bool all = (pcs.w & kAllCons) != 0;
  const uint32_t* lst = all ? g.succ + pls.x : g.cons + pcs.x;
  const uint32_t nl = all ? pls.y : pcs.y;
  int64_t hm = fp;
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
    const int64_t hl = (int64_t)warp_max_u64(leader ? (uint64_t)arr : 0ull);
    hm = hl > hm ? hl : hm;
    S.log_event(leader, S.kc.make(fp, kAlloc, p), du);
    bool rel = false;
    int64_t tr = arr;
    if (leader) {
      rel = true;
      for (uint32_t u = 0; u < nl; ++u) {
        const uint32_t c = __ldg(lst + u);
        if (S.row[c] != du) continue;
        const int64_t fc = S.fin(c);
        if (fc <= 0) {  // not started yet
          rel = false;
          break;
        }
        tr = fc > tr ? fc : tr;
      }
    }
    S.log_event(rel, S.kc.make(tr, kFree, p), du);
  }
  // source copy
  bool pending = false;
  uint64_t mx = 0;
  for (uint32_t c0 = 0; c0 < nl; c0 += 32) {
    const uint32_t t = c0 + lane;
    if (t < nl) {
      const uint32_t c = __ldg(lst + t);
      if (S.row[c] == dp) {
        const int64_t fc = S.fin(c);
        if (fc <= 0) pending = true;
        else mx = (uint64_t)fc > mx ? (uint64_t)fc : mx;
      }
    }
  }
  if (__any_sync(kFullMask, pending)) return;
  const int64_t m = (int64_t)warp_max_u64(mx);
  S.log_event(lane == 0, S.kc.make(m > hm ? m : hm, kFree, p), dp);
}

template <bool kReg, bool kKey, bool kT32, bool kTypes, bool kBatch>
__global__ void __launch_bounds__(128, kBatch ? kBatchBlocksPerSM : 7) sim_inc_kernel(const __grid_constant__ SimParams P) {
  extern __shared__ __align__(16) uint8_t smem[];
  const unsigned wib = threadIdx.x >> 5;
  const int64_t slot = (int64_t)blockIdx.x * (blockDim.x >> 5) + wib;
  Sim<kReg, kInc, kKey, kT32, kTypes, kBatch> S(P);
  setup_slot(S, P, wib, slot, smem);
  S.rb = P.base.rb;
  S.fb = P.base.fb;
  uint8_t* crow = P.scratch + slot * P.slot_bytes + P.off_row;
  for (int64_t k = take_candidate(P.next_k); k < P.K; k = take_candidate(P.next_k)) inc_candidate(S, P, k, crow);
}

}  // namespace

// Instances by (accelerator state in registers, accelerator id in the event
// key, 32-bit times, accelerator types, batched sweep).  32-bit times are only
// chosen with the accelerator id in the key; the batched sweep only with
// accelerator state in shared memory and the id in the key.
template <bool R, bool K, bool T32, bool B>
const void* inc_ptr5(bool types) {
  return types ? (const void*)sim_inc_kernel<R, K, T32, true, B> : (const void*)sim_inc_kernel<R, K, T32, false, B>;
}
const void* inc_kernel_ptr(bool reg, bool key, bool t32, bool types, bool batch) {
  if (reg) {
    if (!key) return inc_ptr5<true, false, false, false>(types);
    return t32 ? inc_ptr5<true, true, true, false>(types) : inc_ptr5<true, true, false, false>(types);
  }
  if (!key) return inc_ptr5<false, false, false, false>(types);
  if (batch) return t32 ? inc_ptr5<false, true, true, true>(types) : inc_ptr5<false, true, false, true>(types);
  return t32 ? inc_ptr5<false, true, true, false>(types) : inc_ptr5<false, true, false, false>(types);
}

}  // namespace gsim
