// Host side of the C ABI (include/gmgsim.h): validation, the device layout
// of a GMG, scratch sizing and kernel launches.  No device memory is ever
// allocated here: every buffer is the caller's.

#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include "gmg_access.h"
#include "gmg_arb.h"
#include "gmg_arbw.h"

namespace gsim {
// launchers (gmgsim_kernels.cu)
size_t select_rank_bytes();
const void* full_kernel_ptr(bool reg, bool key, bool t32, bool types, bool batch);
const void* inc_kernel_ptr(bool reg, bool key, bool t32, bool types, bool batch);
const void* full_staged_kernel_ptr();
cudaError_t launch_full(bool reg, const SimParams& P, int grid, int block, size_t smem, cudaStream_t st);
cudaError_t launch_full_staged(const SimParams& P, int grid, int block, size_t smem, cudaStream_t st);
cudaError_t launch_inc(bool reg, const SimParams& P, int grid, int block, size_t smem, cudaStream_t st);
cudaError_t launch_base(bool reg, const SimParams& P, size_t smem, cudaStream_t st);
cudaError_t set_smem_limits(int smem);
cudaError_t launch_select(const int32_t* status, const int32_t* viol, const int64_t* score,
                          const int32_t* miss, int32_t K, int32_t mode, void* tmp, int nparts,
                          int64_t* best, cudaStream_t st);
}  // namespace gsim

using namespace gsim;

namespace {

constexpr int64_t kI64Max = 0x7fffffffffffffffll;
constexpr int kMaxOpsLog2 = 28;          // op ids must fit the packed key
constexpr int kDefaultWarpsPerBlock = 4;
constexpr int kSharedQueueEntries = 97;  // 1 + 32 * 3: root, its children, two more groups
// The batched sweep's sizes (compile-time overridable for tuning sweeps).
#ifndef GMG_BATCH_QUEUE_SHARED
#define GMG_BATCH_QUEUE_SHARED 161  // 1 + 32 * 5 (with the log below: 28 warps per SM at 256 accelerators)
#endif
#ifndef GMG_BATCH_OPS_PER_GENERATION
#define GMG_BATCH_OPS_PER_GENERATION 24
#endif
#ifndef GMG_BATCH_LOG_SHARED
#define GMG_BATCH_LOG_SHARED 128
#endif
constexpr int kSharedQueueEntriesBatch = GMG_BATCH_QUEUE_SHARED;
constexpr int kBatchOpsPerGeneration = GMG_BATCH_OPS_PER_GENERATION;
constexpr int kSharedLogEntriesBatch = GMG_BATCH_LOG_SHARED;
constexpr int64_t kDefaultQueueCap = 1 << 16;
constexpr int kSharedLogEntries = 192;
constexpr int64_t kDefaultLogCap = 1 << 17;
constexpr int kSortCap = 128;             // power of two; raised to n_dev's power of two
constexpr int kOpsPerGeneration = 24;     // ~85 HBM events per generation (prefill graphs)
constexpr int kBatchMinDevices = 33;      // the batched sweep serves graphs on more accelerators
constexpr int kCheckpoints = 256;
constexpr int kArbCheckpoints = 64;       // arbitrated bases also keep ~32 bytes per op per checkpoint
constexpr int kCheckpointQueue = 4096;
constexpr int kCheckpointLog = 8192;

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct Layout {
  size_t off_ops, off_succ, off_pred, off_sib, off_cons, off_roots, off_roots_q, off_cap, off_base, off_avail,
      off_dl, off_links, off_durt, off_dtype, off_linkid, off_st_hot, off_st_rel, total;
};

// Everything gmg_create derives from a description.
struct Built {
  int n = 0, E = 0, D = 0, R = 0, Ec = 0, nroots = 0, ib = 1, T = 0;
  bool uniform = true;
  int64_t bw0 = 1, lat0 = 0, time_bound = 0, max_iter = 0, queue_bound = 0, log_bound = 0;
  std::vector<OpRec> ops;
  std::vector<uint32_t> succ, pred, sib, cons;
  std::vector<uint64_t> roots;
  std::vector<int64_t> cap, base, avail0, deadline;
  std::vector<LinkRec> links;
  std::vector<int64_t> durt;  // [n*T] when T >= 2
  std::vector<uint8_t> dtype; // [D] when T >= 2
  std::vector<uint16_t> linkid;  // [D*D] communication link of each ordered pair
  int64_t xfer_bound = 0;     // transfers of one placement at most: sum of min(successors, D-1)
  bool shared_links = false;  // two distinct ordered pairs share a link id
  // compact hot records for a CTA's staged copy (sim_opts_t.gmg_staging = 1)
  bool stage_ready = false;
  std::vector<uint32_t> st_hot;  // [4n]
  std::vector<int32_t> st_rel;   // [n]
  Layout L{};
};

LinkRec make_link(int64_t bw, int64_t lat) {
  LinkRec r{};
  int l = 0;
  while ((int64_t(1) << l) < bw) ++l;  // l = ceil(log2 bw)
  const int s = 53 + l;
  const unsigned __int128 one = 1;
  const unsigned __int128 m = ((one << s) + (unsigned __int128)(bw - 1)) / (unsigned __int128)bw;
  r.magic = (uint64_t)m;
  r.bw = bw;
  r.lat = lat;
  r.shift = s;
  return r;
}

int64_t host_ceil(int64_t n, int64_t d) {
  const int64_t q = n / d;
  return q * d == n ? q : q + 1;
}

void plan(Built& b) {
  Layout& L = b.L;
  size_t o = 0;
  auto take = [&](size_t bytes) {
    const size_t at = o;
    o = align_up(o + std::max<size_t>(bytes, 1), 256);
    return at;
  };
  L.off_ops = take(sizeof(OpRec) * (size_t)b.n);
  L.off_succ = take(4 * (size_t)b.E);
  L.off_pred = take(4 * (size_t)b.E);
  L.off_sib = take(8 * (size_t)b.E);
  L.off_cons = take(4 * (size_t)b.Ec);
  L.off_roots = take(8 * (size_t)b.nroots);
  L.off_roots_q = take(8 * (size_t)b.nroots);
  L.off_cap = take(8 * (size_t)b.D);
  L.off_base = take(8 * (size_t)b.D);
  L.off_avail = take(8 * (size_t)b.D);
  L.off_dl = take(8 * (size_t)b.R);
  L.off_links = take(b.uniform ? 0 : sizeof(LinkRec) * (size_t)b.D * b.D);
  L.off_durt = take(8 * b.durt.size());
  L.off_dtype = take(b.dtype.size());
  L.off_linkid = take(2 * b.linkid.size());
  L.off_st_hot = take(b.stage_ready ? 16 * (size_t)b.n : 0);
  L.off_st_rel = take(b.stage_ready ? align_up(4 * (size_t)b.n, 16) : 0);
  L.total = o;
}

// Validate and derive.  Returns GMG_OK or an error code.
int build(const gmg_desc_t* d, Built& b) {
  if (!d) return GMG_EINVAL;
  const int n = d->n_ops, D = d->n_dev, R = d->n_req;
  if (n < 0 || d->n_edges < 0 || D < 1 || D > 256 || R < 0) return GMG_EINVAL;
  if (n > (1 << kMaxOpsLog2)) return GMG_ERANGE;
  if (!d->pred_off || (d->n_edges > 0 && !d->pred_idx)) return GMG_EINVAL;
  const int T = d->n_types >= 2 ? d->n_types : 0;
  if (d->n_types < 0 || d->n_types > 256) return GMG_EINVAL;
  if (T && (!d->dev_type || (n > 0 && !d->dur_by_type))) return GMG_EINVAL;
  if (n > 0 && ((!T && !d->dur_us) || !d->out_bytes)) return GMG_EINVAL;
  if (D > 1 && (!d->bw_B_per_us || !d->lat_us)) return GMG_EINVAL;
  if (d->pred_off[0] != 0 || d->pred_off[n] != d->n_edges) return GMG_EINVAL;
  for (int i = 0; i < n; ++i)
    if (d->pred_off[i + 1] < d->pred_off[i]) return GMG_EINVAL;
  b.n = n;
  b.E = d->n_edges;
  b.D = D;
  b.R = R;
  b.T = T;
  if (T) {
    b.dtype.assign(d->dev_type, d->dev_type + D);
    for (int e = 0; e < D; ++e)
      if (b.dtype[e] >= T) return GMG_EINVAL;
    b.durt.assign(d->dur_by_type, d->dur_by_type + (size_t)n * T);
  }
  b.ib = 1;
  while ((int64_t(1) << b.ib) < n) ++b.ib;
  // predecessors (topological, no duplicates) and successor counts
  std::vector<uint32_t> nsucc(n, 0);
  b.pred.resize(b.E);
  std::vector<int32_t> seen(n, -1);
  for (int i = 0; i < n; ++i) {
    for (int k = d->pred_off[i]; k < d->pred_off[i + 1]; ++k) {
      const int p = d->pred_idx[k];
      if (p < 0 || p >= n) return GMG_EINVAL;
      if (p >= i) return GMG_ENOTTOPO;
      if (seen[p] == i) return GMG_EINVAL;
      seen[p] = i;
      b.pred[k] = (uint32_t)p;
      ++nsucc[p];
    }
  }
  b.ops.assign(n, OpRec{});
  uint32_t acc = 0;
  for (int i = 0; i < n; ++i) {
    b.ops[i].succ_off = acc;
    acc += nsucc[i];
  }
  b.succ.resize(b.E);
  std::vector<uint32_t> fill(n, 0);
  for (int i = 0; i < n; ++i)
    for (int k = d->pred_off[i]; k < d->pred_off[i + 1]; ++k) {
      const int p = d->pred_idx[k];
      b.succ[b.ops[p].succ_off + fill[p]++] = (uint32_t)i;  // ascending: i increases
    }
  // per-op scalars
  for (int i = 0; i < n; ++i) {
    OpRec& r = b.ops[i];
    if (T) {
      // the bounds below take an op's longest duration over the types
      r.dur = 0;
      for (int t = 0; t < T; ++t) {
        const int64_t v = b.durt[(size_t)i * T + t];
        if (v < 1) return GMG_EINVAL;
        r.dur = std::max(r.dur, v);
      }
    } else {
      r.dur = d->dur_us[i];
    }
    r.bytes = d->out_bytes[i];
    r.release = d->release_us ? d->release_us[i] : 0;
    r.req = d->req_id ? d->req_id[i] : -1;
    const uint8_t sc = d->scored ? d->scored[i] : 1;
    if (r.dur < 1 || r.bytes < 0 || r.release < 0) return GMG_EINVAL;
    if (r.req < -1 || r.req >= R) return GMG_EINVAL;
    if (sc > 1) return GMG_EINVAL;
    if (r.bytes >= (int64_t(1) << 53)) return GMG_ERANGE;
    r.nsucc = nsucc[i];
    r.pred_off = (uint32_t)d->pred_off[i];
    r.npred = (uint32_t)(d->pred_off[i + 1] - d->pred_off[i]);
    r.flags = sc ? kScored : 0u;
  }
  // consumer lists (subsets of the successors) and the hold bits on the
  // consumers' predecessor entries
  auto set_hold = [&](uint32_t c, uint32_t p) {
    for (uint32_t k = b.ops[c].pred_off; k < b.ops[c].pred_off + b.ops[c].npred; ++k)
      if ((b.pred[k] & kIdMask) == p) {
        b.pred[k] |= kHoldBit;
        return;
      }
  };
  if (!d->cons_off) {
    for (int i = 0; i < n; ++i) {
      b.ops[i].flags |= kAllCons;
      b.ops[i].cons_off = b.ops[i].succ_off;
      b.ops[i].ncons = b.ops[i].nsucc;
      for (uint32_t k = 0; k < b.ops[i].nsucc; ++k) set_hold(b.succ[b.ops[i].succ_off + k], i);
    }
  } else {
    if (d->cons_off[0] != 0) return GMG_EINVAL;
    for (int i = 0; i < n; ++i)
      if (d->cons_off[i + 1] < d->cons_off[i]) return GMG_EINVAL;
    if (d->cons_off[n] > 0 && !d->cons_idx) return GMG_EINVAL;
    std::vector<int32_t> mark(n, -1);
    for (int i = 0; i < n; ++i) {
      OpRec& r = b.ops[i];
      for (uint32_t k = 0; k < r.nsucc; ++k) mark[b.succ[r.succ_off + k]] = i;
      const int a = d->cons_off[i], e = d->cons_off[i + 1];
      for (int k = a; k < e; ++k) {
        const int c = d->cons_idx[k];
        if (c < 0 || c >= n || mark[c] != i) return GMG_EINVAL;  // not a successor, or repeated
        mark[c] = -2 - i;
      }
      if ((uint32_t)(e - a) == r.nsucc) {
        r.flags |= kAllCons;
        r.cons_off = r.succ_off;
        r.ncons = r.nsucc;
        for (uint32_t k = 0; k < r.nsucc; ++k) set_hold(b.succ[r.succ_off + k], i);
      } else {
        r.cons_off = (uint32_t)b.cons.size();
        r.ncons = (uint32_t)(e - a);
        for (int k = a; k < e; ++k) {
          b.cons.push_back((uint32_t)d->cons_idx[k]);
          set_hold((uint32_t)d->cons_idx[k], i);
        }
      }
    }
  }
  b.Ec = (int)b.cons.size();
  // For every (predecessor p -> holding consumer c) entry: the other listed
  // consumer of p, so that c can tell whether it is p's last one there.
  b.sib.assign(b.E, kSibNone);
  // Bounded reachability along successors (ids are topological, so a search
  // never needs to pass the target id); "unknown" simply keeps the run-time
  // check.
  std::vector<uint32_t> stack;
  std::vector<int32_t> seen_at(n, -1);
  int stamp = 0;
  auto reaches = [&](uint32_t from, uint32_t to) {
    ++stamp;
    stack.assign(1, from);
    int visited = 0;
    while (!stack.empty() && visited < 256) {
      const uint32_t x = stack.back();
      stack.pop_back();
      ++visited;
      const OpRec& rx = b.ops[x];
      for (uint32_t k = 0; k < rx.nsucc; ++k) {
        const uint32_t y = b.succ[rx.succ_off + k];
        if (y == to) return true;
        if (y < to && seen_at[y] != stamp) {
          seen_at[y] = stamp;
          stack.push_back(y);
        }
      }
    }
    return false;
  };
  for (int p = 0; p < n; ++p) {
    const OpRec& r = b.ops[p];
    const uint32_t* lst = (r.flags & kAllCons) ? b.succ.data() + r.succ_off : b.cons.data() + r.cons_off;
    for (uint32_t u = 0; u < r.ncons; ++u) {
      const uint32_t c = lst[u];
      uint32_t v = kSibNone;
      if (r.ncons == 2) {
        const uint32_t o = lst[1 - u];
        // A fixed finishing order between the two consumers (one depends on
        // the other) settles the release without a run-time check.
        if (o < c && reaches(o, c)) v = kSibNone;           // c always finishes last
        else if (o > c && reaches(c, o)) v = o | kSibLater;  // o always finishes later
        else v = o;
      } else if (r.ncons > 2) {
        v = kSibMany;
      }
      for (uint32_t k = b.ops[c].pred_off; k < b.ops[c].pred_off + b.ops[c].npred; ++k)
        if ((b.pred[k] & kIdMask) == (uint32_t)p) b.sib[k] = v;
    }
  }
  // request sinks: no successor in the same request
  for (int i = 0; i < n; ++i) {
    OpRec& r = b.ops[i];
    if (r.req < 0) continue;
    bool sink = true;
    for (uint32_t k = 0; k < r.nsucc && sink; ++k)
      if (b.ops[b.succ[r.succ_off + k]].req == r.req) sink = false;
    if (sink) r.flags |= kReqSink;
  }
  // accelerators
  b.cap.resize(D);
  b.base.resize(D);
  b.avail0.resize(D);
  for (int e = 0; e < D; ++e) {
    b.cap[e] = d->cap_bytes ? d->cap_bytes[e] : kI64Max;
    b.base[e] = d->base_bytes ? d->base_bytes[e] : 0;
    b.avail0[e] = d->avail0_us ? d->avail0_us[e] : 0;
    if (b.cap[e] < 0 || b.base[e] < 0 || b.base[e] > b.cap[e] || b.avail0[e] < 0) return GMG_EINVAL;
  }
  b.deadline.resize(R);
  for (int r = 0; r < R; ++r) b.deadline[r] = d->deadline_us ? d->deadline_us[r] : kI64Max;
  // links
  int64_t min_bw = kI64Max, max_lat = 0;
  b.uniform = true;
  bool first = true;
  for (int s = 0; s < D; ++s)
    for (int e = 0; e < D; ++e) {
      if (s == e) continue;
      const int64_t bw = d->bw_B_per_us[(size_t)s * D + e], lat = d->lat_us[(size_t)s * D + e];
      if (bw < 1 || lat < 0) return GMG_EINVAL;
      if (bw >= (int64_t(1) << 62)) return GMG_ERANGE;
      if (first) {
        b.bw0 = bw;
        b.lat0 = lat;
        first = false;
      } else if (bw != b.bw0 || lat != b.lat0) {
        b.uniform = false;
      }
      min_bw = std::min(min_bw, bw);
      max_lat = std::max(max_lat, lat);
    }
  if (D == 1) {
    min_bw = 1;
    b.bw0 = 1;
    b.lat0 = 0;
  }
  if (!b.uniform) {
    b.links.resize((size_t)D * D);
    for (int s = 0; s < D; ++s)
      for (int e = 0; e < D; ++e)
        b.links[(size_t)s * D + e] =
            s == e ? make_link(1, 0)
                   : make_link(d->bw_B_per_us[(size_t)s * D + e], d->lat_us[(size_t)s * D + e]);
  }
  for (int i = 0; i < n; ++i) b.ops[i].xq = host_ceil(b.ops[i].bytes, b.bw0);
  // communication links of the arbitrated transfers
  for (int s = 0; s < D; ++s)
    for (int e = 0; e < D; ++e) {
      const size_t k = (size_t)s * D + e;
      const int64_t id = d->link_id ? d->link_id[k] : (int64_t)k;
      if (s != e && (id < 0 || id >= (int64_t)D * D)) return GMG_EINVAL;
    }
  {
    b.linkid.resize((size_t)D * D);
    std::vector<int> uses((size_t)D * D, 0);
    for (size_t k = 0; k < b.linkid.size(); ++k) {
      const bool diag = k / D == k % D;
      b.linkid[k] = (uint16_t)(d->link_id && !diag ? d->link_id[k] : (int32_t)k);
      if (!diag && ++uses[b.linkid[k]] > 1) b.shared_links = true;
    }
  }
  // Bounds: every time <= start + all durations + one transfer per edge and
  // per op; it must fit the packed key (61 - ib bits); scores and byte totals
  // must fit int64.
  typedef __int128 i128;
  i128 t = 0, mem = 0, iters = 16, qb = 16, lb = 16;
  for (int e = 0; e < D; ++e) {
    t = std::max<i128>(t, b.avail0[e]);
    mem += b.base[e];
  }
  for (int i = 0; i < n; ++i) t = std::max<i128>(t, b.ops[i].release);
  const i128 tlim = i128(1) << (61 - b.ib);
  for (int i = 0; i < n; ++i) {
    const OpRec& r = b.ops[i];
    const i128 mx = i128(r.bytes / min_bw + 1) + max_lat;
    const uint32_t copies = std::min<uint32_t>(r.nsucc, (uint32_t)(D - 1));
    t += r.dur + mx * i128(r.nsucc + 1);
    mem += i128(r.bytes) * i128(copies + 1);
    iters += 1;
    qb += r.npred ? 1 : 0;
    lb += 2 + 2 * i128(copies);
    b.xfer_bound += copies;
    if (t >= tlim || mem >= (i128(1) << 62)) return GMG_ERANGE;
  }
  if (t * i128(std::max(n, 1)) >= (i128(1) << 62)) return GMG_ERANGE;
  b.time_bound = (int64_t)t;
  b.max_iter = (int64_t)iters;
  b.queue_bound = (int64_t)qb;
  b.log_bound = (int64_t)lb;
  // roots, by (release, id)
  for (int i = 0; i < n; ++i)
    if (b.ops[i].npred == 0)
      b.roots.push_back(((uint64_t)b.ops[i].release << (b.ib + 2)) | (uint64_t)i);
  std::sort(b.roots.begin(), b.roots.end());
  b.nroots = (int)b.roots.size();
  // compact records for the staged copy: one accelerator type, uniform links,
  // every time below 2^31, lists addressable in 24 bits with fewer than 256
  // entries per op, transfer sizes (xq) below 2^29
  b.stage_ready = !b.T && b.uniform && b.time_bound < (int64_t(1) << 31) && b.E < (1 << 24);
  for (int i = 0; i < n && b.stage_ready; ++i) {
    const OpRec& r = b.ops[i];
    b.stage_ready = r.nsucc < 256 && r.npred < 256 && r.xq < (int64_t(1) << 29);
  }
  if (b.stage_ready) {
    b.st_hot.resize(4 * (size_t)n);
    b.st_rel.resize(n);
    for (int i = 0; i < n; ++i) {
      const OpRec& r = b.ops[i];
      b.st_hot[4 * (size_t)i] = (uint32_t)r.dur;
      b.st_hot[4 * (size_t)i + 1] = (uint32_t)r.xq | ((r.flags & 7u) << 29);
      b.st_hot[4 * (size_t)i + 2] = r.succ_off | (r.nsucc << 24);
      b.st_hot[4 * (size_t)i + 3] = r.pred_off | (r.npred << 24);
      b.st_rel[i] = (int32_t)r.release;
    }
  }
  plan(b);
  return GMG_OK;
}

int device_sms() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return -1;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return -1;
  return sms;
}

}  // namespace

struct gmg {
  DevGmg dg;
  gmg_info_t info;
  int64_t queue_bound;
  int64_t log_bound;
  const uint16_t* linkid;  // device [D*D]
  int32_t shared_links;    // 1 if two distinct ordered pairs share a link id
  int64_t xfer_bound;
};

const DevGmg* gsim::gmg_device_graph(const gmg_t* g) { return g ? &g->dg : nullptr; }

struct gmg_base {
  DevBase db;
  const gmg* g;
  uint8_t* slot;
  int qs, qcap;
  int arb;     // 1: an arbitrated snapshot, which serves arbitrated candidates only
  ArbCk ck;    // its arbiter arenas
};

namespace {

struct Launch {
  bool reg;
  int wpb, grid;
  size_t smem;
  int64_t slots;
  SimParams P;  // sizes and slot offsets filled
};

int queue_cap(const gmg* g, const sim_opts_t* o) {
  const int64_t c = (o && o->queue_cap > 0) ? o->queue_cap : std::min<int64_t>(g->queue_bound, kDefaultQueueCap);
  return (int)std::max<int64_t>(c, 1);
}

int log_cap(const gmg* g, const sim_opts_t* o) {
  const int64_t c = (o && o->queue_cap > 0) ? 2 * (int64_t)o->queue_cap
                                           : std::min<int64_t>(g->log_bound, kDefaultLogCap);
  return (int)std::max<int64_t>(c, 1);
}

size_t smem_per_warp(const SimParams& P) {
  const size_t side = P.no_side ? 0 : 1;
  return align_up((size_t)P.qs * 8 + (size_t)P.ms * (8 + side) + (size_t)P.sortcap * (8 + side) + (size_t)P.opcap * 4,
                  16) +
         (size_t)P.dev_bytes;
}

// Shared bytes of accelerator state per warp: live bytes; peaks unless they
// are kept in global scratch (more than 32 accelerators); free times (of
// tbytes each) unless lanes hold them in registers (at most 32).
int dev_smem_bytes(int D, size_t tbytes) {
  const bool reg = D <= 32;
  return (int)align_up((size_t)D * 8 + (reg ? (size_t)D * 8 : 0) + (reg ? 0 : (size_t)D * tbytes), 16);
}

bool g_smem_set = false;

// Slot layout and grid for K candidates of kind `inc` (sweep: the graph's
// batched sweep if it has one; the arbitrated kernels take keys one at a time).
int plan_launch(const gmg* g, int32_t K, const sim_opts_t* o, bool inc, Launch& L, bool sweep_batch = true) {
  const DevGmg& G = g->dg;
  const bool batch = G.batch && sweep_batch;
  L.reg = G.D <= 32;
  L.wpb = (o && o->warps_per_block > 0) ? o->warps_per_block : kDefaultWarpsPerBlock;
  if (L.wpb > 4) return GMG_EINVAL;
  SimParams& P = L.P;
  std::memset(&P, 0, sizeof(P));
  P.g = G;
  P.qcap = queue_cap(g, o);
  P.qs = batch ? kSharedQueueEntriesBatch : kSharedQueueEntries;  // >= 33 (the root's children are
                                                                     // always in shared memory)
  P.mcap = log_cap(g, o);
  P.ms = batch ? kSharedLogEntriesBatch : kSharedLogEntries;
  P.sortcap = kSortCap;
  while (P.sortcap < G.D) P.sortcap <<= 1;
  P.drain_trigger = batch ? kBatchOpsPerGeneration : kOpsPerGeneration;
  P.opcap = batch ? kBatchOpsPerGeneration + 32 : kOpsPerGeneration;
  P.dev_bytes = dev_smem_bytes(G.D, G.t32 ? 4 : 8);
  P.no_side = batch ? 1 : 0;  // the batched sweep keeps the accelerator inside the entry
  L.smem = (size_t)L.wpb * smem_per_warp(P);
  size_t o2 = 0;
  auto take = [&](size_t bytes) {
    const size_t at = o2;
    o2 = align_up(o2 + std::max<size_t>(bytes, 1), 256);
    return (int64_t)at;
  };
  const int64_t qspill = std::max<int64_t>(P.qcap - P.qs, 0);
  const int64_t mspill = std::max<int64_t>(P.mcap - P.ms, 0);
  P.off_f = take(8 * (size_t)G.n);
  P.off_hold = take(8 * (size_t)G.n);
  P.off_bits = take(4 * (size_t)((G.n + 31) / 32) + 16);
  P.off_creq = take(8 * (size_t)G.R);
  P.off_qk = take(8 * (size_t)qspill);
  P.off_mk = take(8 * (size_t)mspill);
  P.off_md = take((size_t)mspill);
  P.off_row = take(inc ? (size_t)align_up(std::max(G.n, 1), 16) : 0);
  P.off_pk = L.reg ? -1 : take(8 * (size_t)G.D);
  P.slot_bytes = (int64_t)o2;
  const int sms = device_sms();
  if (sms <= 0) return GMG_ECUDA;
  if (!g_smem_set) {
    // the largest per-block request: 4 warps with 256 accelerators
    SimParams big = P;
    big.g.D = 256;
    big.sortcap = 256;
    big.opcap = std::max(kOpsPerGeneration, kBatchOpsPerGeneration + 32);
    big.qs = std::max(kSharedQueueEntries, kSharedQueueEntriesBatch);
    big.ms = std::max(kSharedLogEntries, kSharedLogEntriesBatch);
    big.dev_bytes = 24 * 256;
    big.no_side = 0;
    if (set_smem_limits(4 * (int)smem_per_warp(big)) != cudaSuccess) return GMG_ECUDA;
    g_smem_set = true;
  }
  int bps = 0;
  const bool types = G.ntypes >= 2;
  const void* fn = inc ? inc_kernel_ptr(L.reg, G.dev_key != 0, G.t32 != 0, types, batch)
                       : full_kernel_ptr(L.reg, G.dev_key != 0, G.t32 != 0, types, batch);
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&bps, fn, 32 * L.wpb, L.smem) != cudaSuccess)
    return GMG_ECUDA;
  bps = std::max(bps, 1);
  const int64_t need = (std::max<int64_t>(K, 1) + L.wpb - 1) / L.wpb;
  L.grid = (int)std::min<int64_t>(need, (int64_t)sms * bps);
  L.slots = (int64_t)L.grid * L.wpb;
  P.g = G;
  return GMG_OK;
}

bool aligned(const void* p, size_t a) { return ((uintptr_t)p % a) == 0; }

int check_out(const sim_out_t* o, const sim_opts_t* opts) {
  if (!o || !o->makespan || !o->score || !o->status || !o->viol_flag || !o->viol_op ||
      !o->viol_dev || !o->viol_time || !o->peak || !o->sla_miss || !o->events)
    return GMG_EINVAL;
  if (opts && opts->n_trace < 0) return GMG_EINVAL;
  if (opts && opts->n_trace > 0 && (!opts->d_trace_k || !o->trace_start || !o->trace_finish))
    return GMG_EINVAL;
  if (opts) {
    for (int r : opts->reserved)
      if (r != 0) return GMG_EINVAL;
    if (opts->transfer_mode != GMG_TRANSFER_LATENCY && opts->transfer_mode != GMG_TRANSFER_ARBITRATED)
      return GMG_EINVAL;
    if (opts->gmg_staging < GMG_STAGING_DEFAULT || opts->gmg_staging > GMG_STAGING_L1) return GMG_EINVAL;
  }
  return GMG_OK;
}

bool staged(const sim_opts_t* o) { return o && o->gmg_staging == GMG_STAGING_SHARED; }
bool l1_path(const sim_opts_t* o) { return o && o->gmg_staging == GMG_STAGING_L1; }

bool g_stage_smem_set = false;

// sim_batch with the GMG staged in shared memory: one CTA per SM with as many
// warps (up to kStageMaxWarps) as fit beside the staged copy.
int plan_staged(const gmg* g, int32_t K, const sim_opts_t* o, Launch& L) {
  const DevGmg& G = g->dg;
  if (!G.stage_ok || (o && o->transfer_mode != GMG_TRANSFER_LATENCY)) return GMG_EINVAL;
  int rc = plan_launch(g, K, o, false, L);
  if (rc) return rc;
  int dev = 0, optin = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
    return GMG_ECUDA;
  SimParams& P = L.P;
  P.stage_bytes = (int32_t)stage_smem_bytes(G.n, G.n_edges);
  const size_t spw = smem_per_warp(P);
  const int64_t room = (int64_t)optin - P.stage_bytes;
  const int64_t fit = std::min<int64_t>(kStageMaxWarps, room > 0 ? room / (int64_t)spw : 0);
  if (fit < 1) return GMG_EINVAL;
  // as many warps per CTA as spread the candidates over every SM (few
  // candidates: small CTAs on many SMs; many: up to what fits beside the copy)
  const int sms = device_sms();
  if (sms <= 0) return GMG_ECUDA;
  const int w = (int)std::min<int64_t>(fit, std::max<int64_t>(1, ((int64_t)std::max(K, 1) + sms - 1) / sms));
  if (!g_stage_smem_set) {
    if (cudaFuncSetAttribute(full_staged_kernel_ptr(), cudaFuncAttributeMaxDynamicSharedMemorySize, optin) !=
        cudaSuccess)
      return GMG_ECUDA;
    g_stage_smem_set = true;
  }
  L.wpb = w;
  L.smem = (size_t)P.stage_bytes + (size_t)w * spw;
  L.grid = (int)std::min<int64_t>(sms, ((int64_t)std::max(K, 1) + w - 1) / w);
  L.slots = (int64_t)L.grid * w;
  return GMG_OK;
}

// Full placements with pure-latency transfers: the staged-GMG kernel when the
// caller asks for it (an error if it cannot serve the graph) or by default
// when it can, else the L1 path.  *stg tells which.
int plan_full(const gmg* g, int32_t K, const sim_opts_t* o, Launch& L, bool* stg) {
  *stg = false;
  if (l1_path(o)) return plan_launch(g, K, o, false, L);
  const int rc = plan_staged(g, K, o, L);
  if (rc == GMG_OK) {
    *stg = true;
    return GMG_OK;
  }
  if (staged(o) || rc != GMG_EINVAL) return rc;
  return plan_launch(g, K, o, false, L);
}

bool arbitrated(const sim_opts_t* o) { return o && o->transfer_mode == GMG_TRANSFER_ARBITRATED; }

void fill_out(SimParams& P, const sim_out_t* o, const sim_opts_t* opts) {
  P.out.makespan = o->makespan;
  P.out.score = o->score;
  P.out.status = o->status;
  P.out.viol_flag = o->viol_flag;
  P.out.viol_op = o->viol_op;
  P.out.viol_dev = o->viol_dev;
  P.out.viol_time = o->viol_time;
  P.out.peak = o->peak;
  P.out.sla_miss = o->sla_miss;
  P.out.events = o->events;
  P.out.req_done = o->req_done;
  P.out.trace_start = o->trace_start;
  P.out.trace_finish = o->trace_finish;
  P.n_trace = opts ? opts->n_trace : 0;
  P.trace_k = opts ? opts->d_trace_k : nullptr;
}

// Arbitrated transfers: the full simulation's slot plus the transfer state.
// At most 32 accelerators (endpoint sets are bit masks, link ids < 1024),
// op ids below 2^27 (an intent packs op << 5 | destination) and accelerator
// ids that fit beside the packed key.
// mode: kFull (sim_batch), kBase (the arbitrated base snapshot, 64-bit
// times) or kInc (candidates resumed from it; the slot also holds the
// candidate's row).
int plan_arb(const gmg* g, int32_t K, const sim_opts_t* o, Launch& L, ArbParams& A, int mode = kFull) {
  const DevGmg& G = g->dg;
  if (G.D > 32 || !g->linkid) return GMG_EINVAL;
  if (!G.dev_key || G.n >= (1 << 27)) return GMG_ERANGE;
  const int64_t xcap = std::max<int64_t>(g->xfer_bound, 1);
  if (xcap > (int64_t(1) << 29)) return GMG_ERANGE;
  int rc = plan_launch(g, K, o, mode == kInc, L, false);
  if (rc) return rc;
  std::memset(&A, 0, sizeof(A));
  SimParams& P = L.P;
  size_t o2 = (size_t)P.slot_bytes;
  auto take = [&](size_t bytes) {
    const size_t at = o2;
    o2 = align_up(o2 + std::max<size_t>(bytes, 1), 256);
    return (int64_t)at;
  };
  A.xcap = (int32_t)xcap;
  A.shared_links = g->shared_links;
  A.heads_shared = G.D <= 16 ? 1 : 0;
  const size_t n = (size_t)G.n, DD = (size_t)G.D * G.D;
  A.off_cnt = take(4 * n);
  A.off_rmax = take((G.t32 && mode != kBase ? 4 : 8) * n);
  A.off_refs = take(4 * n);
  A.off_rmask = take(4 * n);
  A.off_nextop = take(4 * n);
  A.off_xent = take(4 * (size_t)xcap);
  A.off_xnext = take(4 * (size_t)xcap);
  A.off_qhead = take(A.heads_shared ? 0 : 4 * DD);
  A.off_qtail = take(4 * DD);
  P.slot_bytes = (int64_t)o2;
  A.smem_arb = (int32_t)align_up(128 + (A.heads_shared ? 4 * DD : 0), 16);
  A.smem_std = (int64_t)L.smem;
  L.smem += (size_t)L.wpb * (size_t)A.smem_arb;
  const int sms = device_sms();
  if (sms <= 0) return GMG_ECUDA;
  int bps = 0;
  const void* fn = mode == kInc ? arb_inc_kernel_ptr(G.t32 != 0, G.ntypes >= 2)
                                : arb_kernel_ptr(G.t32 != 0, G.ntypes >= 2);
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&bps, fn, 32 * L.wpb, L.smem) != cudaSuccess)
    return GMG_ECUDA;
  bps = std::max(bps, 1);
  const int64_t need = (std::max<int64_t>(K, 1) + L.wpb - 1) / L.wpb;
  L.grid = (int)std::min<int64_t>(need, (int64_t)sms * bps);
  L.slots = (int64_t)L.grid * L.wpb;
  A.link = g->linkid;
  return GMG_OK;
}

// Arbitrated transfers on 33..256 accelerators: per-accelerator transfer
// state in tables.  Op ids below 2^24 (an intent packs op << 8 | destination).
int plan_arbw(const gmg* g, int32_t K, const sim_opts_t* o, Launch& L, ArbWParams& A) {
  const DevGmg& G = g->dg;
  if (G.D <= 32 || G.D > 256 || !g->linkid) return GMG_EINVAL;
  if (!G.dev_key || G.n >= (1 << 24)) return GMG_ERANGE;
  const int64_t xcap = std::max<int64_t>(g->xfer_bound, 1);
  if (xcap > (int64_t(1) << 29)) return GMG_ERANGE;
  int rc = plan_launch(g, K, o, false, L, false);
  if (rc) return rc;
  std::memset(&A, 0, sizeof(A));
  SimParams& P = L.P;
  size_t o2 = (size_t)P.slot_bytes;
  auto take = [&](size_t bytes) {
    const size_t at = o2;
    o2 = align_up(o2 + std::max<size_t>(bytes, 1), 256);
    return (int64_t)at;
  };
  const size_t n = (size_t)G.n, D = (size_t)G.D, DD = D * D, tsz = G.t32 ? 4 : 8;
  A.xcap = (int32_t)xcap;
  A.shared_links = g->shared_links;
  A.words = (int32_t)((D + 31) / 32);
  A.off_cnt = take(4 * n);
  A.off_rmax = take(tsz * n);
  A.off_refs = take(4 * n);
  A.off_nextop = take(4 * n);
  A.off_xent = take(4 * (size_t)xcap);
  A.off_xnext = take(4 * (size_t)xcap);
  A.off_qhead = take(4 * DD);
  A.off_qtail = take(4 * DD);
  A.off_xd = take(tsz * D);
  A.off_xp = take(4 * D);
  A.off_xe = take(4 * D);
  A.off_fh = take(4 * D);
  A.off_ft = take(4 * D);
  A.off_fa = take(tsz * D);
  A.off_pm = take(4 * D * (size_t)A.words);
  A.off_lb = take(4 * ((DD + 31) / 32));
  P.slot_bytes = (int64_t)o2;
  A.smem_arb = 128;  // four 8-word bit sets
  A.smem_std = (int64_t)L.smem;
  L.smem += (size_t)L.wpb * (size_t)A.smem_arb;
  const int sms = device_sms();
  if (sms <= 0) return GMG_ECUDA;
  int bps = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&bps, arbw_kernel_ptr(G.t32 != 0, G.ntypes >= 2), 32 * L.wpb,
                                                    L.smem) != cudaSuccess)
    return GMG_ECUDA;
  bps = std::max(bps, 1);
  const int64_t need = (std::max<int64_t>(K, 1) + L.wpb - 1) / L.wpb;
  L.grid = (int)std::min<int64_t>(need, (int64_t)sms * bps);
  L.slots = (int64_t)L.grid * L.wpb;
  A.link = g->linkid;
  return GMG_OK;
}

// Either arbitrated kernel, by accelerator count.
struct ArbPlan {
  bool wide = false;
  ArbParams A;
  ArbWParams AW;
};

int plan_arb_any(const gmg* g, int32_t K, const sim_opts_t* o, Launch& L, ArbPlan& Q) {
  Q.wide = g->dg.D > 32;
  return Q.wide ? plan_arbw(g, K, o, L, Q.AW) : plan_arb(g, K, o, L, Q.A);
}

cudaError_t launch_arb_any(const gmg* g, Launch& L, ArbPlan& Q, const int32_t* pre_status, cudaStream_t st) {
  if (Q.wide) {
    Q.AW.P = L.P;
    Q.AW.pre_status = pre_status;
    return launch_arbw(g->dg.t32 != 0, g->dg.ntypes >= 2, Q.AW, L.grid, 32 * L.wpb, L.smem, st);
  }
  Q.A.P = L.P;
  Q.A.pre_status = pre_status;
  return launch_arb(g->dg.t32 != 0, g->dg.ntypes >= 2, Q.A, L.grid, 32 * L.wpb, L.smem, st);
}


struct BasePlan {
  size_t off_row, off_rb, off_fb, off_status, off_res, off_peak, off_creq, off_cktime,
      off_cksc, off_ckdev, off_ckcreq, off_ckqk, off_ckmk, off_ckmd, off_arena, off_slot, total;
  int nck, ckq, ckm, ld, stride;
  bool arb;     // an arbitrated base snapshot (also keeps the arbiter's state)
  ArbParams A;  // its launch parameters (arena offsets inside A.ck)
  Launch L;
};

int plan_base(const gmg* g, const sim_opts_t* o, BasePlan& B) {
  const DevGmg& G = g->dg;
  Launch& L = B.L;
  B.arb = arbitrated(o);
  int rc = B.arb ? plan_arb(g, 1, o, L, B.A, kBase) : plan_launch(g, 1, o, false, L);
  if (rc) return rc;
  L.wpb = 1;
  L.P.dev_bytes = dev_smem_bytes(G.D, 8);  // the base snapshot keeps 64-bit times
  L.smem = smem_per_warp(L.P);
  if (B.arb) {
    B.A.smem_std = (int64_t)L.smem;
    L.smem += (size_t)B.A.smem_arb;
  }
  B.nck = B.arb ? kArbCheckpoints : kCheckpoints;
  B.ckq = std::min(L.P.qcap, kCheckpointQueue);
  B.ckm = std::min(L.P.mcap, kCheckpointLog);
  B.ld = (int)align_up(std::max(G.n, 1), 16);
  B.stride = std::max(1, G.n / (B.nck - 1));
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align_up(off + std::max<size_t>(bytes, 1), 256);
    return at;
  };
  B.off_row = take(B.ld);
  B.off_rb = take(8 * (size_t)G.n);
  B.off_fb = take(8 * (size_t)G.n);
  B.off_status = take(16);
  B.off_res = take(64);
  B.off_peak = take(8 * (size_t)G.D);
  B.off_creq = take(8 * (size_t)G.R);
  B.off_cktime = take(8 * (size_t)B.nck);
  B.off_cksc = take(64 * (size_t)B.nck);
  B.off_ckdev = take(24 * (size_t)G.D * B.nck);
  B.off_ckcreq = take(8 * (size_t)G.R * B.nck);
  B.off_ckqk = take(8 * (size_t)B.ckq * B.nck);
  B.off_ckmk = take(8 * (size_t)B.ckm * B.nck);
  B.off_ckmd = take((size_t)B.ckm * B.nck);
  B.off_arena = 0;
  if (B.arb) {
    // one arena per checkpoint: the arbiter's per-op arrays (times as int64),
    // intents, pair queues, lane and warp state
    ArbCk& K = B.A.ck;
    size_t a = 0;
    auto at = [&](size_t bytes) {
      const size_t r = a;
      a = align_up(a + std::max<size_t>(bytes, 1), 256);
      return (int64_t)r;
    };
    const size_t n = (size_t)G.n, DD = (size_t)G.D * G.D, xc = (size_t)B.A.xcap;
    K.off_cnt = at(4 * n);
    K.off_rmax = at(8 * n);
    K.off_refs = at(4 * n);
    K.off_rmask = at(4 * n);
    K.off_nextop = at(4 * n);
    K.off_hold = at(8 * n);
    K.off_xent = at(4 * xc);
    K.off_xnext = at(4 * xc);
    K.off_qhead = at(4 * DD);
    K.off_qtail = at(4 * DD);
    K.off_lanes = at(7 * 8 * 32);
    K.off_warp = at(4 * 8 + 32 * 4);
    K.bytes = (int64_t)a;
    B.off_arena = take((size_t)K.bytes * B.nck);
  }
  B.off_slot = take((size_t)L.P.slot_bytes);
  B.total = off;
  return GMG_OK;
}

}  // namespace

extern "C" {

size_t gmg_workspace_bytes(const gmg_desc_t* desc) {
  Built b;
  if (build(desc, b) != GMG_OK) return 0;
  return b.L.total;
}

int gmg_create(const gmg_desc_t* desc, void* d_ws, size_t ws_bytes, gmg_stream_t stream, gmg_t** out) {
  if (!out) return GMG_EINVAL;
  *out = nullptr;
  Built b;
  int rc = build(desc, b);
  if (rc) return rc;
  if (!d_ws || !aligned(d_ws, 256) || ws_bytes < b.L.total) return GMG_EWS;
  std::vector<uint8_t> host;
  try {
    host.assign(b.L.total, 0);
  } catch (const std::bad_alloc&) {
    return GMG_ENOMEM;
  }
  const Layout& L = b.L;
  auto put = [&](size_t off, const void* src, size_t bytes) {
    if (bytes) std::memcpy(host.data() + off, src, bytes);
  };
  put(L.off_ops, b.ops.data(), sizeof(OpRec) * b.ops.size());
  put(L.off_succ, b.succ.data(), 4 * b.succ.size());
  put(L.off_pred, b.pred.data(), 4 * b.pred.size());
  {
    std::vector<uint32_t> ps(2 * (size_t)b.E);
    for (int k = 0; k < b.E; ++k) {
      ps[2 * (size_t)k] = b.pred[k];
      ps[2 * (size_t)k + 1] = b.sib[k];
    }
    put(L.off_sib, ps.data(), 4 * ps.size());
  }
  put(L.off_cons, b.cons.data(), 4 * b.cons.size());
  put(L.off_roots, b.roots.data(), 8 * b.roots.size());
  // The batched sweep: graphs on more accelerators than a warp has lanes
  // (accelerator state in shared memory) whose READY keys have room for the
  // duration class; its root keys carry the class of the op's shortest
  // duration over the accelerator types.
  int tb = 1;
  while (tb < 62 && (int64_t(1) << tb) <= b.time_bound) ++tb;
  const bool dev_key = tb + b.ib + 2 + 8 <= 63;
  const bool batch = b.D >= kBatchMinDevices && dev_key && tb + b.ib + 2 + kQB <= 63;
  if (batch) {
    std::vector<uint64_t> rq(b.roots.size());
    for (size_t r = 0; r < b.roots.size(); ++r) {
      const uint32_t i = (uint32_t)(b.roots[r] & ((uint64_t(1) << b.ib) - 1));
      int64_t lo = b.ops[i].dur;
      if (b.T)
        for (int t = 0; t < b.T; ++t) lo = std::min(lo, b.durt[(size_t)i * b.T + t]);
      uint32_t q = 0;
      while (q < 31 && (int64_t(2) << q) <= lo) ++q;
      rq[r] = (b.roots[r] << kQB) | q;
    }
    put(L.off_roots_q, rq.data(), 8 * rq.size());
  }
  put(L.off_cap, b.cap.data(), 8 * b.cap.size());
  put(L.off_base, b.base.data(), 8 * b.base.size());
  put(L.off_avail, b.avail0.data(), 8 * b.avail0.size());
  put(L.off_dl, b.deadline.data(), 8 * b.deadline.size());
  if (!b.uniform) put(L.off_links, b.links.data(), sizeof(LinkRec) * b.links.size());
  if (b.T) {
    put(L.off_durt, b.durt.data(), 8 * b.durt.size());
    put(L.off_dtype, b.dtype.data(), b.dtype.size());
  }
  put(L.off_linkid, b.linkid.data(), 2 * b.linkid.size());
  if (b.stage_ready) {
    put(L.off_st_hot, b.st_hot.data(), 4 * b.st_hot.size());
    put(L.off_st_rel, b.st_rel.data(), 4 * b.st_rel.size());
  }
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(d_ws, host.data(), b.L.total, cudaMemcpyHostToDevice, st) != cudaSuccess)
    return GMG_ECUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return GMG_ECUDA;
  gmg* g = new (std::nothrow) gmg();
  if (!g) return GMG_ENOMEM;
  uint8_t* w = static_cast<uint8_t*>(d_ws);
  DevGmg& G = g->dg;
  G.ops = reinterpret_cast<const OpRec*>(w + L.off_ops);
  G.succ = reinterpret_cast<const uint32_t*>(w + L.off_succ);
  G.pred = reinterpret_cast<const uint32_t*>(w + L.off_pred);
  G.predsib = reinterpret_cast<const uint2*>(w + L.off_sib);
  G.cons = reinterpret_cast<const uint32_t*>(w + L.off_cons);
  G.root_keys = reinterpret_cast<const uint64_t*>(w + L.off_roots);
  G.root_keys_q = reinterpret_cast<const uint64_t*>(w + L.off_roots_q);
  G.cap = reinterpret_cast<const int64_t*>(w + L.off_cap);
  G.base = reinterpret_cast<const int64_t*>(w + L.off_base);
  G.avail0 = reinterpret_cast<const int64_t*>(w + L.off_avail);
  G.deadline = reinterpret_cast<const int64_t*>(w + L.off_dl);
  G.links = b.uniform ? nullptr : reinterpret_cast<const LinkRec*>(w + L.off_links);
  G.ntypes = b.T;
  G.durt = b.T ? reinterpret_cast<const int64_t*>(w + L.off_durt) : nullptr;
  G.dtype = b.T ? w + L.off_dtype : nullptr;
  G.lat0 = b.lat0;
  G.max_iter = b.max_iter;
  G.n = b.n;
  G.D = b.D;
  G.R = b.R;
  G.nroots = b.nroots;
  G.ib = b.ib;
  G.tb = tb;
  G.dev_key = dev_key ? 1 : 0;
  G.batch = batch ? 1 : 0;
  G.st_hot = reinterpret_cast<const uint4*>(w + L.off_st_hot);
  G.st_rel = reinterpret_cast<const int32_t*>(w + L.off_st_rel);
  G.n_edges = b.E;
  G.ws = w;
  G.ws_bytes = (int64_t)L.total;
  // every time < 2^tb fits int32; the 32-bit instances also take the
  // accelerator id from the event key
  G.t32 = (G.tb <= 31 && G.dev_key) ? 1 : 0;
  G.stage_ok = (b.stage_ready && G.t32 && G.D <= 32) ? 1 : 0;
  G.uniform = b.uniform ? 1 : 0;
  gmg_info_t& I = g->info;
  std::memset(&I, 0, sizeof(I));
  I.n_ops = b.n;
  I.n_edges = b.E;
  I.n_dev = b.D;
  I.n_req = b.R;
  I.n_roots = b.nroots;
  I.id_bits = b.ib;
  I.time_bits = 61 - b.ib;
  I.uniform_links = G.uniform;
  I.time_bound = b.time_bound;
  g->queue_bound = b.queue_bound;
  g->log_bound = b.log_bound;
  g->linkid = b.linkid.empty() ? nullptr : reinterpret_cast<const uint16_t*>(w + L.off_linkid);
  g->xfer_bound = b.xfer_bound;
  g->shared_links = b.shared_links ? 1 : 0;
  I.default_queue_cap = std::min<int64_t>(b.queue_bound, kDefaultQueueCap);
  I.batched_sweep = G.batch;
  I.t32 = G.t32;
  // staged only where the copy also fits beside a warp's areas on this device
  I.stageable = 0;
  if (G.stage_ok) {
    Launch Ls;
    I.stageable = plan_staged(g, 1, nullptr, Ls) == GMG_OK ? 1 : 0;
  }
  *out = g;
  return GMG_OK;
}

void gmg_destroy(gmg_t* g) { delete g; }

int gmg_get_info(const gmg_t* g, gmg_info_t* info) {
  if (!g || !info) return GMG_EINVAL;
  *info = g->info;
  return GMG_OK;
}

size_t sim_scratch_bytes(const gmg_t* g, int32_t K, const sim_opts_t* opts) {
  if (!g || K < 0) return 0;
  Launch L;
  if (arbitrated(opts)) {
    ArbPlan Q;
    if (plan_arb_any(g, K, opts, L, Q)) return 0;
  } else {
    bool stg = false;
    if (plan_full(g, K, opts, L, &stg)) return 0;
  }
  return (size_t)L.slots * (size_t)L.P.slot_bytes;
}

int sim_batch(const gmg_t* g, const uint8_t* d_place, int32_t K, int32_t ld, const sim_opts_t* opts,
              const sim_out_t* d_out, void* d_scratch, size_t scratch_bytes, gmg_stream_t stream) {
  if (!g || K < 0) return GMG_EINVAL;
  int rc = check_out(d_out, opts);
  if (rc) return rc;
  if (K == 0) return GMG_OK;
  if (!d_place || ld < g->dg.n || ld % 16 != 0 || !aligned(d_place, 16)) return GMG_EINVAL;
  Launch L;
  ArbPlan Q;
  const bool arb = arbitrated(opts);
  bool stg = false;
  rc = arb ? (staged(opts) ? GMG_EINVAL : plan_arb_any(g, K, opts, L, Q)) : plan_full(g, K, opts, L, &stg);
  if (rc) return rc;
  if (!d_scratch || !aligned(d_scratch, 256) ||
      scratch_bytes < (size_t)L.slots * (size_t)L.P.slot_bytes)
    return GMG_EWS;
  SimParams& P = L.P;
  fill_out(P, d_out, opts);
  P.place = d_place;
  P.ld = ld;
  P.K = K;
  P.scratch = static_cast<uint8_t*>(d_scratch);
  const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = arb ? launch_arb_any(g, L, Q, nullptr, st)
                      : stg ? launch_full_staged(P, L.grid, 32 * L.wpb, L.smem, st)
                            : launch_full(L.reg, P, L.grid, 32 * L.wpb, L.smem, st);
  return e == cudaSuccess ? GMG_OK : GMG_ECUDA;
}

// ---------------------------------------------------------------------------
// sim_batch_noalloc: sim_batch for callers that cannot allocate device memory.
//
// Its per-warp scratch is a fixed buffer that lives in the library itself
// (below), so a caller hands over only the placements and the output arrays.
// The buffer is GMG_NOALLOC_SCRATCH_BYTES large and exists on every GPU that
// loads the library until the process exits.  Every call reuses it and finds
// the previous call's contents there; the kernel initialises every scratch
// word it reads for each candidate, so nothing has to be cleared between
// calls.  Two calls whose kernels could overlap on the GPU would race on the
// buffer: order them on one stream (or with events).
// ---------------------------------------------------------------------------
static __device__ __align__(256) uint8_t g_noalloc_scratch[GMG_NOALLOC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
void* g_noalloc_ptr[kMaxDevices] = {};

// The buffer's device address on the current device.  Host code may not use
// the symbol itself as an address, so the runtime is asked once per device
// (with that device current) and the answer is kept.
int noalloc_scratch(uint8_t** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return GMG_ECUDA;
  if (dev < 0 || dev >= kMaxDevices) return GMG_ECUDA;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return GMG_ECUDA;
    g_noalloc_ptr[dev] = p;
  }
  *out = static_cast<uint8_t*>(g_noalloc_ptr[dev]);
  return GMG_OK;
}

}  // namespace

extern "C" int sim_batch_noalloc(const gmg_t* g, const uint8_t* d_place, int32_t K, int32_t ld,
                                 const sim_opts_t* opts, const sim_out_t* d_out, gmg_stream_t stream) {
  if (!g || K < 0) return GMG_EINVAL;
  int rc = check_out(d_out, opts);
  if (rc) return rc;
  if (K == 0) return GMG_OK;
  if (!d_place || ld < g->dg.n || ld % 16 != 0 || !aligned(d_place, 16)) return GMG_EINVAL;
  if (staged(opts)) return GMG_EINVAL;  // the staged copy's CTA shape is not planned for the fixed buffer
  Launch L;
  ArbPlan Q;
  const bool arb = arbitrated(opts);
  rc = arb ? plan_arb_any(g, K, opts, L, Q) : plan_launch(g, K, opts, false, L);
  if (rc) return rc;
  // As many warp slots as the fixed buffer holds (each warp then takes more
  // candidates in turn); a graph whose single slot does not fit is refused.
  const int64_t fit = (int64_t)(GMG_NOALLOC_SCRATCH_BYTES / (size_t)L.P.slot_bytes);
  if (fit < 1) return GMG_EWS;
  if (fit < L.wpb) {
    sim_opts_t one = opts ? *opts : sim_opts_t{};
    one.warps_per_block = 1;
    rc = arb ? plan_arb_any(g, K, &one, L, Q) : plan_launch(g, K, &one, false, L);
    if (rc) return rc;
  }
  L.grid = (int)std::min<int64_t>(L.grid, fit / L.wpb);
  uint8_t* scratch = nullptr;
  rc = noalloc_scratch(&scratch);
  if (rc) return rc;
  SimParams& P = L.P;
  fill_out(P, d_out, opts);
  P.place = d_place;
  P.ld = ld;
  P.K = K;
  P.scratch = scratch;
  const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const cudaError_t e = arb ? launch_arb_any(g, L, Q, nullptr, st) : launch_full(L.reg, P, L.grid, 32 * L.wpb, L.smem, st);
  return e == cudaSuccess ? GMG_OK : GMG_ECUDA;
}

size_t base_workspace_bytes(const gmg_t* g, const sim_opts_t* opts) {
  if (!g) return 0;
  BasePlan B;
  if (plan_base(g, opts, B)) return 0;
  return B.total;
}

int base_create(const gmg_t* g, const uint8_t* d_base_place, const sim_opts_t* opts, void* d_base_ws,
                size_t ws_bytes, gmg_stream_t stream, gmg_base_t** out) {
  if (!out) return GMG_EINVAL;
  *out = nullptr;
  if (!g || !d_base_place || !aligned(d_base_place, 16)) return GMG_EINVAL;
  if (opts) {
    for (int r : opts->reserved)
      if (r != 0) return GMG_EINVAL;
    if (opts->transfer_mode != GMG_TRANSFER_LATENCY && opts->transfer_mode != GMG_TRANSFER_ARBITRATED)
      return GMG_EINVAL;
    if (opts->gmg_staging == GMG_STAGING_SHARED) return GMG_EINVAL;
  }
  BasePlan B;
  int rc = plan_base(g, opts, B);
  if (rc) return rc;
  if (!d_base_ws || !aligned(d_base_ws, 256) || ws_bytes < B.total) return GMG_EWS;
  gmg_base* b = new (std::nothrow) gmg_base();
  if (!b) return GMG_ENOMEM;
  uint8_t* w = static_cast<uint8_t*>(d_base_ws);
  DevBase& D = b->db;
  D.row = w + B.off_row;
  D.rb = reinterpret_cast<int64_t*>(w + B.off_rb);
  D.fb = reinterpret_cast<int64_t*>(w + B.off_fb);
  D.status = reinterpret_cast<int32_t*>(w + B.off_status);
  D.res_scalars = reinterpret_cast<int64_t*>(w + B.off_res);
  D.res_peak = reinterpret_cast<int64_t*>(w + B.off_peak);
  D.res_creq = reinterpret_cast<int64_t*>(w + B.off_creq);
  D.ck_time = reinterpret_cast<int64_t*>(w + B.off_cktime);
  D.ck_scalars = reinterpret_cast<int64_t*>(w + B.off_cksc);
  D.ck_dev = reinterpret_cast<int64_t*>(w + B.off_ckdev);
  D.ck_creq = reinterpret_cast<int64_t*>(w + B.off_ckcreq);
  D.ck_qkey = reinterpret_cast<uint64_t*>(w + B.off_ckqk);
  D.ck_mkey = reinterpret_cast<uint64_t*>(w + B.off_ckmk);
  D.ck_mdev = w + B.off_ckmd;
  D.nck = B.nck;
  D.ckq = B.ckq;
  D.ckm = B.ckm;
  D.ld = B.ld;
  D.stride_pops = B.stride;
  b->g = g;
  b->slot = w + B.off_slot;
  b->qs = B.L.P.qs;
  b->qcap = B.L.P.qcap;
  b->arb = B.arb ? 1 : 0;
  SimParams P = B.L.P;
  P.base = D;
  P.place = d_base_place;
  P.ld = B.ld;
  P.K = 1;
  P.scratch = b->slot;
  cudaError_t e;
  if (B.arb) {
    ArbParams A = B.A;
    A.P = P;
    A.ck.arena = w + B.off_arena;
    b->ck = A.ck;
    e = launch_arb_base(g->dg.ntypes >= 2, A, B.L.smem, reinterpret_cast<cudaStream_t>(stream));
  } else {
    e = launch_base(B.L.reg, P, B.L.smem, reinterpret_cast<cudaStream_t>(stream));
  }
  if (e != cudaSuccess) {
    delete b;
    return GMG_ECUDA;
  }
  *out = b;
  return GMG_OK;
}

void base_destroy(gmg_base_t* b) { delete b; }

// Arbitrated incremental candidates: [moved rows K x ld | move statuses K | slots].
static size_t arb_inc_bytes(const gmg_t* g, int32_t K, const sim_opts_t* opts, size_t* off_status, size_t* off_slots) {
  Launch L;
  ArbPlan Q;
  if (plan_arb_any(g, K, opts, L, Q)) return 0;
  const size_t ld = align_up((size_t)std::max(g->dg.n, 1), 16);
  const size_t os = align_up((size_t)K * ld, 256);
  const size_t oz = os + align_up(4 * (size_t)std::max(K, 1), 256);
  if (off_status) *off_status = os;
  if (off_slots) *off_slots = oz;
  return oz + (size_t)L.slots * (size_t)L.P.slot_bytes;
}

// Candidates resumed from an arbitrated base snapshot (at most 32 accelerators).
static int plan_arb_resumed(const gmg_t* g, int32_t K, const sim_opts_t* opts, Launch& L, ArbParams& A) {
  return plan_arb(g, K, opts, L, A, kInc);
}

size_t inc_scratch_bytes(const gmg_t* g, int32_t K, const sim_opts_t* opts) {
  if (!g || K < 0) return 0;
  if (arbitrated(opts)) {
    // enough for either base: a pure-latency one (moved rows simulated in
    // full) or an arbitrated one (candidates resumed from it)
    size_t need = arb_inc_bytes(g, K, opts, nullptr, nullptr);
    Launch L;
    ArbParams A;
    if (g->dg.D <= 32 && plan_arb_resumed(g, K, opts, L, A) == GMG_OK)
      need = std::max(need, kCounterBytes + (size_t)L.slots * (size_t)L.P.slot_bytes);
    return need;
  }
  Launch L;
  if (plan_launch(g, K, opts, true, L)) return 0;
  return kCounterBytes + (size_t)L.slots * (size_t)L.P.slot_bytes;
}

// A resumed incremental launch's scratch: the candidate counter, zeroed on
// the stream, then the slots.
static int take_counter(SimParams& P, void* d_scratch, size_t scratch_bytes, const Launch& L, cudaStream_t st) {
  if (!d_scratch || !aligned(d_scratch, 256) ||
      scratch_bytes < kCounterBytes + (size_t)L.slots * (size_t)L.P.slot_bytes)
    return GMG_EWS;
  P.next_k = static_cast<uint32_t*>(d_scratch);
  P.scratch = static_cast<uint8_t*>(d_scratch) + kCounterBytes;
  return cudaMemsetAsync(P.next_k, 0, sizeof(uint32_t), st) == cudaSuccess ? GMG_OK : GMG_ECUDA;
}

int sim_incremental(const gmg_t* g, const gmg_base_t* b, const int32_t* d_move_off, const int32_t* d_move_op,
                    const uint8_t* d_move_dev, int32_t K, const sim_opts_t* opts, const sim_out_t* d_out,
                    void* d_scratch, size_t scratch_bytes, gmg_stream_t stream) {
  if (!g || !b || b->g != g || K < 0) return GMG_EINVAL;
  int rc = check_out(d_out, opts);
  if (rc) return rc;
  if (staged(opts)) return GMG_EINVAL;  // staging applies to sim_batch
  if (K == 0) return GMG_OK;
  if (!d_move_off) return GMG_EINVAL;
  if (b->arb && !arbitrated(opts)) return GMG_EINVAL;  // an arbitrated snapshot serves arbitrated candidates
  if (b->arb) {
    // resumed from the arbitrated base snapshot
    Launch L;
    ArbParams A;
    rc = plan_arb_resumed(g, K, opts, L, A);
    if (rc) return rc;
    SimParams& P = L.P;
    rc = take_counter(P, d_scratch, scratch_bytes, L, reinterpret_cast<cudaStream_t>(stream));
    if (rc) return rc;
    fill_out(P, d_out, opts);
    P.base = b->db;
    P.ld = b->db.ld;
    P.K = K;
    P.move_off = d_move_off;
    P.move_op = d_move_op;
    P.move_dev = d_move_dev;
    A.P = P;
    A.ck = b->ck;
    A.pre_status = nullptr;
    return launch_arb_inc(g->dg.t32 != 0, g->dg.ntypes >= 2, A, L.grid, 32 * L.wpb, L.smem,
                          reinterpret_cast<cudaStream_t>(stream)) == cudaSuccess
               ? GMG_OK
               : GMG_ECUDA;
  }
  if (arbitrated(opts)) {
    // Arbitrated transfers: every candidate's moved placement is simulated in
    // full (the base snapshot's resume points hold no transfer state).
    size_t os = 0, oz = 0;
    const size_t need = arb_inc_bytes(g, K, opts, &os, &oz);
    if (need == 0) {
      Launch L0;
      ArbPlan Q0;
      const int prc = plan_arb_any(g, K, opts, L0, Q0);
      return prc ? prc : GMG_EINVAL;
    }
    if (!d_scratch || !aligned(d_scratch, 256) || scratch_bytes < need) return GMG_EWS;
    Launch L;
    ArbPlan Q;
    rc = plan_arb_any(g, K, opts, L, Q);
    if (rc) return rc;
    uint8_t* sc = static_cast<uint8_t*>(d_scratch);
    const int32_t ld = b->db.ld;
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (launch_expand_moves(b->db.row, b->db.status, ld, g->dg.n, g->dg.D, d_move_off, d_move_op, d_move_dev, K,
                            sc, reinterpret_cast<int32_t*>(sc + os), st) != cudaSuccess)
      return GMG_ECUDA;
    SimParams& P = L.P;
    fill_out(P, d_out, opts);
    P.place = sc;
    P.ld = ld;
    P.K = K;
    P.scratch = sc + oz;
    return launch_arb_any(g, L, Q, reinterpret_cast<const int32_t*>(sc + os), st) == cudaSuccess ? GMG_OK
                                                                                                : GMG_ECUDA;
  }
  Launch L;
  rc = plan_launch(g, K, opts, true, L);
  if (rc) return rc;
  SimParams& P = L.P;
  rc = take_counter(P, d_scratch, scratch_bytes, L, reinterpret_cast<cudaStream_t>(stream));
  if (rc) return rc;
  fill_out(P, d_out, opts);
  P.base = b->db;
  P.ld = b->db.ld;
  P.K = K;
  P.move_off = d_move_off;
  P.move_op = d_move_op;
  P.move_dev = d_move_dev;
  cudaError_t e = launch_inc(L.reg, P, L.grid, 32 * L.wpb, L.smem, reinterpret_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? GMG_OK : GMG_ECUDA;
}

size_t select_best_tmp_bytes(int32_t K) {
  if (K < 0) return 0;
  const int nparts = (int)std::min<int64_t>(std::max<int64_t>((K + 255) / 256, 1), 1024);
  return (size_t)nparts * select_rank_bytes();
}

int select_best(const sim_out_t* d_out, int32_t K, int32_t score_mode, int64_t* d_best, void* d_tmp,
                size_t tmp_bytes, gmg_stream_t stream) {
  if (!d_out || !d_best || K < 0 || (score_mode != 0 && score_mode != 1)) return GMG_EINVAL;
  if (!d_out->status || !d_out->viol_flag || !d_out->score || !d_out->sla_miss) return GMG_EINVAL;
  const int nparts = (int)std::min<int64_t>(std::max<int64_t>((K + 255) / 256, 1), 1024);
  if (!d_tmp || tmp_bytes < (size_t)nparts * select_rank_bytes() || !aligned(d_tmp, 16)) return GMG_EWS;
  cudaError_t e = launch_select(d_out->status, d_out->viol_flag, d_out->score, d_out->sla_miss, K,
                                score_mode, d_tmp, nparts, d_best, reinterpret_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? GMG_OK : GMG_ECUDA;
}

const char* gmg_strerror(int code) {
  switch (code) {
    case GMG_OK: return "ok";
    case GMG_EINVAL: return "invalid argument or graph";
    case GMG_ENOTTOPO: return "predecessor id not smaller than its op id";
    case GMG_ERANGE: return "times or byte totals exceed the supported range";
    case GMG_EWS: return "workspace or scratch too small or misaligned";
    case GMG_ECUDA: return "CUDA runtime error";
    case GMG_ENOMEM: return "host allocation failed";
    case GMG_SIM_BADDEV: return "candidate: placement device id out of range";
    case GMG_SIM_MOVE_RANGE: return "candidate: move op or device out of range";
    case GMG_SIM_MOVE_DUP: return "candidate: op moved twice";
    case GMG_SIM_BADBASE: return "candidate: invalid base placement";
    case GMG_SIM_QUEUE: return "candidate: event queue capacity exceeded";
    case GMG_SIM_LOOP: return "candidate: event loop iteration cap exceeded";
    default: return "unknown code";
  }
}

int64_t gmg_ceil_div_host(int64_t n, int64_t d) {
  if (n < 0 || d < 1 || n >= (int64_t(1) << 53) || d >= (int64_t(1) << 62)) return -1;
  return ceil_div_link(n, make_link(d, 0));
}

}  // extern "C"
