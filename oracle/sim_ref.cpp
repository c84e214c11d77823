// CPU oracle for the what-if placement simulation of the Global Simulator.
//
// TEST INFRASTRUCTURE ONLY.  This file is the plain, slow reference that the
// CUDA path is checked against.  Only the test suite, the smoke check and the
// CPU-baseline leg of the benchmark may load it; the product library never
// calls, links or includes it, and it includes nothing of the product.
//
// What it computes, and where the paper defines it:
//
//  * Ready time (Sec. 3.3.2, "Simulator Construction"): an issued operator
//    becomes ready once every predecessor is done and its output has arrived
//    in local HBM: local predecessors contribute their completion time,
//    remote ones the arrival time of the transferred output.  Its own arrival
//    (release) time is one more input.
//  * Transfer estimator (Sec. 3.3.1): t = alpha * size + c per accelerator
//    pair, here in integer form ceil(size / bw[d][e]) + lat[d][e], 0 on the
//    same accelerator.  Integer durations stand in for the operator
//    estimator's output; the operator estimator is kept per (accelerator
//    type, operator), so with several accelerator types an operator's
//    duration is the one of the type it is placed on.
//  * Queue rule (Sec. 3.3.2 and Sec. 3.5.1): each accelerator queue runs at
//    most one operator at a time; the operator started is the ready, issued
//    one with the earliest ready time (ties: lowest op id).
//  * Event-driven simulation (Sec. 3.3.3): keep the running operators with
//    their predicted completion times, repeatedly take the earliest
//    completion, apply its cascade (successor inputs arrive), and start one
//    ready operator on the freed queue.  Equal-time order: completions (by op
//    id), then arrivals, then dispatch on every idle accelerator.
//  * HBM residency (Sec. 3.3.2; Recv allocates before Send, Sec. 3.5.2): an
//    operator's output is allocated on its accelerator when it starts; a
//    receive copy is allocated on every other accelerator that runs a
//    successor when the transfer starts (at the producer's completion); a
//    copy is released when the last listed consumer on that accelerator
//    finishes, and not before its transfer has arrived (source copy: not
//    before every outgoing transfer has arrived, nor before the producer
//    finishes).  Frees precede allocations at equal times.
//  * Feasibility and score (Sec. 3.4.2, Algorithm 1): a placement whose
//    simulated HBM use exceeds an accelerator's capacity is discarded; among
//    the rest the one with the smallest average completion time of the
//    scored operators wins (sum of finish times, same argmin), ties to the
//    lowest candidate index.
//  * Arbitrated transfers (Sec. 3.5.2, "Tensor Transfer Arbitration"; the
//    transfer_mode = 1 variant).  A producer's completion raises one transfer
//    intent per distinct remote accelerator of its successors.  The master
//    keeps the pending intents and activates a conflict-free set of them at
//    every trigger: the arrival of an intent or the completion of a
//    transfer.  An active transfer s -> e holds s's sending endpoint, e's
//    receiving endpoint and the communication link of the pair (link ids are
//    an input; by default every ordered pair has its own link).  The paper
//    leaves the choice among conflicting intents open; here, after every
//    completion and intent at time t, the pending intents are visited in
//    (intent time, producer id, destination id) order and each one that
//    conflicts with no active transfer starts at t.  It lasts the transfer
//    estimate; the receive buffer (Recv) is allocated when it starts, and the
//    consumers' input arrives when it completes.
//  * Incremental what-if (Sec. 3.4.2): a candidate given as moves against a
//    base placement is, by definition, the full simulation of the moved
//    placement; its event count is the number of operators whose base ready
//    time is at or after the resume time T0 = min over moved ops x of
//    (min over predecessors p of the base finish of p, or x's release if it
//    has none).  With arbitrated transfers the moved placement is simulated
//    in full and the event count is the number of operators.
//
// Everything is int64; no floating point is involved.

#include <algorithm>
#include <cstdint>
#include <cstring>
#include <functional>
#include <limits>
#include <map>
#include <queue>
#include <set>
#include <thread>
#include <tuple>
#include <vector>

namespace {

constexpr int64_t kI64Max = std::numeric_limits<int64_t>::max();

// Error codes of orc_check (same meaning as the library's, defined here
// independently).
constexpr int kEInval = -1;
constexpr int kENotTopo = -2;
constexpr int kERange = -3;

// Per-candidate status codes.
constexpr int32_t kSimOk = 0;
constexpr int32_t kSimBadDev = 1;
constexpr int32_t kSimMoveRange = 2;
constexpr int32_t kSimMoveDup = 3;
constexpr int32_t kSimBadBase = 4;

}  // namespace

extern "C" {

typedef struct {
  int32_t n_ops, n_edges, n_dev, n_req;
  const int32_t* pred_off;
  const int32_t* pred_idx;
  const int32_t* cons_off;   // NULL: consumers = successors
  const int32_t* cons_idx;
  const int64_t* dur;
  const int64_t* out_bytes;
  const int64_t* release;    // NULL: 0
  const int32_t* req_id;     // NULL: -1
  const uint8_t* scored;     // NULL: all scored
  const int64_t* deadline;   // NULL: none
  const int64_t* cap;        // NULL: unlimited
  const int64_t* base;       // NULL: 0
  const int64_t* avail0;     // NULL: 0
  const int64_t* bw;         // n_dev*n_dev, row = source
  const int64_t* lat;
  int32_t n_types;           // >= 2: durations per (op, accelerator type)
  const uint8_t* dev_type;   // [n_dev]
  const int64_t* dur_type;   // [n_ops * n_types], op-major
  int32_t transfer_mode;     // 0 = transfers are pure latency, 1 = arbitrated
  const int32_t* link_id;    // [n_dev*n_dev] link of each ordered pair; NULL: its own
} orc_graph;

typedef struct {
  int32_t status;
  int32_t viol_flag;
  int32_t viol_op;
  int32_t viol_dev;
  int64_t viol_time;
  int64_t makespan;
  int64_t score;
  int64_t events;
  int32_t sla_miss;
  int32_t reserved;
} orc_summary;

}  // extern "C"

namespace {

// A validated graph with derived successor and consumer lists.
struct Graph {
  int n = 0, e = 0, D = 0, R = 0;
  std::vector<std::vector<int>> pred, succ, cons;
  std::vector<int64_t> dur, bytes, release, deadline, cap, base, avail0, bw, lat;
  std::vector<int> req;
  std::vector<uint8_t> scored;
  int T = 0;                     // accelerator types (0: one type, dur)
  std::vector<uint8_t> dev_type;  // [D]
  std::vector<int64_t> dur_type;  // [n*T]
  int mode = 0;                   // 1: arbitrated transfers
  std::vector<int> link;          // [D*D] link id of each ordered pair
};

// Duration of op i on accelerator d.
int64_t dur_on(const Graph& g, int i, int d) {
  return g.T ? g.dur_type[size_t(i) * g.T + g.dev_type[d]] : g.dur[i];
}

int64_t ceil_div(int64_t a, int64_t b) {
  int64_t q = a / b;
  return (q * b == a) ? q : q + 1;
}

// Transfer estimator: 0 on the same accelerator, else ceil(bytes/bw) + lat.
int64_t xfer(const Graph& g, int d, int e, int64_t b) {
  if (d == e) return 0;
  return ceil_div(b, g.bw[size_t(d) * g.D + e]) + g.lat[size_t(d) * g.D + e];
}

int build(const orc_graph* in, Graph& g) {
  if (!in) return kEInval;
  const int n = in->n_ops, D = in->n_dev, R = in->n_req;
  if (n < 0 || in->n_edges < 0 || D < 1 || D > 256 || R < 0) return kEInval;
  if (!in->pred_off || (in->n_edges > 0 && !in->pred_idx)) return kEInval;
  if (in->n_types < 0 || in->n_types > 256) return kEInval;
  g.T = in->n_types >= 2 ? in->n_types : 0;
  if (g.T && (!in->dev_type || (n > 0 && !in->dur_type))) return kEInval;
  if (n > 0 && ((!g.T && !in->dur) || !in->out_bytes)) return kEInval;
  if (D > 1 && (!in->bw || !in->lat)) return kEInval;
  g.n = n; g.e = in->n_edges; g.D = D; g.R = R;
  if (in->pred_off[0] != 0 || in->pred_off[n] != in->n_edges) return kEInval;
  for (int i = 0; i < n; ++i)
    if (in->pred_off[i + 1] < in->pred_off[i]) return kEInval;
  g.pred.assign(n, {});
  g.succ.assign(n, {});
  for (int i = 0; i < n; ++i) {
    int a = in->pred_off[i], b = in->pred_off[i + 1];
    for (int k = a; k < b; ++k) {
      int p = in->pred_idx[k];
      if (p < 0 || p >= n) return kEInval;
      if (p >= i) return kENotTopo;
      g.pred[i].push_back(p);
    }
    std::vector<int> s = g.pred[i];
    std::sort(s.begin(), s.end());
    if (std::adjacent_find(s.begin(), s.end()) != s.end()) return kEInval;
    for (int p : g.pred[i]) g.succ[p].push_back(i);
  }
  g.cons.assign(n, {});
  if (in->cons_off) {
    if (in->cons_off[0] != 0) return kEInval;
    for (int i = 0; i < n; ++i)
      if (in->cons_off[i + 1] < in->cons_off[i]) return kEInval;
    if (in->cons_off[n] > 0 && !in->cons_idx) return kEInval;
    for (int i = 0; i < n; ++i) {
      int a = in->cons_off[i], b = in->cons_off[i + 1];
      std::set<int> seen;
      for (int k = a; k < b; ++k) {
        int c = in->cons_idx[k];
        if (c < 0 || c >= n) return kEInval;
        if (std::find(g.succ[i].begin(), g.succ[i].end(), c) == g.succ[i].end()) return kEInval;
        if (!seen.insert(c).second) return kEInval;
        g.cons[i].push_back(c);
      }
    }
  } else {
    g.cons = g.succ;
  }
  g.dur.resize(n); g.bytes.resize(n); g.release.resize(n); g.req.resize(n); g.scored.resize(n);
  for (int i = 0; i < n; ++i) {
    if (g.T) {
      // an op's longest duration over the types bounds its times
      g.dur[i] = 0;
      for (int t = 0; t < g.T; ++t) {
        const int64_t v = in->dur_type[size_t(i) * g.T + t];
        if (v < 1) return kEInval;
        g.dur[i] = std::max(g.dur[i], v);
      }
    } else {
      g.dur[i] = in->dur[i];
    }
    g.bytes[i] = in->out_bytes[i];
    g.release[i] = in->release ? in->release[i] : 0;
    g.req[i] = in->req_id ? in->req_id[i] : -1;
    g.scored[i] = in->scored ? in->scored[i] : 1;
    if (g.dur[i] < 1 || g.bytes[i] < 0 || g.release[i] < 0) return kEInval;
    if (g.req[i] < -1 || g.req[i] >= R) return kEInval;
    if (g.scored[i] > 1) return kEInval;
  }
  g.deadline.resize(R);
  for (int r = 0; r < R; ++r) g.deadline[r] = in->deadline ? in->deadline[r] : kI64Max;
  g.cap.resize(D); g.base.resize(D); g.avail0.resize(D);
  for (int d = 0; d < D; ++d) {
    g.cap[d] = in->cap ? in->cap[d] : kI64Max;
    g.base[d] = in->base ? in->base[d] : 0;
    g.avail0[d] = in->avail0 ? in->avail0[d] : 0;
    if (g.cap[d] < 0 || g.base[d] < 0 || g.base[d] > g.cap[d] || g.avail0[d] < 0) return kEInval;
  }
  if (g.T) {
    g.dev_type.assign(in->dev_type, in->dev_type + D);
    for (int d = 0; d < D; ++d)
      if (g.dev_type[d] >= g.T) return kEInval;
    g.dur_type.assign(in->dur_type, in->dur_type + size_t(n) * g.T);
  }
  g.bw.assign(size_t(D) * D, 1);
  g.lat.assign(size_t(D) * D, 0);
  for (int d = 0; d < D; ++d)
    for (int e = 0; e < D; ++e) {
      if (d == e) continue;
      g.bw[size_t(d) * D + e] = in->bw[size_t(d) * D + e];
      g.lat[size_t(d) * D + e] = in->lat[size_t(d) * D + e];
      if (g.bw[size_t(d) * D + e] < 1 || g.lat[size_t(d) * D + e] < 0) return kEInval;
    }
  if (in->transfer_mode < 0 || in->transfer_mode > 1) return kEInval;
  g.mode = in->transfer_mode;
  g.link.assign(size_t(D) * D, 0);
  for (int d = 0; d < D; ++d)
    for (int e = 0; e < D; ++e) {
      const size_t k = size_t(d) * D + e;
      g.link[k] = in->link_id ? in->link_id[k] : int(k);
      if (d != e && (g.link[k] < 0 || g.link[k] >= D * D)) return kEInval;
    }
  // Overflow guard: every time stays below (start + all durations + one
  // transfer per edge and per op), every score below n times that, every
  // live-memory figure below base + every copy of every tensor.
  using i128 = __int128;
  const i128 lim = i128(1) << 62;
  int64_t min_bw = kI64Max, max_lat = 0;
  for (int d = 0; d < D; ++d)
    for (int e = 0; e < D; ++e)
      if (d != e) {
        min_bw = std::min(min_bw, g.bw[size_t(d) * D + e]);
        max_lat = std::max(max_lat, g.lat[size_t(d) * D + e]);
      }
  if (D == 1) min_bw = 1;
  i128 t = 0, mem = 0;
  for (int d = 0; d < D; ++d) {
    t = std::max<i128>(t, g.avail0[d]);
    mem += g.base[d];
  }
  for (int i = 0; i < n; ++i) t = std::max<i128>(t, g.release[i]);
  for (int i = 0; i < n; ++i) {
    i128 mx = i128(g.bytes[i] / min_bw + 1) + max_lat;
    t += g.dur[i] + mx * i128(g.succ[i].size() + 1);
    mem += i128(g.bytes[i]) * i128(g.succ[i].size() + 1);
    if (t >= lim || mem >= lim) return kERange;
  }
  if (t * i128(std::max(n, 1)) >= lim) return kERange;
  return 0;
}

// One cross-accelerator transfer of op p's output to accelerator e.
struct Transfer {
  int p, e;
  int64_t intent, start, done;
};

struct Result {
  orc_summary s;
  std::vector<int64_t> peak, req_done, ready, start, finish;
  std::vector<Transfer> xfers;  // arbitrated mode: every transfer
};

// A copy of op i's output on another accelerator: allocated when its
// transfer starts, present there once the transfer has arrived.
struct Copy {
  int e;
  int64_t alloc, arrive;
};

void fill_invalid(const Graph& g, int32_t status, Result& res) {
  res.s = orc_summary{};
  res.s.status = status;
  res.s.viol_op = -1;
  res.s.viol_dev = -1;
  res.s.viol_time = -1;
  res.s.score = kI64Max;
  res.peak.assign(g.D, 0);
  res.req_done.assign(g.R, 0);
  res.ready.assign(g.n, 0);
  res.start.assign(g.n, 0);
  res.finish.assign(g.n, 0);
}

// HBM residency, request completion, score and summary of one simulated
// placement, given every op's ready, start and finish time and the remote
// copies of every op's output (Sec. 3.3.2, Sec. 3.4.2).
void settle(const Graph& g, const uint8_t* dev, std::vector<int64_t>& r, std::vector<int64_t>& s,
            std::vector<int64_t>& f, const std::vector<std::vector<Copy>>& copies, Result& res) {
  const int n = g.n, D = g.D;
  // per accelerator, every copy is an interval [alloc, free)
  struct MemEv {
    int64_t t;
    int cls;  // 0 = free, 1 = alloc (frees first at equal times)
    int op;
    int64_t delta;
  };
  std::vector<std::vector<MemEv>> mem(D);
  for (int i = 0; i < n; ++i) {
    const int d = dev[i];
    const int64_t b = g.bytes[i];
    std::map<int, int64_t> last_use;  // accelerator -> latest finish of a listed consumer
    for (int c : g.cons[i]) {
      auto it = last_use.find(dev[c]);
      if (it == last_use.end()) last_use[dev[c]] = f[c];
      else it->second = std::max(it->second, f[c]);
    }
    int64_t src_free = f[i];
    for (const Copy& c : copies[i]) src_free = std::max(src_free, c.arrive);
    if (last_use.count(d)) src_free = std::max(src_free, last_use[d]);
    mem[d].push_back({s[i], 1, i, b});
    mem[d].push_back({src_free, 0, i, -b});
    for (const Copy& c : copies[i]) {
      int64_t t_free = c.arrive;
      if (last_use.count(c.e)) t_free = std::max(t_free, last_use[c.e]);
      mem[c.e].push_back({c.alloc, 1, i, b});
      mem[c.e].push_back({t_free, 0, i, -b});
    }
  }
  res.peak.assign(D, 0);
  bool viol = false;
  int64_t vt = 0;
  int vop = -1, vdev = -1;
  for (int d = 0; d < D; ++d) {
    std::sort(mem[d].begin(), mem[d].end(), [](const MemEv& a, const MemEv& b) {
      return std::tie(a.t, a.cls, a.op) < std::tie(b.t, b.cls, b.op);
    });
    int64_t live = g.base[d], peak = g.base[d];
    for (const MemEv& e : mem[d]) {
      live += e.delta;
      if (e.cls == 1) {
        peak = std::max(peak, live);
        if (live > g.cap[d]) {
          auto key = std::make_tuple(e.t, e.op, d);
          if (!viol || key < std::make_tuple(vt, vop, vdev)) {
            viol = true; vt = e.t; vop = e.op; vdev = d;
          }
        }
      }
    }
    res.peak[d] = peak;
  }

  // Per-request completion and SLA.
  res.req_done.assign(g.R, 0);
  for (int i = 0; i < n; ++i)
    if (g.req[i] >= 0) res.req_done[g.req[i]] = std::max(res.req_done[g.req[i]], f[i]);
  int32_t miss = 0;
  for (int q = 0; q < g.R; ++q) miss += res.req_done[q] > g.deadline[q] ? 1 : 0;

  int64_t makespan = 0, score = 0;
  for (int i = 0; i < n; ++i) {
    makespan = std::max(makespan, f[i]);
    if (g.scored[i]) score += f[i];
  }
  res.s = orc_summary{};
  res.s.status = kSimOk;
  res.s.viol_flag = viol ? 1 : 0;
  res.s.viol_op = viol ? vop : -1;
  res.s.viol_dev = viol ? vdev : -1;
  res.s.viol_time = viol ? vt : -1;
  res.s.makespan = makespan;
  res.s.score = viol ? kI64Max : score;
  res.s.events = n;
  res.s.sla_miss = miss;
  res.ready = std::move(r);
  res.start = std::move(s);
  res.finish = std::move(f);
}


// Sec. 3.3.3 with the arbitrated transfers of Sec. 3.5.2: the same
// event-driven loop, where a remote input arrives when its transfer, started
// by the arbiter, completes.  Equal-time order: operator and transfer
// completions, new intents, arbitration (repeated while a transfer started
// at this time also completes at it), then input arrivals, then dispatch on
// every idle accelerator.
void simulate_arb(const Graph& g, const uint8_t* dev, Result& res) {
  const int n = g.n, D = g.D;
  std::vector<int64_t> r(n, 0), s(n, -1), f(n, -1);
  std::vector<Transfer> X;

  // Event: (time, class, id).  Class 0 = an operator completes (id >= 0) or
  // an accelerator becomes available (id = -1 - d); class 1 = transfer id
  // completes; class 2 = one input of operator id arrives (a local
  // predecessor's output, a transferred one, or the op's own release).
  typedef std::tuple<int64_t, int, int> Ev;
  std::priority_queue<Ev, std::vector<Ev>, std::greater<Ev>> events;
  std::vector<int> arrived(n, 0);
  std::vector<std::set<std::pair<int64_t, int>>> ready_q(D);
  std::vector<int> running(D, -1);
  // the communication graph: pending intents in arbitration order, and the
  // endpoints and links held by the active transfers
  std::set<std::tuple<int64_t, int, int, int>> pending;  // (intent time, p, e, transfer id)
  std::vector<bool> sending(D, false), receiving(D, false);
  std::set<int> links_busy;
  for (int i = 0; i < n; ++i) events.push(Ev(g.release[i], 2, i));
  for (int d = 0; d < D; ++d)
    if (g.avail0[d] > 0) events.push(Ev(g.avail0[d], 0, -1 - d));

  auto at_now = [&](int64_t now, int cls) {
    return !events.empty() && std::get<0>(events.top()) == now && std::get<1>(events.top()) == cls;
  };
  while (!events.empty()) {
    const int64_t now = std::get<0>(events.top());
    while (at_now(now, 0) || at_now(now, 1)) {
      bool trigger = false;
      // (i) operator completions: local successors get their input now; one
      // intent per distinct remote accelerator of a successor.
      while (at_now(now, 0)) {
        const int id = std::get<2>(events.top());
        events.pop();
        if (id < 0) continue;
        running[dev[id]] = -1;
        std::set<int> remote;
        for (int j : g.succ[id]) {
          if (dev[j] == dev[id]) events.push(Ev(now, 2, j));
          else remote.insert(dev[j]);
        }
        for (int e : remote) {
          X.push_back({id, e, now, -1, -1});
          pending.insert(std::make_tuple(now, id, e, int(X.size()) - 1));
          trigger = true;
        }
      }
      // (ii) transfer completions: release the endpoints and the link; the
      // successors on the destination get their input now.
      while (at_now(now, 1)) {
        const int x = std::get<2>(events.top());
        events.pop();
        Transfer& t = X[x];
        t.done = now;
        const int src = dev[t.p];
        sending[src] = false;
        receiving[t.e] = false;
        links_busy.erase(g.link[size_t(src) * D + t.e]);
        for (int j : g.succ[t.p])
          if (dev[j] == t.e) events.push(Ev(now, 2, j));
        trigger = true;
      }
      // (iii) arbitration: start every pending intent, in order, whose
      // endpoints and link are free.
      if (trigger) {
        for (auto it = pending.begin(); it != pending.end();) {
          const int x = std::get<3>(*it);
          Transfer& t = X[x];
          const int src = dev[t.p];
          const int lk = g.link[size_t(src) * D + t.e];
          if (sending[src] || receiving[t.e] || links_busy.count(lk)) {
            ++it;
            continue;
          }
          sending[src] = true;
          receiving[t.e] = true;
          links_busy.insert(lk);
          t.start = now;
          events.push(Ev(now + xfer(g, src, t.e, g.bytes[t.p]), 1, x));
          it = pending.erase(it);
        }
      }
    }
    // (iv) input arrivals: an op whose inputs are all present is ready.
    while (at_now(now, 2)) {
      const int j = std::get<2>(events.top());
      events.pop();
      arrived[j] += 1;
      r[j] = now;
      if (arrived[j] == int(g.pred[j].size()) + 1) ready_q[dev[j]].insert({r[j], j});
    }
    // (v) every idle queue starts its ready op with the earliest ready time.
    for (int d = 0; d < D; ++d) {
      if (running[d] >= 0 || g.avail0[d] > now || ready_q[d].empty()) continue;
      const int i = ready_q[d].begin()->second;
      ready_q[d].erase(ready_q[d].begin());
      running[d] = i;
      s[i] = now;
      f[i] = now + dur_on(g, i, d);
      events.push(Ev(f[i], 0, i));
    }
  }

  std::vector<std::vector<Copy>> copies(n);
  for (const Transfer& t : X) copies[t.p].push_back({t.e, t.start, t.done});
  std::sort(X.begin(), X.end(), [](const Transfer& a, const Transfer& b) {
    return std::tie(a.intent, a.p, a.e) < std::tie(b.intent, b.p, b.e);
  });
  settle(g, dev, r, s, f, copies, res);
  res.xfers = std::move(X);
}

// Sec. 3.3.3: event-driven simulation of one placement.
void simulate(const Graph& g, const uint8_t* dev, Result& res) {
  const int n = g.n, D = g.D;
  for (int i = 0; i < n; ++i)
    if (dev[i] >= D) {
      fill_invalid(g, kSimBadDev, res);
      return;
    }
  if (g.mode == 1) {
    simulate_arb(g, dev, res);
    return;
  }
  std::vector<int64_t> r(n, 0), s(n, -1), f(n, -1);

  // Event: (time, class, id).  Class 0 = an operator completes (id >= 0) or
  // an accelerator becomes available (id = -1 - d); class 1 = one input of
  // operator id arrives (a predecessor's output, or the op's own release).
  typedef std::tuple<int64_t, int, int> Ev;
  std::priority_queue<Ev, std::vector<Ev>, std::greater<Ev>> events;
  std::vector<int> arrived(n, 0);
  std::vector<std::set<std::pair<int64_t, int>>> ready_q(D);  // (ready time, op)
  std::vector<int> running(D, -1);
  for (int i = 0; i < n; ++i) events.push(Ev(g.release[i], 1, i));
  for (int d = 0; d < D; ++d)
    if (g.avail0[d] > 0) events.push(Ev(g.avail0[d], 0, -1 - d));

  while (!events.empty()) {
    const int64_t now = std::get<0>(events.top());
    // (i) completions at `now`: free the queue, send outputs to successors.
    while (!events.empty() && std::get<0>(events.top()) == now && std::get<1>(events.top()) == 0) {
      int id = std::get<2>(events.top());
      events.pop();
      if (id < 0) continue;  // accelerator becomes available
      running[dev[id]] = -1;
      for (int j : g.succ[id]) events.push(Ev(now + xfer(g, dev[id], dev[j], g.bytes[id]), 1, j));
    }
    // (ii) input arrivals at `now`: an op whose inputs are all present is
    // ready, with ready time = its last arrival.
    while (!events.empty() && std::get<0>(events.top()) == now && std::get<1>(events.top()) == 1) {
      int j = std::get<2>(events.top());
      events.pop();
      arrived[j] += 1;
      r[j] = now;
      if (arrived[j] == int(g.pred[j].size()) + 1) ready_q[dev[j]].insert({r[j], j});
    }
    // (iii) every idle queue starts its ready op with the earliest ready time.
    for (int d = 0; d < D; ++d) {
      if (running[d] >= 0 || g.avail0[d] > now || ready_q[d].empty()) continue;
      int i = ready_q[d].begin()->second;
      ready_q[d].erase(ready_q[d].begin());
      running[d] = i;
      s[i] = now;
      f[i] = now + dur_on(g, i, d);
      events.push(Ev(f[i], 0, i));
    }
  }

  // Transfers are pure latency: every remote copy is allocated when the
  // producer completes and arrives one transfer estimate later.
  std::vector<std::vector<Copy>> copies(n);
  for (int i = 0; i < n; ++i) {
    std::map<int, int64_t> arrival;  // remote accelerator -> arrival time
    for (int j : g.succ[i])
      if (dev[j] != dev[i]) arrival[dev[j]] = f[i] + xfer(g, dev[i], dev[j], g.bytes[i]);
    for (auto& kv : arrival) copies[i].push_back({kv.first, f[i], kv.second});
  }
  settle(g, dev, r, s, f, copies, res);
}

void write_out(const Graph& g, const Result& res, int64_t k, orc_summary* out, int64_t* peak,
               int64_t* req_done) {
  out[k] = res.s;
  if (peak) std::memcpy(peak + k * g.D, res.peak.data(), sizeof(int64_t) * g.D);
  if (req_done && g.R) std::memcpy(req_done + k * g.R, res.req_done.data(), sizeof(int64_t) * g.R);
}

template <class F>
void parallel_for(int32_t K, int32_t nthreads, F fn) {
  if (nthreads <= 1 || K <= 1) {
    for (int32_t k = 0; k < K; ++k) fn(k);
    return;
  }
  nthreads = std::min<int32_t>(nthreads, K);
  std::vector<std::thread> th;
  for (int32_t t = 0; t < nthreads; ++t) {
    int32_t a = int32_t(int64_t(K) * t / nthreads), b = int32_t(int64_t(K) * (t + 1) / nthreads);
    th.emplace_back([=]() {
      for (int32_t k = a; k < b; ++k) fn(k);
    });
  }
  for (auto& x : th) x.join();
}

}  // namespace

extern "C" {

int orc_check(const orc_graph* in) {
  Graph g;
  return build(in, g);
}

int32_t orc_hw_threads(void) {
  unsigned t = std::thread::hardware_concurrency();
  return t ? int32_t(t) : 1;
}

// One candidate; ready/start/finish (n_ops each) and req_done (n_req) may be NULL.
int orc_simulate(const orc_graph* in, const uint8_t* place, orc_summary* out, int64_t* peak,
                 int64_t* req_done, int64_t* ready, int64_t* start, int64_t* finish) {
  Graph g;
  int rc = build(in, g);
  if (rc) return rc;
  Result res;
  simulate(g, place, res);
  write_out(g, res, 0, out, peak, req_done);
  if (ready) std::memcpy(ready, res.ready.data(), sizeof(int64_t) * g.n);
  if (start) std::memcpy(start, res.start.data(), sizeof(int64_t) * g.n);
  if (finish) std::memcpy(finish, res.finish.data(), sizeof(int64_t) * g.n);
  return 0;
}

// Arbitrated mode: the transfers of one candidate in arbitration order, as
// rows (producer, destination, intent time, start, completion); returns
// their number (rows beyond `cap` are not written) or a negative error.
int64_t orc_transfers(const orc_graph* in, const uint8_t* place, int64_t* rows, int64_t cap) {
  Graph g;
  int rc = build(in, g);
  if (rc) return rc;
  if (g.mode != 1) return kEInval;
  Result res;
  simulate(g, place, res);
  const int64_t m = int64_t(res.xfers.size());
  for (int64_t x = 0; x < std::min(m, cap); ++x) {
    const Transfer& t = res.xfers[x];
    const int64_t v[5] = {t.p, t.e, t.intent, t.start, t.done};
    std::memcpy(rows + 5 * x, v, sizeof(v));
  }
  return m;
}

// K candidates, row k of `place` at place + k*ld (Algorithm 1: each
// candidate partition is simulated independently).
int orc_simulate_batch(const orc_graph* in, const uint8_t* place, int64_t ld, int32_t K,
                       int32_t nthreads, orc_summary* out, int64_t* peak, int64_t* req_done) {
  Graph g;
  int rc = build(in, g);
  if (rc) return rc;
  if (K < 0 || ld < g.n) return kEInval;
  parallel_for(K, nthreads, [&](int32_t k) {
    Result res;
    simulate(g, place + int64_t(k) * ld, res);
    write_out(g, res, k, out, peak, req_done);
  });
  return 0;
}

// K candidates given as move lists against a base placement.  With
// arbitrated transfers, `resumed` says what `events` counts: 0 -- the
// candidate's moved placement simulated in full (events = n); 1 -- resumed at
// T0 from the arbitrated base (events = ops whose arbitrated base ready time
// is >= T0, as with pure-latency transfers; every intent, transfer and buffer
// of a moved op's predecessors happens at or after their finish, so nothing
// before T0 changes).
int orc_incremental_batch(const orc_graph* in, const uint8_t* base_place, const int32_t* move_off,
                          const int32_t* move_op, const uint8_t* move_dev, int32_t K,
                          int32_t nthreads, orc_summary* out, int64_t* peak, int64_t* req_done,
                          int32_t resumed) {
  Graph g;
  int rc = build(in, g);
  if (rc) return rc;
  if (K < 0 || move_off[0] != 0) return kEInval;
  for (int32_t k = 0; k < K; ++k)
    if (move_off[k + 1] < move_off[k]) return kEInval;
  Result base;
  simulate(g, base_place, base);
  const bool base_ok = base.s.status == kSimOk;
  parallel_for(K, nthreads, [&](int32_t k) {
    Result res;
    if (!base_ok) {
      fill_invalid(g, kSimBadBase, res);
      write_out(g, res, k, out, peak, req_done);
      return;
    }
    const int32_t a = move_off[k], b = move_off[k + 1];
    bool bad_range = false, dup = false;
    std::set<int32_t> seen;
    for (int32_t m = a; m < b; ++m) {
      if (move_op[m] < 0 || move_op[m] >= g.n || move_dev[m] >= g.D) bad_range = true;
      else if (!seen.insert(move_op[m]).second) dup = true;
    }
    if (bad_range || dup) {
      fill_invalid(g, bad_range ? kSimMoveRange : kSimMoveDup, res);
      write_out(g, res, k, out, peak, req_done);
      return;
    }
    std::vector<uint8_t> place(base_place, base_place + g.n);
    int64_t t0 = kI64Max;
    for (int32_t m = a; m < b; ++m) {
      const int x = move_op[m];
      if (move_dev[m] == base_place[x]) continue;  // a move to its own device is a no-op
      place[x] = move_dev[m];
      int64_t t = g.release[x];
      if (!g.pred[x].empty()) {
        t = kI64Max;
        for (int p : g.pred[x]) t = std::min(t, base.finish[p]);
      }
      t0 = std::min(t0, t);
    }
    simulate(g, place.data(), res);
    int64_t ev = 0;
    if (g.mode == 1 && !resumed) {
      ev = g.n;  // arbitrated transfers: the moved placement is simulated in full
    } else if (t0 != kI64Max) {
      for (int i = 0; i < g.n; ++i) ev += base.ready[i] >= t0 ? 1 : 0;
    }
    res.s.events = ev;
    write_out(g, res, k, out, peak, req_done);
  });
  return 0;
}

// Algorithm 1, BestRecordedCandidateResult: lexicographic argmin over the
// feasible candidates with status OK of score (mode 0) or (sla_miss, score)
// (mode 1); ties go to the lowest index.  Returns -1 if none.
int64_t orc_select_best(const orc_summary* s, int32_t K, int32_t mode, int64_t* best_score) {
  int64_t best = -1, bscore = kI64Max;
  int32_t bmiss = std::numeric_limits<int32_t>::max();
  for (int32_t k = 0; k < K; ++k) {
    if (s[k].status != kSimOk || s[k].viol_flag) continue;
    bool better;
    if (mode == 1)
      better = best < 0 || s[k].sla_miss < bmiss || (s[k].sla_miss == bmiss && s[k].score < bscore);
    else
      better = best < 0 || s[k].score < bscore;
    if (better) {
      best = k;
      bscore = s[k].score;
      bmiss = s[k].sla_miss;
    }
  }
  if (best_score) *best_score = best < 0 ? kI64Max : bscore;
  return best;
}

}  // extern "C"
