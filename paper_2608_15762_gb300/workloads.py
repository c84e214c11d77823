"""Seeded synthetic workloads for what-if placement simulation.

This module only generates inputs: operator DAGs with the shape of a decoder
layer, integer durations and tensor sizes, request releases and deadlines,
accelerator capacities, link tables, candidate placements and move lists.  It
contains none of the simulator's arithmetic and is shared by the CPU oracle's
tests and by the CUDA path, which is the only thing the two sides share.

Workload recipe (stand-in for the paper's production traces and Llama3-8B
graphs, which are not available):

* One scheduling operator per decoder sub-layer (the paper coarsens ATen ops
  into layer-level scheduling units, Sec. 5.1 "Operator granularity").  A layer
  is the 12-op block ``rms1 -> qkv -> rope -> {attn, kvw}``,
  ``attn -> oproj -> add1 <- in``, ``add1 -> rms2 -> gateup -> silu -> down ->
  add2 <- add1``; every request adds ``embed`` first and ``lm_head`` last, so a
  request of L layers has 12L + 2 ops and 14L + 1 edges.
* Durations are integer microseconds; sizes are integer bytes.  Transfer
  links are ``bytes / bandwidth + latency`` in integer units (the transfer
  estimator of Sec. 3.3.1).
* Idle gaps of the incremental workload follow the idle-slice distribution of
  Sec. 2 (p50 2.55 s, p90 10.9 s), clamped to [10 ms, 20 s] as in Fig. 2's
  selection rule.

Five workloads (``make_workload(1..5)``):

1. tiny: 1 request, L=4, D=2, 24 GiB, 50 GB/s + 5 us, K=256 random placements.
2. 8 requests x L=32 (N=3088), D=8, 80 GiB, 400 GB/s + 10 us, lognormal
   durations (median 200 us, sigma 1) clamped to [5, 50000], deadline
   1.5 x critical path, K=4096 random placements.
3. incremental: 32 requests x L=32 (N=12352) on D=16; requests 0-15 are
   online, pinned to device t and split into 4 segments of 8 layers whose
   starts are released after an idle gap; requests 16-31 are offline on
   device t-16.  K=16384 candidates each move 1-16 offline ops to another
   device, preferring a device whose online request is in an idle gap at the
   op's contention-free start estimate.
4. memory-tight: 8 tenants x 64 decode steps x L=32 (N=197632) on D=8 with KV
   tensors growing linearly with the step; the per-device capacity is a stored
   calibration (about 30% of the K=8192 random placements violate it).
5. large: 128 tenants with L in {16, 32, 80}, requests at t=0 plus Poisson
   arrivals (0.5-5 req/s per tenant) in [0, 0.75 s), D=256, deadlines
   1.2-2.0 x critical path, K=65536 candidates: the first half random full
   placements, the second half 1-64 moves against a base placement.
"""
from __future__ import annotations

import json
import os
import dataclasses
from dataclasses import dataclass
from typing import List, Optional, Sequence

import numpy as np

MiB = 1 << 20
GiB = 1 << 30
INT64_MAX = np.iinfo(np.int64).max

# Per-layer op order (topological): indices inside a layer block.
LAYER_OPS = ("rms1", "qkv", "rope", "attn", "kvw", "oproj", "add1", "rms2",
             "gateup", "silu", "down", "add2")
OPS_PER_LAYER = len(LAYER_OPS)
_K = {name: i for i, name in enumerate(LAYER_OPS)}


@dataclass
class GmgDesc:
    """Host-side description of a Global Mapping Graph (all numpy arrays).

    Op ids are topological (every predecessor id is smaller).  ``cons_off`` /
    ``cons_idx`` list, per op, the consumers whose completion releases its
    output; ``None`` means "all successors".
    """
    n_dev: int
    pred_off: np.ndarray
    pred_idx: np.ndarray
    dur: np.ndarray
    out_bytes: np.ndarray
    release: np.ndarray
    req_id: np.ndarray
    scored: np.ndarray
    deadline: np.ndarray
    cap: np.ndarray
    base: np.ndarray
    avail0: np.ndarray
    bw: np.ndarray
    lat: np.ndarray
    cons_off: Optional[np.ndarray] = None
    cons_idx: Optional[np.ndarray] = None
    # heterogeneous accelerators: the type of each accelerator and every op's
    # duration on every type ([N, T]); None = one type, `dur` everywhere
    dev_type: Optional[np.ndarray] = None
    dur_by_type: Optional[np.ndarray] = None
    # arbitrated transfers: the communication link of every ordered accelerator
    # pair ([D*D], row = source, ids in [0, D*D)); transfers over pairs with
    # one id compete for that link.  None = every ordered pair its own link.
    link_id: Optional[np.ndarray] = None

    @property
    def n_types(self) -> int:
        return 0 if self.dur_by_type is None else int(np.asarray(self.dur_by_type).shape[1])

    def dur_on(self, i: int, d: int) -> int:
        """Duration of op i on accelerator d."""
        if self.dur_by_type is None:
            return int(self.dur[i])
        return int(self.dur_by_type[i][int(self.dev_type[d])])

    @property
    def n_ops(self) -> int:
        return int(self.dur.shape[0])

    @property
    def n_edges(self) -> int:
        return int(self.pred_idx.shape[0])

    @property
    def n_req(self) -> int:
        return int(self.deadline.shape[0])

    def normalized(self) -> "GmgDesc":
        """Return a copy with contiguous arrays of the exact dtypes the ABIs take."""
        def c(a, dt):
            return None if a is None else np.ascontiguousarray(a, dtype=dt)
        return GmgDesc(
            n_dev=int(self.n_dev),
            pred_off=c(self.pred_off, np.int32), pred_idx=c(self.pred_idx, np.int32),
            dur=c(self.dur, np.int64), out_bytes=c(self.out_bytes, np.int64),
            release=c(self.release, np.int64), req_id=c(self.req_id, np.int32),
            scored=c(self.scored, np.uint8), deadline=c(self.deadline, np.int64),
            cap=c(self.cap, np.int64), base=c(self.base, np.int64),
            avail0=c(self.avail0, np.int64), bw=c(self.bw, np.int64),
            lat=c(self.lat, np.int64), cons_off=c(self.cons_off, np.int32),
            cons_idx=c(self.cons_idx, np.int32), dev_type=c(self.dev_type, np.uint8),
            dur_by_type=c(self.dur_by_type, np.int64), link_id=c(self.link_id, np.int32))


@dataclass
class Moves:
    """Per-candidate move lists in CSR form: candidate k moves op[off[k]:off[k+1]]."""
    off: np.ndarray   # int32 [K+1]
    op: np.ndarray    # int32 [M]
    dev: np.ndarray   # uint8 [M]

    @property
    def n_cand(self) -> int:
        return int(self.off.shape[0] - 1)

    def subset(self, ks: Sequence[int]) -> "Moves":
        """The move lists of candidates ks, in that order."""
        off = [0]
        ops, devs = [], []
        for k in ks:
            a, b = int(self.off[k]), int(self.off[k + 1])
            ops.append(self.op[a:b])
            devs.append(self.dev[a:b])
            off.append(off[-1] + b - a)
        return Moves(np.array(off, np.int32),
                     np.concatenate(ops).astype(np.int32) if ops else np.zeros(0, np.int32),
                     np.concatenate(devs).astype(np.uint8) if devs else np.zeros(0, np.uint8))


@dataclass
class Workload:
    name: str
    config: int
    desc: GmgDesc
    n_full: int                 # candidates evaluated by full simulation
    place_seed: int             # seed of the counter-based placement rows
    base_place: Optional[np.ndarray] = None   # uint8 [N]
    moves: Optional[Moves] = None             # incremental candidates

    @property
    def ld(self) -> int:
        return placement_ld(self.desc.n_ops)

    def full_rows(self, ks: Sequence[int]) -> np.ndarray:
        """Placement rows of the given full candidates, uint8 [len(ks), ld]."""
        return random_rows(self.place_seed, ks, self.desc.n_ops, self.desc.n_dev)

    def all_full_rows(self) -> np.ndarray:
        return self.full_rows(range(self.n_full))

    def structured_full_rows(self, ks: Sequence[int]) -> np.ndarray:
        """Structured placements (contiguous per-request stages on random
        accelerators) of the given full candidates."""
        return structured_rows(self.place_seed, ks, self.desc.req_id, self.desc.n_dev)


def placement_ld(n_ops: int) -> int:
    """Row pitch of a placement array: n_ops rounded up to 16 bytes."""
    return max(16, (n_ops + 15) // 16 * 16)


def random_rows(seed: int, ks: Sequence[int], n_ops: int, n_dev: int) -> np.ndarray:
    """Uniform i.i.d. device ids; row k is drawn from its own seeded stream so
    any subset of rows can be regenerated independently."""
    ld = placement_ld(n_ops)
    ks = list(ks)
    out = np.zeros((len(ks), ld), dtype=np.uint8)
    for r, k in enumerate(ks):
        g = np.random.default_rng(np.random.SeedSequence([seed, 1000, int(k)]))
        out[r, :n_ops] = g.integers(0, n_dev, size=n_ops, dtype=np.uint8) if n_ops else 0
    return out


def structured_rows(seed: int, ks: Sequence[int], req_id: np.ndarray, n_dev: int,
                    stages=(1, 2, 4, 8)) -> np.ndarray:
    """Placements built like the pre-defined partitions of Sec. 3.4.2: each
    request's ops, in id order, are cut into S contiguous stages of (nearly)
    equal size, S drawn from `stages`, and each stage goes to a uniformly
    drawn accelerator; ops outside any request are placed uniformly.  Row k
    comes from its own seeded stream."""
    req_id = np.asarray(req_id)
    n = req_id.shape[0]
    ld = placement_ld(n)
    tenants = [np.flatnonzero(req_id == r) for r in range(int(req_id.max()) + 1)] if n else []
    loose = np.flatnonzero(req_id < 0)
    ks = list(ks)
    out = np.zeros((len(ks), ld), dtype=np.uint8)
    for r, k in enumerate(ks):
        g = np.random.default_rng(np.random.SeedSequence([seed, 2000, int(k)]))
        for ops in tenants:
            if ops.size == 0:
                continue
            S = int(g.choice(stages))
            for part in np.array_split(ops, min(S, ops.size)):
                out[r, part] = g.integers(0, n_dev)
        if loose.size:
            out[r, loose] = g.integers(0, n_dev, size=loose.size, dtype=np.uint8)
    return out


# ----------------------------------------------------------------------------
# DAG templates
# ----------------------------------------------------------------------------

class _Builder:
    """Accumulates ops with explicit predecessor lists (ids are appended in
    topological order by construction)."""

    def __init__(self):
        self.preds: List[List[int]] = []
        self.kind: List[int] = []      # layer-op index, or -1 embed, -2 lm_head
        self.layer: List[int] = []
        self.step: List[int] = []

    def add(self, preds, kind, layer=-1, step=0) -> int:
        self.preds.append(sorted(preds))
        self.kind.append(kind)
        self.layer.append(layer)
        self.step.append(step)
        return len(self.preds) - 1


def _request_ops(b: _Builder, n_layers: int, step: int = 0, prev_embed_pred=None,
                 prev_kvw=None):
    """Append one embed + n_layers decoder layers + lm_head.  ``prev_kvw`` maps
    layer -> kvw op id of the previous decode step (KV-cache edges)."""
    emb = b.add([] if prev_embed_pred is None else [prev_embed_pred], -1, -1, step)
    x = emb
    kvw_ids = []
    for l in range(n_layers):
        rms1 = b.add([x], _K["rms1"], l, step)
        qkv = b.add([rms1], _K["qkv"], l, step)
        rope = b.add([qkv], _K["rope"], l, step)
        kv_prev = [] if prev_kvw is None else [prev_kvw[l]]
        attn = b.add([rope] + kv_prev, _K["attn"], l, step)
        kvw = b.add([rope] + kv_prev, _K["kvw"], l, step)
        oproj = b.add([attn], _K["oproj"], l, step)
        add1 = b.add([x, oproj], _K["add1"], l, step)
        rms2 = b.add([add1], _K["rms2"], l, step)
        gateup = b.add([rms2], _K["gateup"], l, step)
        silu = b.add([gateup], _K["silu"], l, step)
        down = b.add([silu], _K["down"], l, step)
        add2 = b.add([add1, down], _K["add2"], l, step)
        kvw_ids.append(kvw)
        x = add2
    head = b.add([x], -2, -1, step)
    return emb, head, kvw_ids


@dataclass
class _Template:
    pred_off: np.ndarray
    pred_idx: np.ndarray
    kind: np.ndarray
    layer: np.ndarray
    step: np.ndarray

    @property
    def n(self):
        return int(self.kind.shape[0])


def _finish(b: _Builder) -> _Template:
    lens = np.array([len(p) for p in b.preds], dtype=np.int64)
    off = np.zeros(len(b.preds) + 1, dtype=np.int64)
    np.cumsum(lens, out=off[1:])
    idx = np.fromiter((q for p in b.preds for q in p), dtype=np.int64, count=int(off[-1]))
    return _Template(off, idx, np.array(b.kind, np.int64), np.array(b.layer, np.int64),
                     np.array(b.step, np.int64))


_TEMPLATE_CACHE = {}


def prefill_template(n_layers: int) -> _Template:
    key = ("prefill", n_layers)
    if key not in _TEMPLATE_CACHE:
        b = _Builder()
        _request_ops(b, n_layers)
        _TEMPLATE_CACHE[key] = _finish(b)
    return _TEMPLATE_CACHE[key]


def decode_template(n_layers: int, n_steps: int) -> _Template:
    key = ("decode", n_layers, n_steps)
    if key not in _TEMPLATE_CACHE:
        b = _Builder()
        head, kvw = None, None
        for s in range(n_steps):
            _, head, kvw = _request_ops(b, n_layers, s, head, kvw)
        _TEMPLATE_CACHE[key] = _finish(b)
    return _TEMPLATE_CACHE[key]


def _concat(templates: Sequence[_Template]):
    """Concatenate request templates into one global CSR; returns arrays and
    the op offset of each request."""
    offs = np.zeros(len(templates) + 1, dtype=np.int64)
    offs[1:] = np.cumsum([t.n for t in templates])
    pred_off = [np.zeros(1, np.int64)]
    pred_idx = []
    e0 = 0
    for t, o in zip(templates, offs[:-1]):
        pred_off.append(t.pred_off[1:] + e0)
        pred_idx.append(t.pred_idx + o)
        e0 += t.pred_idx.shape[0]
    return (np.concatenate(pred_off), np.concatenate(pred_idx) if pred_idx else
            np.zeros(0, np.int64), offs)


# ----------------------------------------------------------------------------
# Value distributions
# ----------------------------------------------------------------------------

def _rng(seed: int, stream: int) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([seed, stream]))


def lognormal_durations(g: np.random.Generator, n: int) -> np.ndarray:
    """Median 200 us, sigma 1.0, rounded and clamped to [5, 50000] us."""
    x = np.rint(g.lognormal(mean=np.log(200.0), sigma=1.0, size=n))
    return np.clip(x, 5, 50000).astype(np.int64)


def uniform_bytes(g: np.random.Generator, n: int, lo: int, hi: int) -> np.ndarray:
    return g.integers(lo, hi + 1, size=n, dtype=np.int64)


def uniform_links(n_dev: int, bw_B_per_us: int, lat_us: int):
    bw = np.full(n_dev * n_dev, bw_B_per_us, dtype=np.int64)
    lat = np.full(n_dev * n_dev, lat_us, dtype=np.int64)
    return bw, lat


def contention_free_start(pred_off, pred_idx, dur, release) -> np.ndarray:
    """Earliest start of every op ignoring devices and transfers:
    est_i = max(release_i, max_p est_p + dur_p).  Used only to place deadlines,
    releases and move targets of the synthetic inputs."""
    n = dur.shape[0]
    po = pred_off.tolist()
    pi = pred_idx.tolist()
    d = dur.tolist()
    rel = release.tolist()
    est = [0] * n
    for i in range(n):
        e = rel[i]
        for k in range(po[i], po[i + 1]):
            p = pi[k]
            v = est[p] + d[p]
            if v > e:
                e = v
        est[i] = e
    return np.array(est, dtype=np.int64)


def deadlines_from_critical_path(pred_off, pred_idx, dur, release, req_id, n_req,
                                 arrival, num, den) -> np.ndarray:
    """deadline_r = arrival_r + floor(cp_r * num_r / den), where cp_r is the
    request's contention-free critical path measured from its arrival."""
    est = contention_free_start(pred_off, pred_idx, dur, release)
    fin = est + dur
    cp_end = np.full(n_req, -1, dtype=np.int64)
    np.maximum.at(cp_end, req_id, fin)
    cp = cp_end - arrival
    num = np.broadcast_to(np.asarray(num, dtype=np.int64), (n_req,))
    return arrival + (cp * num) // den


# ----------------------------------------------------------------------------
# The five workloads
# ----------------------------------------------------------------------------

def _desc(n_dev, pred_off, pred_idx, dur, out_bytes, release, req_id, deadline,
          cap, bw, lat) -> GmgDesc:
    n = dur.shape[0]
    return GmgDesc(
        n_dev=n_dev, pred_off=pred_off, pred_idx=pred_idx, dur=dur,
        out_bytes=out_bytes, release=release, req_id=req_id,
        scored=np.ones(n, np.uint8), deadline=deadline,
        cap=np.full(n_dev, cap, np.int64), base=np.zeros(n_dev, np.int64),
        avail0=np.zeros(n_dev, np.int64), bw=bw, lat=lat).normalized()


def config1(seed: int = 1) -> Workload:
    t = prefill_template(4)
    pred_off, pred_idx, _ = _concat([t])
    n = t.n
    g = _rng(seed, 1)
    dur = g.integers(10, 2001, size=n, dtype=np.int64)
    out_bytes = uniform_bytes(g, n, 1 * MiB, 256 * MiB)
    bw, lat = uniform_links(2, 50_000, 5)
    d = _desc(2, pred_off, pred_idx, dur, out_bytes, np.zeros(n, np.int64),
              np.zeros(n, np.int32), np.array([INT64_MAX], np.int64), 24 * GiB, bw, lat)
    return Workload("tiny-prefill-N50-D2-K256", 1, d, n_full=256, place_seed=seed)


def config2(seed: int = 2) -> Workload:
    reqs = [prefill_template(32)] * 8
    pred_off, pred_idx, offs = _concat(reqs)
    n = int(offs[-1])
    g = _rng(seed, 1)
    dur = lognormal_durations(g, n)
    out_bytes = uniform_bytes(g, n, 1 * MiB, 256 * MiB)
    req_id = np.repeat(np.arange(8), np.diff(offs)).astype(np.int32)
    release = np.zeros(n, np.int64)
    dl = deadlines_from_critical_path(pred_off, pred_idx, dur, release, req_id, 8,
                                      np.zeros(8, np.int64), 3, 2)
    bw, lat = uniform_links(8, 400_000, 10)
    d = _desc(8, pred_off, pred_idx, dur, out_bytes, release, req_id, dl, 80 * GiB, bw, lat)
    return Workload("prefill-8x32L-N3088-D8-K4096", 2, d, n_full=4096, place_seed=seed)


def _gap_samples(g: np.random.Generator, n: int) -> np.ndarray:
    """Idle-slice lengths: lognormal with median 2.55 s and p90 10.9 s
    (sigma = ln(10.9/2.55)/z_0.9), clamped to [10 ms, 20 s]; in microseconds."""
    z90 = 1.2815515655446004
    sigma = np.log(10.9 / 2.55) / z90
    x = np.rint(g.lognormal(mean=np.log(2.55e6), sigma=sigma, size=n))
    return np.clip(x, 1e4, 2e7).astype(np.int64)


def config3(seed: int = 3, n_cand: int = 16384) -> Workload:
    L, T, D = 32, 32, 16
    t = prefill_template(L)
    pred_off, pred_idx, offs = _concat([t] * T)
    n = int(offs[-1])
    g = _rng(seed, 1)
    dur = lognormal_durations(g, n)
    out_bytes = uniform_bytes(g, n, 1 * MiB, 256 * MiB)
    req_id = np.repeat(np.arange(T), np.diff(offs)).astype(np.int32)
    release = np.zeros(n, np.int64)
    gaps = _gap_samples(_rng(seed, 2), 16 * 3).reshape(16, 3)
    # Online requests 0..15: segment j (layers 8j..8j+7) starts when its first
    # rms1 is released, an idle gap after the previous segment's
    # contention-free finish.
    seg_first = []   # [u][j] op id of rms1 of layer 8j
    seg_last = []    # [u][j] op id of add2 of layer 8j+7
    for u in range(16):
        o = int(offs[u])
        seg_first.append([o + 1 + 12 * (8 * j) + _K["rms1"] for j in range(4)])
        seg_last.append([o + 1 + 12 * (8 * j + 7) + _K["add2"] for j in range(4)])
    windows = [[] for _ in range(16)]   # idle windows of online request u's device
    for j in range(1, 4):
        est = contention_free_start(pred_off, pred_idx, dur, release)
        for u in range(16):
            fin = int(est[seg_last[u][j - 1]] + dur[seg_last[u][j - 1]])
            release[seg_first[u][j]] = fin + int(gaps[u, j - 1])
            windows[u].append((fin, fin + int(gaps[u, j - 1])))
    est = contention_free_start(pred_off, pred_idx, dur, release)
    for u in range(16):
        last = int(offs[u + 1]) - 1
        windows[u].append((int(est[last] + dur[last]), INT64_MAX))
    dl = deadlines_from_critical_path(pred_off, pred_idx, dur, release, req_id, T,
                                      np.zeros(T, np.int64), 3, 2)
    bw, lat = uniform_links(D, 400_000, 10)
    d = _desc(D, pred_off, pred_idx, dur, out_bytes, release, req_id, dl, 80 * GiB, bw, lat)
    base = np.empty(n, np.uint8)
    for r in range(T):
        base[offs[r]:offs[r + 1]] = r if r < 16 else r - 16
    # Idle mask of every offline op: devices whose online request is inside an
    # idle window at the op's contention-free start.
    off_ops = np.arange(int(offs[16]), n)
    t_op = est[off_ops]
    idle = np.zeros((off_ops.shape[0], 16), dtype=bool)
    for u in range(16):
        for (a, b_) in windows[u]:
            idle[:, u] |= (t_op >= a) & (t_op < b_)
    mo_off = np.zeros(n_cand + 1, np.int32)
    mo_op, mo_dev = [], []
    for k in range(n_cand):
        gk = np.random.default_rng(np.random.SeedSequence([seed, 3000, k]))
        m = int(gk.integers(1, 17))
        sel = gk.choice(off_ops.shape[0], size=m, replace=False)
        for s in sel:
            op = int(off_ops[s])
            cur = int(base[op])
            cand = [u for u in range(16) if idle[s, u] and u != cur]
            if not cand:
                cand = [u for u in range(16) if u != cur]
            mo_op.append(op)
            mo_dev.append(cand[int(gk.integers(0, len(cand)))])
        mo_off[k + 1] = len(mo_op)
    moves = Moves(mo_off, np.array(mo_op, np.int32), np.array(mo_dev, np.uint8))
    return Workload("incremental-32x32L-N12352-D16-K16384", 3, d, n_full=0,
                    place_seed=seed, base_place=base, moves=moves)


def _caps_file():
    return os.path.join(os.path.dirname(os.path.abspath(__file__)), "workload_caps.json")


def stored_cap(config: int) -> Optional[int]:
    """Per-device capacity calibrated by the oracle's calibration script
    (``oracle/calibrate_caps.py``) so that about 30% of the random placements
    of the memory-tight workload violate it; ``None`` if not calibrated."""
    p = _caps_file()
    if not os.path.exists(p):
        return None
    with open(p) as f:
        v = json.load(f).get(str(config))
    return None if v is None else int(v["cap_bytes"])


def config4(seed: int = 4, cap: Optional[int] = None, n_cand: int = 8192) -> Workload:
    L, S, T, D = 32, 64, 8, 8
    t = decode_template(L, S)
    pred_off, pred_idx, offs = _concat([t] * T)
    n = int(offs[-1])
    g = _rng(seed, 1)
    dur = lognormal_durations(g, n)
    out_bytes = uniform_bytes(g, n, 1 * MiB, 16 * MiB)
    kv0 = g.integers(1, 5, size=T, dtype=np.int64) * MiB
    kind = np.tile(t.kind, T)
    step = np.tile(t.step, T)
    tenant = np.repeat(np.arange(T), np.diff(offs))
    is_kv = kind == _K["kvw"]
    out_bytes[is_kv] = kv0[tenant[is_kv]] * (step[is_kv] + 1)
    req_id = tenant.astype(np.int32)
    release = np.zeros(n, np.int64)
    dl = deadlines_from_critical_path(pred_off, pred_idx, dur, release, req_id, T,
                                      np.zeros(T, np.int64), 3, 2)
    if cap is None:
        cap = stored_cap(4)
    if cap is None:
        cap = INT64_MAX
    bw, lat = uniform_links(D, 400_000, 10)
    d = _desc(D, pred_off, pred_idx, dur, out_bytes, release, req_id, dl, cap, bw, lat)
    return Workload("decode-memtight-8x64x32L-N197632-D8-K8192", 4, d, n_full=n_cand,
                    place_seed=seed)


def config5(seed: int = 5, n_cand: int = 65536) -> Workload:
    T, D = 128, 256
    Ls = (16, 32, 80)
    g = _rng(seed, 1)
    lam = g.uniform(0.5, 5.0, size=T)
    req_tenant, req_arrival, templates = [], [], []
    for t_ in range(T):
        arr = [0]
        tt = 0.0
        while True:
            tt += g.exponential(1.0 / lam[t_])
            if tt >= 0.75:
                break
            arr.append(int(tt * 1e6))
        for a in arr:
            req_tenant.append(t_)
            req_arrival.append(a)
            templates.append(prefill_template(Ls[t_ % 3]))
    R = len(templates)
    pred_off, pred_idx, offs = _concat(templates)
    n = int(offs[-1])
    dur = lognormal_durations(g, n)
    out_bytes = uniform_bytes(g, n, 1 * MiB, 256 * MiB)
    req_id = np.repeat(np.arange(R), np.diff(offs)).astype(np.int32)
    release = np.zeros(n, np.int64)
    arrival = np.array(req_arrival, np.int64)
    release[offs[:-1]] = arrival                     # the embed op of each request
    num = g.integers(12, 21, size=R, dtype=np.int64)
    dl = deadlines_from_critical_path(pred_off, pred_idx, dur, release, req_id, R,
                                      arrival, num, 10)
    bw, lat = uniform_links(D, 400_000, 10)
    d = _desc(D, pred_off, pred_idx, dur, out_bytes, release, req_id, dl, 80 * GiB, bw, lat)
    # Base placement: first half of a request's layers on device 2t, second
    # half (and lm_head) on device 2t+1.
    base = np.empty(n, np.uint8)
    for r in range(R):
        t_ = req_tenant[r]
        L = Ls[t_ % 3]
        o = int(offs[r])
        half = o + 1 + 12 * (L // 2)
        base[o:half] = 2 * t_
        base[half:int(offs[r + 1])] = 2 * t_ + 1
    n_full = n_cand // 2
    n_inc = n_cand - n_full
    mo_off = np.zeros(n_inc + 1, np.int32)
    mo_op, mo_dev = [], []
    for k in range(n_inc):
        gk = np.random.default_rng(np.random.SeedSequence([seed, 3000, k]))
        m = int(gk.integers(1, 65))
        ops = gk.choice(n, size=m, replace=False)
        r = gk.integers(0, D - 1, size=m)
        cur = base[ops].astype(np.int64)
        dev = np.where(r < cur, r, r + 1)
        mo_op.append(ops.astype(np.int32))
        mo_dev.append(dev.astype(np.uint8))
        mo_off[k + 1] = mo_off[k] + m
    moves = Moves(mo_off, np.concatenate(mo_op), np.concatenate(mo_dev))
    return Workload(f"large-128t-N{n}-D256-K{n_cand}", 5, d, n_full=n_full,
                    place_seed=seed, base_place=base, moves=moves)


def config6(seed: int = 6) -> Workload:
    """The prefill workload on two accelerator types: accelerators 0-3 of
    type 0, 4-7 of type 1, slower by a factor drawn per operator kind (the
    operator estimator is per (accelerator type, template operator),
    Sec. 3.3.1) from U[1.3, 2.5]; deadlines from type-0 critical paths."""
    t = prefill_template(32)
    reqs = [t] * 8
    pred_off, pred_idx, offs = _concat(reqs)
    n = int(offs[-1])
    g = _rng(seed, 1)
    dur = lognormal_durations(g, n)
    out_bytes = uniform_bytes(g, n, 1 * MiB, 256 * MiB)
    kinds = np.tile(t.kind, 8)
    uk = np.unique(kinds)
    factor = dict(zip(uk.tolist(), _rng(seed, 2).uniform(1.3, 2.5, size=uk.shape[0]).tolist()))
    slow = np.maximum(1, np.rint(dur * np.array([factor[k] for k in kinds.tolist()]))).astype(np.int64)
    req_id = np.repeat(np.arange(8), np.diff(offs)).astype(np.int32)
    release = np.zeros(n, np.int64)
    dl = deadlines_from_critical_path(pred_off, pred_idx, dur, release, req_id, 8,
                                      np.zeros(8, np.int64), 3, 2)
    bw, lat = uniform_links(8, 400_000, 10)
    d = _desc(8, pred_off, pred_idx, dur, out_bytes, release, req_id, dl, 80 * GiB, bw, lat)
    d = dataclasses.replace(d, dev_type=np.array([0, 0, 0, 0, 1, 1, 1, 1], np.uint8),
                            dur_by_type=np.stack([dur, slow], axis=1)).normalized()
    return Workload("hetero-prefill-8x32L-N3088-D8-T2-K4096", 6, d, n_full=4096, place_seed=seed)


def make_workload(config: int, **kw) -> Workload:
    return {1: config1, 2: config2, 3: config3, 4: config4, 5: config5, 6: config6}[config](**kw)


# ----------------------------------------------------------------------------
# Small random DAGs for parity and property tests
# ----------------------------------------------------------------------------

def random_desc(seed: int, n_ops: int, n_dev: int, n_req: int = 2, max_pred: int = 3,
                edge_p: float = 0.3, dur_hi: int = 50, bytes_hi: int = 1 << 12,
                cap=None, explicit_cons: bool = False, with_release: bool = True,
                with_avail0: bool = True, link_hetero: bool = True,
                deadline: bool = True, n_types: int = 0, window: int = 12) -> GmgDesc:
    """A random topologically numbered DAG with small integer values (with
    n_types >= 2: accelerator types and per-type durations, drawn from a
    stream of their own so the other fields match the one-type graph).
    Predecessors are drawn among the previous ``window`` ops: a wide window
    gives many ops that are ready at once."""
    g = _rng(seed, 77)
    preds = []
    for i in range(n_ops):
        cand = np.arange(max(0, i - window), i)
        if cand.size and g.random() < 0.9:
            k = int(g.integers(0, min(max_pred, cand.size) + 1))
            p = sorted(g.choice(cand, size=k, replace=False).tolist()) if k else []
        else:
            p = []
        if cand.size and g.random() < edge_p and not p:
            p = [int(g.choice(cand))]
        preds.append(p)
    pred_off = np.zeros(n_ops + 1, np.int64)
    pred_off[1:] = np.cumsum([len(p) for p in preds])
    pred_idx = np.array([q for p in preds for q in p], np.int64)
    dur = g.integers(1, dur_hi + 1, size=n_ops, dtype=np.int64)
    out_bytes = g.integers(0, bytes_hi + 1, size=n_ops, dtype=np.int64)
    release = (g.integers(0, 3 * dur_hi, size=n_ops, dtype=np.int64) *
               (g.random(n_ops) < 0.3)) if with_release else np.zeros(n_ops, np.int64)
    req_id = g.integers(-1, n_req, size=n_ops).astype(np.int32) if n_req else \
        np.full(n_ops, -1, np.int32)
    scored = (g.random(n_ops) < 0.8).astype(np.uint8)
    dl = (g.integers(0, 8 * dur_hi, size=n_req, dtype=np.int64) if deadline
          else np.full(n_req, INT64_MAX, np.int64))
    if cap is None:
        capv = g.integers(2 * bytes_hi, 8 * bytes_hi, size=n_dev, dtype=np.int64)
    else:
        capv = np.full(n_dev, cap, np.int64)
    base = np.minimum(g.integers(0, bytes_hi, size=n_dev, dtype=np.int64), capv)
    avail0 = (g.integers(0, 2 * dur_hi, size=n_dev, dtype=np.int64) if with_avail0
              else np.zeros(n_dev, np.int64))
    if link_hetero:
        bw = g.integers(1, 400, size=n_dev * n_dev, dtype=np.int64)
        lat = g.integers(0, 20, size=n_dev * n_dev, dtype=np.int64)
    else:
        bw, lat = uniform_links(n_dev, int(g.integers(1, 400)), int(g.integers(0, 20)))
    cons_off = cons_idx = None
    if explicit_cons:
        succ = [[] for _ in range(n_ops)]
        for i, p in enumerate(preds):
            for q in p:
                succ[q].append(i)
        co = [0]
        ci = []
        for i in range(n_ops):
            s = succ[i]
            keep = [c for c in s if g.random() < 0.7]
            ci.extend(keep)
            co.append(len(ci))
        cons_off = np.array(co, np.int64)
        cons_idx = np.array(ci, np.int64)
    dev_type = dur_by_type = None
    if n_types >= 2:
        gt = _rng(seed, 78)
        dev_type = gt.integers(0, n_types, size=n_dev).astype(np.uint8)
        dur_by_type = gt.integers(1, dur_hi + 1, size=(n_ops, n_types), dtype=np.int64)
    return GmgDesc(n_dev=n_dev, pred_off=pred_off, pred_idx=pred_idx, dur=dur,
                   out_bytes=out_bytes, release=release, req_id=req_id, scored=scored,
                   deadline=dl, cap=capv, base=base, avail0=avail0, bw=bw, lat=lat,
                   cons_off=cons_off, cons_idx=cons_idx, dev_type=dev_type,
                   dur_by_type=dur_by_type).normalized()


def random_moves(seed: int, n_cand: int, base: np.ndarray, n_dev: int, max_moves: int,
                 allow_noop: bool = True) -> Moves:
    """Random move lists with distinct ops per candidate (some may target the
    op's own base device, which is a no-op)."""
    n = base.shape[0]
    off = np.zeros(n_cand + 1, np.int32)
    ops, devs = [], []
    for k in range(n_cand):
        g = np.random.default_rng(np.random.SeedSequence([seed, 4000, k]))
        m = int(g.integers(0, min(max_moves, n) + 1)) if n else 0
        sel = g.choice(n, size=m, replace=False) if m else np.zeros(0, np.int64)
        for op in sel:
            if allow_noop and g.random() < 0.15:
                d = int(base[op])
            else:
                d = int(g.integers(0, n_dev))
            ops.append(int(op))
            devs.append(d)
        off[k + 1] = len(ops)
    return Moves(off, np.array(ops, np.int32), np.array(devs, np.uint8))
