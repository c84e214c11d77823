#!/usr/bin/env python
"""Benchmark: candidate placements simulated per second on one GB300.

Default workload: the large workload -- 128 tenants with 16/32/80-layer
decoder graphs and Poisson request arrivals (N=213,568 ops) on 256 simulated
accelerators, K=65,536 candidates: 32,768 uniform random full placements and
32,768 incremental candidates of 1-64 moves against a base placement.  One
step = base_create + sim_incremental over the move lists (side stream)
concurrently with sim_batch over the full placements (current stream), then
select_best over both halves; inputs resident in HBM, L2 flushed (256 MiB
write) between steps; every step and every kernel timed with CUDA events on
the stream it runs on.

Also reported: the end-to-end rate through the public API with host buffers
(H2D of the placements, base row and move lists from pinned memory and D2H
of the selection inside the timed region), the dominant kernel's roofline
and every kernel's issue fraction, the CPU oracle timed on this host's cores
on a sample of each half (scaled to the whole mix), and the SM clocks sampled
during the timed region.

``--impl reference`` times the CPU oracle (the reference arm of this repo:
there is no upstream implementation) on the same workload and metric.
``--config 1..6`` selects another workload, ``--arbitrated`` the arbitrated
transfers of Sec. 3.5.2, ``--placements structured`` contiguous per-request
stages instead of uniform placements, ``--rounds`` / ``--estimators`` the
scheduling round and the estimator refits (supplementary lines).
Under torchrun the workload's candidates are partitioned: every rank takes a
contiguous block of each half (strong scaling, no data-path collective; the
graph and the base row are replicated); rank 0 prints the line with the max
time, each candidate counted once.
"""
import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "candidate placements simulated/sec (and op-events/sec) vs HBM/issue roofline"
UNIT = "candidates/s"
PROFILE_DIR = os.path.join(ROOT, "profiles")
KERNEL_SOURCES = [os.path.join(ROOT, "paper_2608_15762_gb300", "csrc", f)
                  for f in ("gmgsim_sim.cuh", "gmgsim_full.cu", "gmgsim_inc.cu", "gmgsim_kernels.cu",
                            "gmg_layout.h")]


def _code_only(text: str) -> str:
    """The source without comments or blank lines: a profile stays valid
    across comment edits, which cannot change the compiled kernel."""
    import re
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    lines = []
    for ln in text.splitlines():
        # drop // comments that are not inside string literals
        out, in_str = [], False
        i = 0
        while i < len(ln):
            c = ln[i]
            if c == '"' and (i == 0 or ln[i - 1] != "\\"):
                in_str = not in_str
            if not in_str and ln.startswith("//", i):
                break
            out.append(c)
            i += 1
        s = "".join(out).rstrip()
        if s:
            lines.append(s)
    return "\n".join(lines)


def kernel_hash(extra=()) -> str:
    h = hashlib.sha256()
    for f in list(KERNEL_SOURCES) + [os.path.join(ROOT, "paper_2608_15762_gb300", "csrc", e) for e in extra]:
        with open(f, encoding="utf-8") as fh:
            h.update(_code_only(fh.read()).encode())
    return h.hexdigest()[:16]


def profile_path(kernel: str, workload: str) -> str:
    return os.path.join(PROFILE_DIR, "%s_%s.txt" % (kernel, workload))


def read_profile(path: str, extra=()):
    """Instruction and DRAM counts per candidate of the dominant kernel from
    the committed ncu summary of that kernel on this workload (captured on
    `candidates_per_launch` candidates), if it was taken on the current kernel
    source."""
    if not os.path.exists(path):
        return None
    vals = {}
    with open(path) as f:
        for line in f:
            if ":" in line:
                k, v = line.split(":", 1)
                vals[k.strip()] = v.strip()
    if vals.get("kernel_source_sha256") != kernel_hash(extra):
        return None
    try:
        c = float(vals["candidates_per_launch"])
        return {"inst_per_cand": float(vals["inst_executed_per_launch"]) / c,
                "dram_per_cand": float(vals["dram_bytes_per_launch"]) / c, "captured": int(c)}
    except (KeyError, ValueError, ZeroDivisionError):
        return None


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "sm_max_mhz": d.get("sm_max_mhz", 2070.0), "src": "measured"}
    return {"hbm_gbs": 6800.0, "sm_max_mhz": 2070.0, "src": "fallback"}


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.Q, "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------
# Workload preparation
# ---------------------------------------------------------------------------

class Prepared:
    pass


ARB_SOURCES = ("gmgsim_arb.cu", "gmg_arb.h", "gmg_arb_events.h")
ARBW_SOURCES = ("gmgsim_arbw.cu", "gmg_arbw.h", "gmg_arb_events.h")


def rows_of(wl, ks, structured=False):
    """Full placement rows of candidates ks: uniform i.i.d. device ids, or the
    structured variant (contiguous per-request stages on random accelerators)."""
    return wl.structured_full_rows(ks) if structured else wl.full_rows(ks)


def prepare(config: int, rank: int, world: int, device, cap=None, arbitrated=False, structured=False,
            staging="default"):
    """Inputs of one rank, resident on its device: its contiguous block of
    the full placements and of the incremental move lists (the base row and
    the graph are replicated), outputs, two scratch buffers (the two halves
    run on two streams) and the side stream."""
    import numpy as np
    import torch
    from paper_2608_15762_gb300 import gmgsim as G
    from paper_2608_15762_gb300 import workloads as W
    wl = W.make_workload(config)
    p = Prepared()
    p.wl = wl
    p.arb = arbitrated
    # on up to 32 accelerators the arbitrated base snapshot keeps the
    # arbiter's checkpoints and candidates resume from it; on more, every
    # moved placement is simulated in full
    p.arb_base = arbitrated and wl.desc.n_dev <= 32
    p.structured = structured
    p.staging = {"default": G.GMG_STAGING_DEFAULT, "shared": G.GMG_STAGING_SHARED, "l1": G.GMG_STAGING_L1}[staging]
    if arbitrated and wl.desc.n_dev > 256:
        raise SystemExit("--arbitrated needs at most 256 accelerators")
    if structured and (wl.n_full == 0 or wl.moves is not None):
        raise SystemExit("--placements structured needs a workload of full placements only")
    p.g = G.gmg_create(wl.desc, device=device)
    n_full = wl.n_full
    n_inc = 0 if wl.moves is None else wl.moves.n_cand
    if cap is not None:
        # profiling captures: the first `cap` candidates of each half
        n_full, n_inc = min(n_full, cap), min(n_inc, cap)
    p.n_full_total, p.n_inc_total = n_full, n_inc
    p.full_ks = G.shard_block(rank, world, n_full)
    p.inc_ks = G.shard_block(rank, world, n_inc)
    p.n_full, p.n_inc = len(p.full_ks), len(p.inc_ks)
    p.K = p.n_full + p.n_inc
    p.to_global = G.two_half_index(p.n_full, p.full_ks.start, n_full, p.inc_ks.start)
    p.host_place = None
    if p.n_full:
        rows = rows_of(wl, p.full_ks, structured)
        p.host_place = torch.from_numpy(rows).pin_memory()
        p.place = p.host_place.to(device)
    if p.n_inc:
        moves = wl.moves.subset(p.inc_ks)
        p.host_base = torch.from_numpy(np.ascontiguousarray(wl.base_place)).pin_memory()
        p.base_place = p.host_base.to(device)
        p.host_moves = [torch.from_numpy(np.ascontiguousarray(a)).pin_memory()
                        for a in (moves.off, moves.op, moves.dev)]
        p.moves = [t.to(device) for t in p.host_moves]
    p.out = G.SimOut.empty(max(p.K, 1), wl.desc.n_dev, wl.desc.n_req, device)
    p.scratch = G.Scratch(device)
    p.scratch_inc = G.Scratch(device)
    p.side = torch.cuda.Stream(device)
    p.best = torch.empty(2, dtype=torch.int64, device=device)
    p._base = None
    return p


def _views(out, a, b):
    from paper_2608_15762_gb300 import gmgsim as G
    return G.SimOut(**{k: (None if v is None else v[a:b]) for k, v in out.__dict__.items()})


def run_step(p, ev=None):
    """One pass of the hot path over this rank's batch: the base snapshot and
    the incremental candidates on the side stream, the full placements on the
    current stream (the two run concurrently; the base's single warp is
    launched first so that it is not queued behind the full grid), then the
    selection over both halves.  ``ev``: optional dict of CUDA event pairs
    recorded around each kernel on the stream it runs on.  Returns the
    number of this library's kernel launches."""
    import torch
    from paper_2608_15762_gb300 import gmgsim as G
    launches = 0
    main = torch.cuda.current_stream()
    if p.n_inc:
        p.side.wait_stream(main)
        with torch.cuda.stream(p.side):
            if ev:
                ev["base"][0].record()
            b = G.base_create(p.g, p.base_place, stream=p.side, arbitrated=p.arb_base)
            if ev:
                ev["base"][1].record()
                ev["inc"][0].record()
            G.sim_incremental(p.g, b, *p.moves, out=_views(p.out, p.n_full, p.K), scratch=p.scratch_inc,
                              arbitrated=p.arb, stream=p.side)
            if ev:
                ev["inc"][1].record()
        p._base = b  # keep alive until the stream has used it
        launches += 3 if p.arb and not p.arb_base else 2
    if p.n_full:
        if ev:
            ev["full"][0].record()
        G.sim_batch(p.g, p.place, out=_views(p.out, 0, p.n_full), scratch=p.scratch, arbitrated=p.arb,
                    gmg_staging=p.staging)
        if ev:
            ev["full"][1].record()
        launches += 1
    if p.n_inc:
        main.wait_stream(p.side)
    G.select_best(p.out, p.K, best=p.best)
    launches += 2
    return launches


def run_e2e_step(p):
    """Public API with host buffers: H2D of the inputs, the path, D2H of the
    selection."""
    if p.n_full:
        p.place.copy_(p.host_place, non_blocking=True)
    if p.n_inc:
        p.base_place.copy_(p.host_base, non_blocking=True)
        for d, h in zip(p.moves, p.host_moves):
            d.copy_(h, non_blocking=True)
    run_step(p)
    return p.best.cpu()


def h2d_bytes(p):
    b = 0
    if p.n_full:
        b += p.host_place.numel()
    if p.n_inc:
        b += p.host_base.numel() + sum(t.numel() * t.element_size() for t in p.host_moves)
    return b


def oracle_sample(wl, k_full, k_inc, nthreads, arbitrated=False, structured=False):
    """Callables that run the CPU oracle, as it stands, on the first k_full
    full placements and the first k_inc incremental candidates of the
    workload (either may be 0)."""
    from oracle import oracle as O
    from paper_2608_15762_gb300.workloads import Moves
    runs = []
    if k_full:
        rows = rows_of(wl, range(k_full), structured)
        runs.append(("full", k_full, wl.n_full,
                     lambda nt=nthreads, r=rows: O.simulate_batch(wl.desc, r, nthreads=nt, arbitrated=arbitrated),
                     lambda k1, r=rows: O.simulate_batch(wl.desc, r[:k1], nthreads=1, arbitrated=arbitrated)))
    if k_inc:
        m = wl.moves
        mv = Moves(m.off[:k_inc + 1].copy(), m.op[:m.off[k_inc]], m.dev[:m.off[k_inc]])
        runs.append(("incremental", k_inc, m.n_cand,
                     lambda nt=nthreads, v=mv: O.incremental_batch(wl.desc, wl.base_place, v, nthreads=nt,
                                                                 arbitrated=arbitrated),
                     lambda k1, v=mv: O.incremental_batch(wl.desc, wl.base_place, v.subset(range(k1)),
                                                          nthreads=1, arbitrated=arbitrated)))
    return runs


def cpu_baseline(wl, min_s=10.0, arbitrated=False, structured=False):
    """The CPU oracle as it stands on this host's cores, on a bounded sample
    of each half of the workload, scaled to the workload's whole candidate
    mix: value = K / sum over halves of (candidates of the half x measured
    seconds per candidate).  The sample of a half is sized from a short probe
    pass so that its timed passes take about min_s / (number of halves)
    seconds; whole sample passes repeat until then."""
    from oracle import oracle as O
    nt = O.hw_threads()
    n_inc = 0 if wl.moves is None else wl.moves.n_cand
    halves = [h for h in ((wl.n_full, 0), (0, n_inc)) if h[0] or h[1]]
    per_half = min_s / max(len(halves), 1)
    total_s, total_s1, parts, wall, K, scaled = 0.0, 0.0, [], 0.0, 0, False
    for kf, ki in halves:
        k_all = kf or ki
        if not k_all:
            continue
        K += k_all
        k0 = min(k_all, 2 * nt)
        probe = oracle_sample(wl, k0 if kf else 0, k0 if ki else 0, nt, arbitrated, structured)[0]
        t0 = time.perf_counter()
        probe[3]()
        spc0 = (time.perf_counter() - t0) / k0
        k = int(min(k_all, max(k0, per_half / max(spc0, 1e-9))))
        name, k, _, run, run1 = oracle_sample(wl, k if kf else 0, k if ki else 0, nt, arbitrated, structured)[0]
        scaled = scaled or k < k_all
        reps, t0 = 0, time.perf_counter()
        while True:
            run()
            reps += 1
            dt = time.perf_counter() - t0
            if dt >= per_half:
                break
        wall += dt
        spc = dt / (reps * k)
        # one core: a smaller sample of the same candidates, about 1.5 s of work
        k1 = int(max(1, min(k, 1.5 / (spc * nt))))
        t1 = time.perf_counter()
        run1(k1)
        spc1 = (time.perf_counter() - t1) / k1
        total_s += k_all * spc
        total_s1 += k_all * spc1
        parts.append("%s: %d of %d candidates x %d pass%s, %.4g s/candidate (1 core: first %d, %.4g s)" % (
            name, k, k_all, reps, "" if reps == 1 else "es", spc, k1, spc1))
    return {"value": K / total_s, "unit": UNIT, "cores": nt, "kind": "oracle",
            "sample": "; ".join(parts) + ("; scaled to all %d candidates" % K if scaled else ""),
            "scaled": scaled, "seconds": round(wall, 3),
            "op_events_per_s": wl.n_full * wl.desc.n_ops / total_s if wl.n_full and not n_inc else None,
            "single_core": {"value": K / total_s1, "unit": UNIT, "cores": 1,
                            "sample": "smaller samples of the same candidates, one pass each"}}


def reference_arm(args):
    """--impl reference: time the CPU oracle, as it stands, on the host cores,
    on the same workload, metric and unit.  Each step is a bounded sample of
    the workload with the workload's own mix of full placements and
    incremental candidates (about 3e7 op-events of candidates per step)."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    from oracle import oracle as O
    from paper_2608_15762_gb300 import workloads as W
    wl = W.make_workload(args.config)
    nt = O.hw_threads()
    n_inc = 0 if wl.moves is None else wl.moves.n_cand
    K = wl.n_full + n_inc
    k = min(K, max(16, int(3e7 // max(wl.desc.n_ops, 1))))
    kf = min(wl.n_full, (k * wl.n_full + K - 1) // K)
    ki = min(n_inc, k - kf) if n_inc else 0
    runs = oracle_sample(wl, kf, ki, nt, args.arbitrated, args.placements == "structured")

    def step():
        for r in runs:
            r[3]()
    for _ in range(args.warmup):
        step()
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        step()
        times.append(time.perf_counter() - t0)
    ms = 1000 * statistics.mean(times)
    v = (kf + ki) / (ms / 1000)
    line = {"metric": METRIC, "value": v, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "strong",
            "vs_baseline": None, "dtype": "int64", "data": "synthetic", "impl": "reference",
            "config": {"workload": wl.name, "candidates_per_step": kf + ki, "full_per_step": kf,
                       "incremental_per_step": ki, "n_ops": wl.desc.n_ops,
                       "transfers": "arbitrated" if args.arbitrated else "latency",
                       "placements": args.placements},
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": nt, "kind": "oracle",
                             "sample": "the first %d full placements and %d incremental candidates of the "
                                       "workload per step (its own mix)" % (kf, ki)},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


# ---------------------------------------------------------------------------
# Online estimators (include/gmgest.h): refit + durations + links per step
# ---------------------------------------------------------------------------

EST_METRIC = "estimator feedback samples incorporated/sec (refit of every estimator + durations + links)"


def estimator_workload(seed: int = 7):
    """Executor feedback for the operator estimators (2 accelerator types x 14
    template operators, 5 features, 16,384 samples each) and the transfer
    estimators (8 x 8 accelerator pairs, features (bytes, 1), 4,096 samples
    each), and the ops whose durations are predicted (the decode workload's
    197,632 ops on 2 types)."""
    import numpy as np
    g = np.random.default_rng(seed)
    w = {}
    T, Kk, F, cnt = 2, 14, 5, 16384
    E = T * Kk
    w["op_off"] = (np.arange(E + 1) * cnt).astype(np.int32)
    x = g.uniform(0, 10, (E * cnt, F))
    x[:, -1] = 1.0
    beta = g.uniform(1, 40, (E, F))
    w["op_x"] = x
    w["op_y"] = np.einsum("sf,sf->s", x, np.repeat(beta, cnt, axis=0)) + g.normal(0, 2.0, E * cnt)
    D, ct = 8, 4096
    w["tr_off"] = (np.arange(D * D + 1) * ct).astype(np.int32)
    size = g.uniform(1 << 20, 1 << 28, D * D * ct)
    q = np.repeat(np.arange(D * D), ct)
    inv_bw = 1.0 / g.integers(50_000, 400_000, D * D)
    w["tr_x"] = np.stack([size, np.ones_like(size)], axis=1)
    w["tr_y"] = size * inv_bw[q] + 10 + g.normal(0, 0.5, size.shape[0])
    N = 197_632
    kind = g.integers(0, Kk, N)
    w["est_of"] = np.stack([t * Kk + kind for t in range(T)], axis=1).astype(np.int32)
    xo = g.uniform(0, 10, (N, F))
    xo[:, -1] = 1.0
    w["op_feat"] = xo
    w["dflt"] = g.integers(5, 50_000, N).astype(np.int64)
    w["bw_dflt"] = np.full(D * D, 400_000, np.int64)
    w["lat_dflt"] = np.full(D * D, 10, np.int64)
    w.update(T=T, E=E, F=F, D=D, N=N)
    return w


def run_estimators(args):
    import numpy as np
    import torch
    from paper_2608_15762_gb300 import build as lib_build
    from paper_2608_15762_gb300 import gmgsim as G
    lib_build.build()
    device = torch.device("cuda", 0)
    w = estimator_workload()
    host = {k: torch.from_numpy(np.ascontiguousarray(v)).pin_memory() for k, v in w.items()
            if isinstance(v, np.ndarray)}
    dev = {k: v.to(device) for k, v in host.items()}
    op, tr = G.Estimators(w["E"], w["F"], device), G.Estimators(w["D"] ** 2, 2, device)
    op_tmp, tr_tmp = op.tmp_for(w["op_y"].shape[0]), tr.tmp_for(w["tr_y"].shape[0])
    dur = torch.empty((w["N"], w["T"]), dtype=torch.int64, device=device)

    bw = torch.empty(w["D"] ** 2, dtype=torch.int64, device=device)
    lat = torch.empty_like(bw)
    branch = torch.cuda.Stream(device)

    def step():
        # operator and transfer estimators are independent: two branches
        main = torch.cuda.current_stream()
        branch.wait_stream(main)
        op.update(dev["op_off"], dev["op_x"], dev["op_y"], tmp=op_tmp)
        op.predict_durations(dev["est_of"], dev["op_feat"], dev["dflt"], out=dur)
        with torch.cuda.stream(branch):
            tr.update(dev["tr_off"], dev["tr_x"], dev["tr_y"], tmp=tr_tmp)
            G._check(G.lib().est_links(tr.state.data_ptr(), w["D"], dev["bw_dflt"].data_ptr(),
                                       dev["lat_dflt"].data_ptr(), bw.data_ptr(), lat.data_ptr(),
                                       G._stream_handle(branch)), "est_links")
        main.wait_stream(branch)

    flush = torch.empty(256 << 20, dtype=torch.uint8, device=device)
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()

    def timed(run):
        ev = []
        for _ in range(args.steps):
            flush.fill_(1)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            run()
            b.record()
            ev.append((a, b))
        torch.cuda.synchronize()
        return [a.elapsed_time(b) for a, b in ev]

    # the step's 8 small dependent launches, captured once in a CUDA graph
    graph = torch.cuda.CUDAGraph()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step()
    torch.cuda.current_stream().wait_stream(side)
    with torch.cuda.graph(graph):
        step()
    for _ in range(args.warmup):
        graph.replay()
    torch.cuda.synchronize()
    sampler = ClockSampler(0)
    sampler.start()
    time.sleep(0.3)
    ms_launch = timed(step)
    ms_all = timed(graph.replay)
    clocks = sampler.stop()
    ms = statistics.mean(ms_all)
    samples = w["op_y"].shape[0] + w["tr_y"].shape[0]
    # end to end: the feedback batch and op features copied in, durations out
    t0 = time.perf_counter()
    for _ in range(args.steps):
        for k in ("op_x", "op_y", "tr_x", "tr_y", "op_feat"):
            dev[k].copy_(host[k], non_blocking=True)
        graph.replay()
        out = dur.cpu()
    torch.cuda.synchronize()
    e2e_ms = 1000 * (time.perf_counter() - t0) / args.steps
    in_bytes = sum(host[k].numel() * host[k].element_size() for k in ("op_x", "op_y", "tr_x", "tr_y", "op_feat"))
    alg = (in_bytes + sum(dev[k].numel() * dev[k].element_size() for k in ("op_off", "tr_off", "est_of", "dflt"))
           + dur.numel() * 8)
    pk = peaks()
    line = {"metric": EST_METRIC, "value": samples / (ms / 1000), "unit": "samples/s", "n_gpus": 1,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "ms_per_step_best": min(ms_all),
            "ms_per_step_median": statistics.median(ms_all), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": "estimators-28op-F5x16384-64link-F2x4096-predict-N197632-T2",
                       "l2": "flushed between steps (256 MiB write)"},
            "durations_per_s": w["N"] * w["T"] / (ms / 1000),
            "roofline": {"bound": "hbm", "achieved": alg / (ms / 1000) / 1e9, "peak": pk["hbm_gbs"],
                         "unit": "GB/s", "frac": alg / (ms / 1000) / 1e9 / pk["hbm_gbs"], "traffic": None,
                         "algorithmic_bytes_per_step": alg,
                         "note": "whole step (8 kernels, CUDA-graph replay) timed"},
            "ms_per_step_separate_launches": statistics.mean(ms_launch),
            "e2e": {"value": samples / (e2e_ms / 1000), "unit": "samples/s", "ms_per_step": e2e_ms,
                    "h2d_bytes_per_step": in_bytes, "d2h_bytes_per_step": out.numel() * 8},
            "gpu_launches": 8 * args.steps, "clocks": clocks}
    if not args.no_cpu_baseline:
        from oracle import estimators as OE
        t0 = time.perf_counter()
        o1, o2 = OE.EstimatorsOracle(w["E"], w["F"]), OE.EstimatorsOracle(w["D"] ** 2, 2)
        o1.update(w["op_off"], w["op_x"], w["op_y"])
        o2.update(w["tr_off"], w["tr_x"], w["tr_y"])
        b1, f1 = o1.coefficients()
        b2, f2 = o2.coefficients()
        m = 20_000
        OE.predict_durations(b1, f1, w["est_of"][:m], w["op_feat"][:m], w["dflt"][:m])
        OE.links(b2, f2, w["D"], w["bw_dflt"], w["lat_dflt"])
        dt = time.perf_counter() - t0
        line["cpu_baseline"] = {"value": samples / dt, "unit": "samples/s", "cores": 1, "kind": "oracle",
                                "sample": "one feedback batch (all %d samples), durations of the first %d of %d "
                                          "ops" % (samples, m, w["N"])}
    print(json.dumps(line))
    return 0


# ---------------------------------------------------------------------------
# Scheduling rounds (include/gmground.h)
# ---------------------------------------------------------------------------

ROUND_METRIC = "scheduling rounds/sec (Algorithm 1: frontiers, batch, 14 partition candidates simulated, best committed)"


def round_setup(seed: int = 12):
    """The prefill graph (8 requests x 32 layers): one template, role = op
    position in its request, 14 partitions (8 single accelerators, 4 pairs, 2
    quads) with each request's layers split evenly over a partition's
    accelerators, priority = the request's deadline, budget 128 issued ops,
    batches of at most 64."""
    import numpy as np
    from paper_2608_15762_gb300 import workloads as W
    wl = W.config2()
    d = wl.desc
    per = d.n_ops // 8
    part_off = np.array([0, 1, 2, 3, 4, 5, 6, 7, 8, 10, 12, 14, 16, 20, 24], np.int32)
    part_dev = np.array(list(range(8)) * 3, np.uint8)
    sizes = np.diff(part_off)
    mapping = np.stack([np.arange(per) * sizes[p] // per for p in range(len(sizes))]).astype(np.int32)
    ld = W.placement_ld(d.n_ops)
    place = np.zeros(ld, np.uint8)
    place[:d.n_ops] = np.random.default_rng(seed).integers(0, 8, d.n_ops)
    return dict(desc=d, per=per, part_off=part_off, part_dev=part_dev, mapping=mapping.reshape(-1), place=place,
                prio=np.repeat(d.deadline, per).astype(np.int64), tmpl=np.zeros(d.n_ops, np.int32),
                role=np.tile(np.arange(per), 8).astype(np.int32), budget=128, max_batch=64)


ROUND_PROFILE = os.path.join(PROFILE_DIR, "rounds_prefill-8x32L-N3088-D8-P14-B128-batch64.txt")


def round_roofline(ms):
    """Issue-slot roofline of a round: warp instructions per round (all its
    kernels, from the committed ncu summary, if taken on the current sources)
    over the measured round time."""
    import torch
    pk = peaks()
    props = torch.cuda.get_device_properties(torch.device("cuda", 0))
    peak = props.multi_processor_count * 4 * pk["sm_max_mhz"] * 1e6 / 1e9
    roof = {"bound": "alu", "achieved": None, "peak": peak, "unit": "Ginst/s", "frac": None, "traffic": None,
            "note": "latency-bound: 14 candidates are 14 warps; a round takes one candidate simulation's "
                    "latency plus 8 small launches"}
    vals = {}
    if os.path.exists(ROUND_PROFILE):
        with open(ROUND_PROFILE) as f:
            for line in f:
                if ":" in line and not line.startswith("#"):
                    k, v = line.split(":", 1)
                    vals[k.strip()] = v.strip()
    if vals.get("kernel_source_sha256") == kernel_hash(("gmground.cu",)) and "inst_per_round" in vals:
        ach = float(vals["inst_per_round"]) / (ms / 1000) / 1e9
        roof.update(achieved=ach, frac=ach / peak, inst_src=os.path.relpath(ROUND_PROFILE, ROOT))
    return roof


def run_rounds(args):
    import numpy as np
    import torch
    from paper_2608_15762_gb300 import build as lib_build
    from paper_2608_15762_gb300 import gmgsim as G
    lib_build.build()
    device = torch.device("cuda", 0)
    w = round_setup()
    d = w["desc"]

    def dev(a, dt):
        return torch.from_numpy(np.ascontiguousarray(a, dtype=dt)).to(device)

    g = G.gmg_create(d, device=device)
    state = torch.zeros(d.n_ops, dtype=torch.uint8, device=device)
    place = dev(w["place"], np.uint8)
    rnd = G.Round(g, state, place, dev(w["prio"], np.int64), dev(w["tmpl"], np.int32), dev(w["role"], np.int32),
                  dev(w["part_off"], np.int32), dev(w["part_dev"], np.uint8), dev(w["mapping"], np.int32),
                  w["per"], w["budget"], w["max_batch"])

    def one():
        rnd.step()
        state.masked_fill_(state == 1, 2)   # the executor finishes the issued ops

    def reset():
        state.zero_()
        place.copy_(dev(w["place"], np.uint8))

    # the rounds from an empty schedule until every op is scheduled (counted
    # once with the status read back, then replayed without host reads)
    needed = 0
    while True:
        one()
        needed += 1
        if int(rnd.info[5].item()) != G.ROUND_BATCH or needed > 100000:
            break
    needed -= 1
    for _ in range(args.warmup):
        reset()
        for _ in range(needed):
            one()
    torch.cuda.synchronize()
    sampler = ClockSampler(0)
    sampler.start()
    time.sleep(0.3)
    ev = []
    for _ in range(max(args.steps, 1)):
        reset()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(needed):
            one()
        b.record()
        ev.append((a, b))
    torch.cuda.synchronize()
    ms_all = [a.elapsed_time(b) / needed for a, b in ev]
    clocks = sampler.stop()
    ms = statistics.mean(ms_all)
    rounds = needed * max(args.steps, 1)
    scheduled = int((state != 0).sum().item())
    line = {"metric": ROUND_METRIC, "value": 1000.0 / ms, "unit": "rounds/s", "n_gpus": 1, "steps": rounds,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "int64", "data": "synthetic",
            "config": {"workload": "rounds-prefill-8x32L-N3088-D8-P14-B128-batch64",
                       "rounds_to_schedule_every_op": needed, "ops_scheduled": scheduled},
            "ms_per_step_best": min(ms_all), "ms_per_step_median": statistics.median(ms_all),
            "candidates_per_s": 14 * 1000.0 / ms,
            "roofline": round_roofline(ms),
            "gpu_launches": 9 * rounds, "clocks": clocks}
    if not args.no_cpu_baseline:
        from oracle import round as OR
        st = np.zeros(d.n_ops, np.uint8)
        pl = w["place"].copy()
        t0 = time.perf_counter()
        k = min(needed, 16)
        for _ in range(k):
            _, _, _, _, st, pl = OR.round_step(d, st, pl, w["prio"], w["tmpl"], w["role"], w["part_off"],
                                               w["part_dev"], w["mapping"], w["per"], w["budget"], w["max_batch"])
            st[st == 1] = 2
        dt = (time.perf_counter() - t0) / k
        line["cpu_baseline"] = {"value": 1.0 / dt, "unit": "rounds/s", "cores": 1, "kind": "oracle",
                                "sample": "the first %d rounds (Python frontiers/batch, C++ simulations)" % k}
    print(json.dumps(line))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None,
                    help="timed steps (default: 20, fewer when a step is long -- about a minute of timed work)")
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", type=int, default=5, choices=[1, 2, 3, 4, 5, 6])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--rounds", action="store_true",
                    help="time scheduling rounds (Algorithm 1) instead of the candidate simulation")
    ap.add_argument("--estimators", action="store_true",
                    help="time the online estimators (refit, durations, links) instead of the simulation")
    ap.add_argument("--arbitrated", action="store_true",
                    help="arbitrated transfers (Sec. 3.5.2) instead of pure-latency ones")
    ap.add_argument("--placements", default="uniform", choices=["uniform", "structured"],
                    help="full placement rows: uniform i.i.d. device ids, or contiguous per-request "
                         "stages on random accelerators")
    ap.add_argument("--gmg-staging", default="default", choices=["default", "shared", "l1"],
                    help="full placements: the GMG's hot fields staged in every CTA's shared memory, or read "
                         "through the L1 path (default: the library's choice)")
    ap.add_argument("--candidates", type=int, default=None,
                    help="profiling aid: simulate only the first N candidates of each half "
                         "(the line then describes that smaller batch)")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3
    if args.steps is None and (args.impl == "reference" or args.estimators or args.rounds):
        args.steps = 20
    if args.impl == "reference":
        return reference_arm(args)
    if args.estimators:
        return run_estimators(args)
    if args.rounds:
        return run_rounds(args)

    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)

    from paper_2608_15762_gb300 import build as lib_build
    lib_build.build()
    p = prepare(args.config, rank, world, device, cap=args.candidates, arbitrated=args.arbitrated,
                structured=args.placements == "structured", staging=args.gmg_staging)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=device)

    def barrier():
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()
            torch.cuda.synchronize()

    def max_over_ranks(x):
        if world == 1:
            return x
        t = torch.tensor([x], dtype=torch.float64, device=device)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        return float(t.item())

    warm = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    for i in range(args.warmup):
        if i == args.warmup - 1:
            warm[0].record()
        run_step(p)
        if i == args.warmup - 1:
            warm[1].record()
    barrier()
    steps = args.steps
    if steps is None:
        # about a minute of timed work: 20 steps, fewer when a step is long
        warm_ms = max_over_ranks(warm[0].elapsed_time(warm[1])) if args.warmup else 0.0
        steps = max(3, min(20, int(60000 // max(warm_ms, 1e-3))))
    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    step_ev, kern_ev = [], []
    launches = 0
    names = [n for n, on in (("full", p.n_full), ("base", p.n_inc), ("inc", p.n_inc)) if on]
    for _ in range(steps):
        flush.fill_(1)
        e = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
        ke = {n: (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for n in names}
        e[0].record()
        launches += run_step(p, ev=ke)
        e[1].record()
        step_ev.append((e[0], e[1]))
        kern_ev.append(ke)
    barrier()
    clocks = sampler.stop()
    step_ms = [a.elapsed_time(b) for a, b in step_ev]
    kern_ms = {n: statistics.mean(ke[n][0].elapsed_time(ke[n][1]) for ke in kern_ev) for n in names}
    ms = max_over_ranks(statistics.mean(step_ms))

    # end to end through the public API with host buffers (fewer steps when a
    # step is long: at least 3, about a minute of work)
    e2e_steps = max(3, min(steps, int(60000 // max(ms, 1e-3))))
    run_e2e_step(p)
    barrier()
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        run_e2e_step(p)
    barrier()
    e2e_ms = max_over_ranks(1000 * (time.perf_counter() - t0) / e2e_steps)

    wl = p.wl
    N, D = wl.desc.n_ops, wl.desc.n_dev
    K_all = p.n_full_total + p.n_inc_total      # every rank's candidates, each counted once
    inc_events = int(p.out.events[p.n_full:p.K].sum().item()) if p.n_inc else 0
    ev_local = p.n_full * N + inc_events
    ev_all = ev_local
    if world > 1:
        t = torch.tensor([ev_local], dtype=torch.int64, device=device)
        torch.distributed.all_reduce(t)
        ev_all = int(t.item())
        from paper_2608_15762_gb300 import gmgsim as G
        best = list(G.select_best_across_ranks(p.best, p.to_global))
    else:
        best = p.best.cpu().tolist()
        if best[0] >= 0:
            best[0] = p.to_global(best[0])
    value = K_all / (ms / 1000)
    pk = peaks()
    props = torch.cuda.get_device_properties(device)
    issue_peak = props.multi_processor_count * 4 * pk["sm_max_mhz"] * 1e6 / 1e9  # Ginst/s
    arb_kern = "sim_arb_kernel" if D <= 32 else "sim_arbw_kernel"
    staged_run = p.staging == 1 or (p.staging == 0 and p.g.info["stageable"] == 1 and not p.arb)
    full_kern = "sim_full_staged_kernel" if staged_run else "sim_full_kernel"
    kname = {"full": arb_kern if p.arb else full_kern,
             "inc": "sim_arb_inc_kernel" if p.arb_base else arb_kern if p.arb else "sim_inc_kernel",
             "base": "sim_arb_base_kernel" if p.arb_base else "sim_base_kernel"}
    kcount = {"full": p.n_full, "inc": p.n_inc, "base": 1}
    out_bytes_per_cand = 8 + 8 + 4 + 4 + 4 + 4 + 8 + 4 + 8 + 8 * D
    alg_bytes = {"full": p.n_full * (W_ld(N) + out_bytes_per_cand),
                 "inc": (sum(t.numel() * t.element_size() for t in p.host_moves) + p.n_inc * out_bytes_per_cand)
                 if p.n_inc else 0,
                 "base": W_ld(N) + 16 * N}
    wname = wl.name + ("-structured" if p.structured else "")
    kernels = {}
    for n in names:
        ppath = profile_path(kname[n], wname)
        extra = () if not p.arb or (n == "base" and not p.arb_base) else (ARB_SOURCES if D <= 32 else ARBW_SOURCES)
        prof = read_profile(ppath, extra)
        kd = {"kernel": kname[n], "launch_ms": kern_ms[n], "units": kcount[n],
              "hbm_gbs": alg_bytes[n] / (kern_ms[n] / 1000) / 1e9, "inst_per_launch": None, "issue_frac": None,
              "dram_bytes_per_launch": None}
        if prof:
            inst = prof["inst_per_cand"] * kcount[n]
            kd.update(inst_per_launch=inst, issue_frac=inst / (kern_ms[n] / 1000) / 1e9 / issue_peak,
                      dram_bytes_per_launch=prof["dram_per_cand"] * kcount[n],
                      inst_src="%s (ncu on %d units, scaled to %d)" % (os.path.relpath(ppath, ROOT),
                                                                      prof["captured"], kcount[n]))
        kernels[n] = kd
    dom = max(names, key=lambda n: kern_ms[n])
    kd = kernels[dom]
    roof = {"bound": "alu", "unit": "Ginst/s", "peak": issue_peak,
            "peak_src": "%d SMs x 4 issue slots x %.0f MHz (%s sm_max_mhz)" % (
                props.multi_processor_count, pk["sm_max_mhz"], pk["src"]),
            "achieved": None, "frac": None, "traffic": kd["dram_bytes_per_launch"], "kernel": kd["kernel"],
            "kernel_ms": kd["launch_ms"]}
    if kd["inst_per_launch"] is not None:
        ach = kd["inst_per_launch"] / (kd["launch_ms"] / 1000) / 1e9
        roof.update(achieved=ach, frac=ach / issue_peak, inst_per_launch=kd["inst_per_launch"],
                    inst_src=kd["inst_src"],
                    inst_per_op_event=kd["inst_per_launch"] / max(kcount[dom] * N if dom == "full" else 1, 1)
                    if dom == "full" else None)
    if all(kernels[n]["inst_per_launch"] is not None for n in names):
        tot = sum(kernels[n]["inst_per_launch"] for n in names)
        roof["step"] = {"inst_per_step": tot, "issue_frac": tot / (ms / 1000) / 1e9 / issue_peak,
                        "inst_per_op_event": tot / max(ev_local, 1),
                        "note": "every kernel of the step (instructions from the committed ncu summaries) over "
                                "the whole step time"}
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "strong",
        "vs_baseline": None, "dtype": "int64", "data": "synthetic",
        "ms_per_step_best": min(step_ms), "ms_per_step_median": statistics.median(step_ms),
        "config": {"workload": wl.name, "candidates": K_all, "full_placements": p.n_full_total,
                   "incremental_candidates": p.n_inc_total, "n_ops": N, "n_dev": D,
                   "transfers": "arbitrated" if p.arb else "latency",
                   "incremental": ("resumed from the arbitrated base snapshot" if p.arb_base else
                                   "moved placements simulated in full" if p.arb else
                                   "resumed from the base snapshot") if p.n_inc_total else None,
                   "placements": "structured" if p.structured else "uniform",
                   "gmg_staging": "shared memory (bulk-copied once per CTA)" if staged_run else "L1 path",
                   "l2": "flushed between steps (256 MiB write), each step timed with CUDA events",
                   "parallelism": "dp%d over candidates (contiguous blocks of each half per rank)" % world},
        # full placements simulate every op; an incremental candidate re-simulates
        # the ops its `events` output counts (read after the timed region)
        "op_events_per_s": ev_all / (ms / 1000),
        "roofline": roof,
        "kernels": kernels,
        "hbm": {"achieved": kd["hbm_gbs"], "peak": pk["hbm_gbs"], "unit": "GB/s",
                "frac": kd["hbm_gbs"] / pk["hbm_gbs"], "algorithmic_bytes_per_launch": alg_bytes[dom],
                "dram_bytes_per_candidate": (kd["dram_bytes_per_launch"] / kcount[dom])
                if kd["dram_bytes_per_launch"] else None,
                "algorithmic_bytes_per_candidate": alg_bytes[dom] / max(kcount[dom], 1),
                "note": "placement bytes read + per-candidate outputs written; the kernel is issue/latency-bound"},
        "e2e": {"value": K_all / (e2e_ms / 1000), "unit": UNIT, "ms_per_step": e2e_ms, "steps": e2e_steps,
                "h2d_bytes_per_step": h2d_bytes(p) * world, "d2h_bytes_per_step": 16 * world},
        "gpu_launches": launches,
        "clocks": clocks,
        "best": best,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(wl, arbitrated=p.arb, structured=p.structured)
    if rank == 0:
        print(json.dumps(line))
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def W_ld(n):
    return max(16, (n + 15) // 16 * 16)


if __name__ == "__main__":
    sys.exit(main())
