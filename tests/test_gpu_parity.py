"""GPU parity: the CUDA path through the C ABI against the CPU oracle, bit for
bit on every output field (all times and sizes are int64)."""
import glob
import json
import os

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_common import compare, oracle_rows, torch_place  # noqa: E402
from helpers import mk, row  # noqa: E402
from oracle import oracle as O  # noqa: E402
from paper_2608_15762_gb300 import gmgsim as G  # noqa: E402
from paper_2608_15762_gb300 import workloads as W  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_15762_gb300 import build
    build.build()
    assert torch.cuda.is_available()


def _random_case(seed, n, D, **kw):
    d = W.random_desc(seed, n, D, **kw)
    g = np.random.default_rng(seed)
    K = 37
    ld = W.placement_ld(n)
    rows = np.zeros((K, ld), np.uint8)
    rows[:, :n] = g.integers(0, D, (K, n))
    return d, rows


@pytest.mark.parametrize("seed,n,D,kw", [
    (1, 1, 1, {}),
    (2, 7, 2, {}),
    (3, 33, 3, dict(explicit_cons=True)),
    (4, 64, 4, dict(link_hetero=False)),
    (5, 150, 8, dict(explicit_cons=True, dur_hi=2000)),
    (6, 257, 5, dict(max_pred=6)),
    (7, 300, 32, dict(explicit_cons=True)),
    (8, 200, 33, {}),          # accelerator state in scratch arrays
    (9, 500, 256, dict(explicit_cons=True, bytes_hi=1 << 30)),
    (10, 1000, 16, dict(edge_p=0.9, max_pred=4)),
    (11, 90, 6, dict(with_release=False, with_avail0=False, cap=1 << 40)),
    (15, 300, 8, dict(dur_hi=1 << 32)),               # times beyond 2^31: 64-bit instances
    (16, 200, 40, dict(dur_hi=1 << 31, explicit_cons=True)),
    (17, 150, 4, dict(dur_hi=1 << 40, link_hetero=False)),
    (18, 300, 8, dict(n_types=2)),                    # per-type durations (Sec. 3.3.1)
    (19, 200, 40, dict(n_types=3, explicit_cons=True)),
    (20, 150, 4, dict(n_types=2, dur_hi=1 << 32)),
    (21, 300, 256, dict(n_types=4, explicit_cons=True)),   # typed, accelerator state in shared memory
])
def test_random_dags_bit_exact(seed, n, D, kw):
    d, rows = _random_case(seed, n, D, **kw)
    g = G.gmg_create(d)
    if kw.get("dur_hi", 0) >= 1 << 31:
        assert g.info["time_bound"] >= 1 << 31
    K = rows.shape[0]
    tk = torch.tensor([0, 5, K - 1], dtype=torch.int32, device="cuda")
    out = G.sim_batch(g, torch_place(rows), req_done=True, trace_k=tk)
    best = G.select_best(out)
    best1 = G.select_best(out, score_mode=1)
    torch.cuda.synchronize()
    got = out.to_numpy()
    s, pk, rq = oracle_rows(d, rows)
    compare(got, s, pk, rq)
    for slot, k in enumerate([0, 5, K - 1]):
        r = O.simulate(d, rows[k])
        assert np.array_equal(got["trace_start"][slot], r["start"])
        assert np.array_equal(got["trace_finish"][slot], r["finish"])
    assert best.cpu().tolist() == list(O.select_best(s, 0))
    assert best1.cpu().tolist() == list(O.select_best(s, 1))


def test_bad_device_rows_and_empty_graph():
    d, rows = _random_case(12, 40, 3)
    rows[3, 17] = 3
    rows[9, 39] = 255
    rows[11, 40] = 200       # padding byte beyond n_ops: ignored
    g = G.gmg_create(d)
    out = G.sim_batch(g, torch_place(rows), req_done=True)
    torch.cuda.synchronize()
    s, pk, rq = oracle_rows(d, rows)
    compare(out.to_numpy(), s, pk, rq)
    st = out.status.cpu().numpy()
    assert st[3] == G.SIM_BADDEV and st[9] == G.SIM_BADDEV and st[11] == 0
    e = mk([], [], n_dev=2)
    ge = G.gmg_create(e)
    oe = G.sim_batch(ge, torch_place(np.zeros((4, 16), np.uint8)))
    torch.cuda.synchronize()
    assert oe.status.cpu().tolist() == [0] * 4 and oe.score.cpu().tolist() == [0] * 4


GOLDEN = sorted(glob.glob(os.path.join(os.path.dirname(__file__), "golden", "*.json")))


@pytest.mark.parametrize("path", GOLDEN, ids=[os.path.basename(p) for p in GOLDEN])
def test_golden_examples_on_gpu(path):
    """Each hand-derived worked example, with the transfer model and link
    table the fixture names, through the C ABI: start/finish of every op,
    peaks, makespan, score, SLA, request completions and the first violation."""
    with open(path) as f:
        fx = json.load(f)
    gr = fx["graph"]
    arb = gr.get("transfer_mode", 0) == 1
    for case in fx["cases"]:
        d = mk(gr["preds"], gr["dur"], gr["out_bytes"], n_dev=gr["n_dev"], bw=gr["bw"],
               lat=gr["lat"], release=gr.get("release"), avail0=gr.get("avail0"),
               req_id=gr.get("req_id"), deadline=gr.get("deadline"), cap=case["cap"])
        if gr.get("link_id") is not None:
            d.link_id = np.asarray(gr["link_id"], np.int32)
        g = G.gmg_create(d)
        rows = row(fx["place"])[None, :]
        tk = torch.tensor([0], dtype=torch.int32, device="cuda")
        out = G.sim_batch(g, torch_place(rows), req_done=True, trace_k=tk,
                          arbitrated=arb).to_numpy()
        assert out["status"][0] == 0
        assert out["trace_start"][0].tolist() == case["start"]
        assert out["trace_finish"][0].tolist() == case["finish"]
        assert out["peak"][0].tolist() == case["peak"]
        assert out["makespan"][0] == case["makespan"] and out["score"][0] == case["score"]
        assert out["sla_miss"][0] == case["sla_miss"]
        assert out["req_done"][0].tolist() == case["req_done"]
        viol = None if not out["viol_flag"][0] else [int(out["viol_time"][0]),
                                                     int(out["viol_op"][0]),
                                                     int(out["viol_dev"][0])]
        assert viol == case["viol"]


def test_queue_capacity_status():
    # one op feeding 120 successors: 120 ready keys at once, beyond the
    # 32-key register tier plus a 3-slot heap
    n = 121
    d = mk([[]] + [[0]] * 120, [5] * n, [1] * n, n_dev=4, bw=1, lat=1)
    g = G.gmg_create(d)
    rows = np.zeros((8, 128), np.uint8)
    rows[:, :n] = np.random.default_rng(0).integers(0, 4, (8, n))
    out = G.sim_batch(g, torch_place(rows), queue_cap=3)
    ok = G.sim_batch(g, torch_place(rows))
    torch.cuda.synchronize()
    st = out.status.cpu().numpy()
    assert (st == G.SIM_QUEUE).all()
    assert (out.score.cpu().numpy() == np.iinfo(np.int64).max).all()
    assert G.select_best(out).cpu().tolist()[0] == -1
    s, pk, rq = oracle_rows(d, rows)
    compare(ok.to_numpy(), s, pk, rq)


@pytest.mark.parametrize("wpb", [1, 2, 3, 4])
def test_launch_shapes_agree(wpb):
    d, rows = _random_case(14, 200, 8)
    g = G.gmg_create(d)
    out = G.sim_batch(g, torch_place(rows), req_done=True, warps_per_block=wpb)
    torch.cuda.synchronize()
    s, pk, rq = oracle_rows(d, rows)
    compare(out.to_numpy(), s, pk, rq)


# ---------------------------------------------------------------------------
# The workloads
# ---------------------------------------------------------------------------

def test_workload_tiny_all_candidates():
    wl = W.config1()
    rows = wl.all_full_rows()
    g = G.gmg_create(wl.desc)
    out = G.sim_batch(g, torch_place(rows), req_done=True)
    best = G.select_best(out)
    torch.cuda.synchronize()
    s, pk, rq = oracle_rows(wl.desc, rows)
    compare(out.to_numpy(), s, pk, rq)
    assert best.cpu().tolist() == list(O.select_best(s, 0))


def test_workload_prefill_all_candidates():
    wl = W.config2()
    rows = wl.all_full_rows()
    g = G.gmg_create(wl.desc)
    out = G.sim_batch(g, torch_place(rows), req_done=True)
    best = G.select_best(out)
    best1 = G.select_best(out, score_mode=1)
    torch.cuda.synchronize()
    s, pk, rq = oracle_rows(wl.desc, rows)
    compare(out.to_numpy(), s, pk, rq)
    assert best.cpu().tolist() == list(O.select_best(s, 0))
    assert best1.cpu().tolist() == list(O.select_best(s, 1))
    assert (s["sla_miss"] > 0).any()


def test_workload_two_accelerator_types_all_candidates():
    """Every placement of the prefill graph on two accelerator types."""
    wl = W.config6()
    rows = wl.all_full_rows()
    g = G.gmg_create(wl.desc)
    tk = torch.tensor([0, 4095], dtype=torch.int32, device="cuda")
    out = G.sim_batch(g, torch_place(rows), req_done=True, trace_k=tk)
    best = G.select_best(out)
    torch.cuda.synchronize()
    got = out.to_numpy()
    s, pk, rq = oracle_rows(wl.desc, rows)
    compare(got, s, pk, rq)
    assert best.cpu().tolist() == list(O.select_best(s, 0))
    for slot, k in enumerate([0, 4095]):
        r = O.simulate(wl.desc, rows[k])
        assert np.array_equal(got["trace_start"][slot], r["start"])


def test_workload_memory_tight_all_candidates():
    """Every one of the 8,192 placements of the memory-tight decode workload."""
    wl = W.config4()
    rows = wl.all_full_rows()
    g = G.gmg_create(wl.desc)
    out = G.sim_batch(g, torch_place(rows), req_done=True)
    torch.cuda.synchronize()
    got = out.to_numpy()
    s, pk, rq = oracle_rows(wl.desc, rows)
    compare(got, s, pk, rq)
    frac = float(got["viol_flag"].mean())
    assert 0.25 < frac < 0.35, frac
    assert (got["status"] == 0).all() and (got["events"] == wl.desc.n_ops).all()


def test_workload_large_full_size_sampled():
    """The 256-accelerator workload exactly as the benchmark runs it: every
    full placement and every incremental candidate on the GPU, sampled
    candidates of both halves checked against the oracle."""
    wl = W.config5()
    g = G.gmg_create(wl.desc)
    out = G.sim_batch(g, torch_place(wl.all_full_rows()), req_done=True)
    b = G.base_create(g, torch.from_numpy(wl.base_place).cuda())
    off, op, dv = G.moves_to_device(wl.moves, "cuda")
    inc = G.sim_incremental(g, b, off, op, dv, req_done=True)
    best = G.select_best(out)
    torch.cuda.synchronize()
    got, goti = out.to_numpy(), inc.to_numpy()
    assert (got["status"] == 0).all() and (goti["status"] == 0).all()
    rng = np.random.default_rng(55)
    ks = np.sort(rng.choice(wl.n_full, 256, replace=False))
    s, pk, rq = oracle_rows(wl.desc, wl.full_rows(ks))
    compare(got, s, pk, rq, ks=ks)
    ki = np.sort(rng.choice(wl.moves.n_cand, 256, replace=False))
    si, pki, rqi = O.incremental_batch(wl.desc, wl.base_place, wl.moves.subset(ki))
    compare(goti, si, pki, rqi, ks=ki)
    assert best.cpu().tolist()[1] == int(got["score"].min())


# ---------------------------------------------------------------------------
# The GMG staged in shared memory (sim_opts_t.gmg_staging)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("which", ["tiny", "prefill", "random", "random_wide"])
def test_staged_gmg_bit_exact(which):
    """sim_batch with each CTA's warps reading the hot GMG fields from a
    shared-memory copy made with bulk copies: every candidate against the
    oracle, and the same bytes as the L1 path."""
    if which in ("tiny", "prefill"):
        wl = W.config1() if which == "tiny" else W.config2()
        d, rows = wl.desc, wl.all_full_rows()
    else:
        D = 6 if which == "random" else 32
        d = W.random_desc(61 if which == "random" else 62, 700, D, link_hetero=False, explicit_cons=True,
                          window=12 if which == "random" else 200)
        rows = _random_case(61, 700, D, link_hetero=False)[1]
        rows = np.concatenate([rows] * 40)[:1000]
    g = G.gmg_create(d)
    tk = torch.tensor([0, rows.shape[0] - 1], dtype=torch.int32, device="cuda")
    st = G.sim_batch(g, torch_place(rows), req_done=True, trace_k=tk, gmg_staging=G.GMG_STAGING_SHARED)
    l1 = G.sim_batch(g, torch_place(rows), req_done=True, trace_k=tk, gmg_staging=G.GMG_STAGING_L1)
    torch.cuda.synchronize()
    got = st.to_numpy()
    s, pk, rq = oracle_rows(d, rows)
    compare(got, s, pk, rq)
    ref = l1.to_numpy()
    for f in ("trace_start", "trace_finish", "peak", "req_done", "score", "makespan"):
        assert np.array_equal(got[f], ref[f]), f


def test_staging_refused_where_it_does_not_apply():
    """Two accelerator types, per-pair links or arbitrated transfers: the
    compact staged record does not hold them, and the call says so."""
    rows = np.zeros((4, 320), np.uint8)
    for d, arb in ((W.random_desc(63, 300, 4, n_types=2, link_hetero=False), False),
                   (W.random_desc(64, 300, 4, link_hetero=True), False),
                   (W.random_desc(65, 300, 4, link_hetero=False), True)):
        g = G.gmg_create(d)
        with pytest.raises(G.GmgError) as e:
            G.sim_batch(g, torch_place(rows), gmg_staging=G.GMG_STAGING_SHARED, arbitrated=arb)
        assert e.value.code == G.GMG_EINVAL
        assert g.info["stageable"] == (1 if arb else 0)   # arbitration is refused by the call only


def test_stageable_reports_the_default():
    """gmg_info_t.stageable says whether sim_batch stages the graph by
    default: the prefill graph's copy fits in shared memory, the memory-tight
    decode graph's (N = 197,632) does not, although both have the compact
    fields; an explicit staging request on the latter is refused."""
    assert G.gmg_create(W.make_workload(2).desc).info["stageable"] == 1
    g4 = G.gmg_create(W.make_workload(4).desc)
    assert g4.info["stageable"] == 0
    rows = np.zeros((2, W.placement_ld(g4.n_ops)), np.uint8)
    with pytest.raises(G.GmgError) as e:
        G.sim_batch(g4, torch_place(rows), gmg_staging=G.GMG_STAGING_SHARED)
    assert e.value.code == G.GMG_EINVAL
