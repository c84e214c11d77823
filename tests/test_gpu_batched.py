"""GPU parity of the batched sweep (graphs on more than 32 accelerators: the
kernels start consecutive READY ops together, one per lane) against the
oracle, bit for bit: wide graphs where dozens of ops are ready at once,
batches whose ops share an accelerator, joins whose inputs several ops of
one batch complete, accelerator types, 64-bit times, traces, incremental
candidates and the base snapshot."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_common import compare, oracle_rows, torch_place  # noqa: E402
from helpers import mk  # noqa: E402
from oracle import oracle as O  # noqa: E402
from paper_2608_15762_gb300 import gmgsim as G  # noqa: E402
from paper_2608_15762_gb300 import workloads as W  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_15762_gb300 import build
    build.build()
    assert torch.cuda.is_available()


def _rows(seed, K, n, D, hi=None):
    g = np.random.default_rng(seed)
    rows = np.zeros((K, W.placement_ld(n)), np.uint8)
    rows[:, :n] = g.integers(0, D if hi is None else hi, (K, n))
    return rows


def _check_full(d, rows, traced=(0,)):
    g = G.gmg_create(d)
    assert g.info["batched_sweep"] == 1
    tk = torch.tensor(list(traced), dtype=torch.int32, device="cuda")
    out = G.sim_batch(g, torch_place(rows), req_done=True, trace_k=tk)
    best = G.select_best(out)
    torch.cuda.synchronize()
    got = out.to_numpy()
    s, pk, rq = oracle_rows(d, rows)
    compare(got, s, pk, rq)
    for slot, k in enumerate(traced):
        r = O.simulate(d, rows[k])
        assert np.array_equal(got["trace_start"][slot], r["start"])
        assert np.array_equal(got["trace_finish"][slot], r["finish"])
    assert best.cpu().tolist() == list(O.select_best(s, 0))
    return got


@pytest.mark.parametrize("seed,n,D,kw", [
    (31, 2000, 64, dict(window=400)),
    (32, 3000, 256, dict(window=1000, explicit_cons=True)),
    (33, 1500, 33, dict(window=300, max_pred=5, edge_p=0.9)),
    (34, 2000, 100, dict(window=500, n_types=3)),                   # per-type durations
    (35, 1200, 48, dict(window=300, dur_hi=1 << 30)),               # 64-bit times
    (36, 2500, 200, dict(window=2500, with_release=False, dur_hi=4)),  # many equal times
])
def test_wide_graphs_bit_exact(seed, n, D, kw):
    d = W.random_desc(seed, n, D, **kw)
    _check_full(d, _rows(seed, 41, n, D), traced=(0, 40))
    if kw.get("dur_hi", 0) >= 1 << 30:
        assert G.gmg_create(d).info["t32"] == 0


def test_batches_sharing_an_accelerator():
    """Placements on 2 (or 3) of 64 accelerators: most batches hold several ops
    of one accelerator, which start in key order."""
    d = W.random_desc(41, 2000, 64, window=600)
    for hi in (2, 3):
        _check_full(d, _rows(41 + hi, 37, 2000, 64, hi=hi), traced=(0, 36))


def test_joins_completed_inside_one_batch():
    """Groups of 40 roots with equal release feed one join each (and the
    joins feed a final join): every root of a group is in one batch (or two),
    so several lanes complete a join's inputs at once; the join is queued once."""
    preds, dur = [], []
    joins = []
    for grp in range(6):
        base = len(preds)
        for _ in range(40):
            preds.append([])
            dur.append(3 + grp)
        preds.append(list(range(base, base + 40)))
        dur.append(7)
        joins.append(len(preds) - 1)
    preds.append(joins)
    dur.append(5)
    n = len(preds)
    rel = [10 * (i // 41) if not preds[i] else 0 for i in range(n)]
    d = mk(preds, dur, [1 << 10] * n, n_dev=40, bw=1000, lat=1, release=rel,
           req_id=[0] * n, deadline=[10_000], cap=[1 << 30] * 40)
    rows = _rows(43, 33, n, 40)
    rows[1, :n] = 5               # everything on one accelerator
    rows[2, :n] = np.arange(n) % 40
    _check_full(d, rows, traced=(0, 1, 2))


def test_large_workload_first_candidates_traced():
    """The 256-accelerator workload's first placements, start and finish of
    every one of its 213,568 ops."""
    wl = W.config5()
    rows = wl.full_rows(range(8))
    g = G.gmg_create(wl.desc)
    assert g.info["batched_sweep"] == 1 and g.info["t32"] == 1
    tk = torch.tensor([0, 7], dtype=torch.int32, device="cuda")
    out = G.sim_batch(g, torch_place(rows), req_done=True, trace_k=tk)
    torch.cuda.synchronize()
    got = out.to_numpy()
    s, pk, rq = oracle_rows(wl.desc, rows)
    compare(got, s, pk, rq)
    for slot, k in enumerate((0, 7)):
        r = O.simulate(wl.desc, rows[k])
        assert np.array_equal(got["trace_start"][slot], r["start"])
        assert np.array_equal(got["trace_finish"][slot], r["finish"])


@pytest.mark.parametrize("seed,n,D,kw", [
    (51, 2000, 64, dict(window=400)),
    (52, 2500, 256, dict(window=800, explicit_cons=True)),
    (53, 1500, 40, dict(window=300, n_types=2)),
    (54, 1200, 48, dict(window=300, dur_hi=1 << 30)),
])
def test_incremental_wide_graphs_bit_exact(seed, n, D, kw):
    d = W.random_desc(seed, n, D, **kw)
    base = np.random.default_rng(seed).integers(0, D, n).astype(np.uint8)
    mv = W.random_moves(seed, 200, base, D, max_moves=20)
    g = G.gmg_create(d)
    assert g.info["batched_sweep"] == 1
    b = G.base_create(g, torch.from_numpy(base).cuda())
    off, op, dv = G.moves_to_device(mv, "cuda")
    out = G.sim_incremental(g, b, off, op, dv, req_done=True)
    torch.cuda.synchronize()
    s, pk, rq = O.incremental_batch(d, base, mv)
    compare(out.to_numpy(), s, pk, rq)
    assert G.select_best(out).cpu().tolist() == list(O.select_best(s, 0))
