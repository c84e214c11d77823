"""GPU parity of the incremental path (base_create + sim_incremental) against
the oracle's incremental batch, bit for bit, events included."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_common import compare  # noqa: E402
from oracle import oracle as O  # noqa: E402
from paper_2608_15762_gb300 import gmgsim as G  # noqa: E402
from paper_2608_15762_gb300 import workloads as W  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_15762_gb300 import build
    build.build()
    assert torch.cuda.is_available()


def _run(desc, base, moves, **kw):
    g = G.gmg_create(desc)
    b = G.base_create(g, torch.from_numpy(np.ascontiguousarray(base)).cuda())
    off, op, dv = G.moves_to_device(moves, "cuda")
    out = G.sim_incremental(g, b, off, op, dv, req_done=True, **kw)
    torch.cuda.synchronize()
    return g, b, out


@pytest.mark.parametrize("seed,n,D,kw", [
    (1, 5, 2, {}),
    (2, 40, 3, dict(explicit_cons=True)),
    (3, 120, 4, {}),
    (4, 300, 8, dict(explicit_cons=True, dur_hi=500)),
    (5, 600, 33, {}),
    (6, 400, 256, dict(explicit_cons=True)),
    (7, 1500, 16, dict(edge_p=0.8, max_pred=4, dur_hi=3000)),
    (8, 300, 8, dict(dur_hi=1 << 32)),             # times beyond 2^31: 64-bit instances
    (9, 300, 40, dict(dur_hi=1 << 31, explicit_cons=True)),
    (10, 400, 8, dict(n_types=2)),                 # per-type durations
    (11, 300, 33, dict(n_types=3, explicit_cons=True)),
])
def test_random_incremental_bit_exact(seed, n, D, kw):
    d = W.random_desc(5000 + seed, n, D, **kw)
    if kw.get("dur_hi", 0) >= 1 << 31:
        assert G.gmg_create(d).info["time_bound"] >= 1 << 31
    g0 = np.random.default_rng(seed)
    base = g0.integers(0, D, n).astype(np.uint8)
    mv = W.random_moves(seed, 300, base, D, max_moves=12)
    g, b, out = _run(d, base, mv)
    s, pk, rq = O.incremental_batch(d, base, mv)
    compare(out.to_numpy(), s, pk, rq)
    best = G.select_best(out).cpu().tolist()
    assert best == list(O.select_best(s, 0))


def test_move_status_codes_and_bad_base():
    d = W.random_desc(77, 30, 3)
    base = np.zeros(30, np.uint8)
    mv = W.Moves(np.array([0, 0, 2, 4, 5, 6, 6], np.int32),
                 np.array([1, 2, 3, 3, 31, 4], np.int32),
                 np.array([1, 2, 1, 2, 0, 3], np.uint8))
    g, b, out = _run(d, base, mv)
    s, pk, rq = O.incremental_batch(d, base, mv)
    compare(out.to_numpy(), s, pk, rq)
    bad = base.copy()
    bad[7] = 9
    g, b, out = _run(d, bad, mv)
    assert (out.status.cpu().numpy() == G.SIM_BADBASE).all()


def test_incremental_equals_full_batch_of_applied_moves():
    d = W.random_desc(91, 800, 8, dur_hi=1000)
    base = np.random.default_rng(1).integers(0, 8, 800).astype(np.uint8)
    mv = W.random_moves(3, 128, base, 8, max_moves=20)
    g, b, out = _run(d, base, mv)
    ld = W.placement_ld(800)
    rows = np.zeros((128, ld), np.uint8)
    for k in range(128):
        rows[k, :800] = base
        for m in range(mv.off[k], mv.off[k + 1]):
            rows[k, mv.op[m]] = mv.dev[m]
    full = G.sim_batch(g, torch.from_numpy(rows).cuda(), req_done=True)
    torch.cuda.synchronize()
    a, f = out.to_numpy(), full.to_numpy()
    for key in ("status", "makespan", "score", "viol_flag", "viol_op", "viol_dev", "viol_time",
                "sla_miss", "peak", "req_done"):
        assert np.array_equal(a[key], f[key]), key


def test_workload_incremental_all_candidates():
    """Every one of the 16,384 move lists of the incremental workload."""
    wl = W.config3()
    mv = wl.moves
    g, b, out = _run(wl.desc, wl.base_place, mv)
    got = out.to_numpy()
    s, pk, rq = O.incremental_batch(wl.desc, wl.base_place, mv)
    compare(got, s, pk, rq)
    assert (got["status"] == 0).all()
    assert (got["events"] <= wl.desc.n_ops).all() and (got["events"] > 0).all()
