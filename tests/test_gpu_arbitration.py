"""GPU parity of the arbitrated-transfer simulation (sim_batch with
transfer_mode = GMG_TRANSFER_ARBITRATED, Sec. 3.5.2) against the oracle's
arbitrated mode, bit for bit on every output field and on the traced
schedules: random graphs with shared links, zero-length transfers, 32- and
64-bit times, accelerator types, the hand-worked conflict cases, the
prefill, incremental-shaped and heterogeneous workloads, and the refusals."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_common import compare, torch_place  # noqa: E402
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


def _links(kind, D, g):
    if kind == "pair":          # one link per unordered pair (both directions share it)
        a, b = np.meshgrid(np.arange(D), np.arange(D), indexing="ij")
        return (np.minimum(a, b) * D + np.maximum(a, b)).astype(np.int32).reshape(-1)
    if kind == "uplink":        # accelerators 2m and 2m+1 share one uplink
        return np.repeat(np.arange(D, dtype=np.int32) // 2 * D, D)
    if kind == "random":
        return g.integers(0, max(D * D // 3, 1), D * D).astype(np.int32)
    return None


def _case(seed, n, D, links=None, K=37, zero=False, **kw):
    d = W.random_desc(seed, n, D, **kw)
    g = np.random.default_rng(seed)
    d.link_id = _links(links, D, g)
    if zero:
        d.out_bytes[::2] = 0
        d.lat[:] = 0
    ld = W.placement_ld(n)
    rows = np.zeros((K, ld), np.uint8)
    rows[:, :n] = g.integers(0, D, (K, n))
    return d, rows


def _run_and_compare(d, rows, trace=(0,)):
    g = G.gmg_create(d)
    K = rows.shape[0]
    tk = torch.tensor(list(trace), dtype=torch.int32, device="cuda")
    out = G.sim_batch(g, torch_place(rows), req_done=True, trace_k=tk, arbitrated=True)
    best = G.select_best(out)
    torch.cuda.synchronize()
    got = out.to_numpy()
    s, pk, rq = O.simulate_batch(d, rows, arbitrated=True)
    compare(got, s, pk, rq)
    for slot, k in enumerate(trace):
        r = O.simulate(d, rows[k], arbitrated=True)
        assert np.array_equal(got["trace_start"][slot], r["start"]), k
        assert np.array_equal(got["trace_finish"][slot], r["finish"]), k
    assert best.cpu().tolist() == list(O.select_best(s, 0))
    return got, s


@pytest.mark.parametrize("seed,n,D,links,kw", [
    (1, 1, 1, None, {}),
    (2, 9, 2, None, {}),
    (3, 40, 3, "pair", dict(explicit_cons=True)),
    (4, 64, 4, "uplink", dict(link_hetero=False)),
    (5, 150, 8, None, dict(explicit_cons=True, dur_hi=2000)),
    (6, 257, 5, "random", dict(max_pred=6)),
    (7, 300, 32, "pair", dict(explicit_cons=True)),
    (8, 1000, 16, "uplink", dict(edge_p=0.9, max_pred=4)),
    (9, 90, 6, None, dict(with_release=False, with_avail0=False, cap=1 << 40)),
    (10, 300, 8, "random", dict(dur_hi=1 << 32)),      # 64-bit times
    (12, 300, 8, "pair", dict(n_types=2)),
    (13, 200, 32, "random", dict(n_types=3, explicit_cons=True)),
    (14, 150, 4, None, dict(n_types=2, dur_hi=1 << 32)),
    (15, 400, 7, "uplink", dict(bytes_hi=1 << 20, explicit_cons=True)),
    # more than 32 accelerators: per-accelerator transfer state in tables
    (16, 200, 33, None, {}),
    (17, 300, 40, "pair", dict(explicit_cons=True)),
    (18, 500, 64, "uplink", dict(n_types=2)),
    (19, 300, 100, "random", dict(dur_hi=1 << 32)),
    (20, 600, 256, "pair", dict(explicit_cons=True)),
    (21, 400, 256, None, dict(bytes_hi=1 << 20, n_types=3)),
])
def test_random_dags_bit_exact(seed, n, D, links, kw):
    d, rows = _case(seed, n, D, links, **kw)
    _run_and_compare(d, rows, trace=(0, 5, rows.shape[0] - 1) if rows.shape[0] > 5 else (0,))


@pytest.mark.parametrize("seed", range(6))
def test_zero_length_transfers(seed):
    d, rows = _case(40 + seed, 120, 6 if seed < 4 else 48, "pair" if seed % 2 else None, zero=True, dur_hi=9)
    _run_and_compare(d, rows, trace=(0, 1, 2))


def test_hand_worked_conflicts():
    cases = [
        (mk([[], [0], [0]], [4, 1, 1], out_bytes=[10, 0, 0], n_dev=3, bw=1, lat=0), [0, 1, 2]),
        (mk([[], [], [0, 1]], [3, 3, 2], out_bytes=[5, 7, 0], n_dev=3, bw=1, lat=0), [0, 1, 2]),
        (mk([[], [], [], [0], [1], [2]], [1] * 6, out_bytes=[100, 5, 5, 0, 0, 0], n_dev=4, bw=1, lat=0),
         [0, 2, 2, 1, 1, 3]),
        (mk([[], [], [0], [1]], [1, 1, 1, 1], out_bytes=[10, 10, 0, 0], n_dev=2, bw=1, lat=0,
            cons=[[], [3], [], []], cap=[19, 15]), [0, 0, 1, 1]),
    ]
    link = mk([[], [], [0], [1]], [2, 2, 1, 1], out_bytes=[6, 6, 0, 0], n_dev=2, bw=1, lat=0)
    link.link_id = np.array([0, 1, 1, 0], np.int32)
    cases.append((link, [0, 1, 1, 0]))
    for d, place in cases:
        rows = np.zeros((3, 16), np.uint8)
        rows[:, :len(place)] = place
        rows[1, :len(place)] = [(x + 1) % d.n_dev for x in place]
        _run_and_compare(d, rows, trace=(0, 1, 2))


@pytest.mark.parametrize("cfg", [2, 6])
def test_workloads_every_candidate(cfg):
    """The prefill (8 requests x 32 layers, 8 accelerators) and
    heterogeneous-prefill workloads, all 4,096 candidates, arbitrated."""
    wl = W.make_workload(cfg)
    rows = wl.all_full_rows()
    g = G.gmg_create(wl.desc)
    out = G.sim_batch(g, torch_place(rows), arbitrated=True)
    torch.cuda.synchronize()
    s, pk, rq = O.simulate_batch(wl.desc, rows, arbitrated=True)
    compare(out.to_numpy(), s, pk)
    assert (s["status"] == 0).all()


def test_incremental_workload_graph_all_candidates():
    """The 32 x 32-layer graph on 16 accelerators, its base placement with
    each candidate's moves applied, arbitrated as full placements."""
    wl = W.make_workload(3)
    K = wl.moves.off.shape[0] - 1
    rows = np.zeros((K, wl.ld), np.uint8)
    rows[:, :wl.desc.n_ops] = wl.base_place[:wl.desc.n_ops]
    for k in range(K):
        a, b = wl.moves.off[k], wl.moves.off[k + 1]
        rows[k, wl.moves.op[a:b]] = wl.moves.dev[a:b]
    g = G.gmg_create(wl.desc)
    out = G.sim_batch(g, torch_place(rows), arbitrated=True)
    torch.cuda.synchronize()
    s, pk, _ = O.simulate_batch(wl.desc, rows, arbitrated=True)
    compare(out.to_numpy(), s, pk)


def test_noalloc_equals_scratch_path():
    d, rows = _case(60, 300, 8, "pair")
    g = G.gmg_create(d)
    a = G.sim_batch(g, torch_place(rows), arbitrated=True)
    b = G.sim_batch_noalloc(g, torch_place(rows), arbitrated=True)
    torch.cuda.synchronize()
    ga, gb = a.to_numpy(), b.to_numpy()
    for k in ga:
        if ga[k] is not None:
            assert np.array_equal(ga[k], gb[k]), k


def test_degenerate_inputs_and_refusals():
    # bad device ids, a queue too small, an empty graph
    d, rows = _case(70, 60, 4, None)
    rows[3, 17] = 4
    g = G.gmg_create(d)
    out = G.sim_batch(g, torch_place(rows), arbitrated=True)
    torch.cuda.synchronize()
    s, pk, _ = O.simulate_batch(d, rows, arbitrated=True)
    compare(out.to_numpy(), s, pk)
    assert out.to_numpy()["status"][3] == G.SIM_BADDEV
    # a star: 120 successors ready at once overflow a 3-entry READY queue
    n = 121
    star = mk([[]] + [[0]] * 120, [5] * n, [1] * n, n_dev=4, bw=1, lat=1)
    gs = G.gmg_create(star)
    srows = np.zeros((8, 128), np.uint8)
    srows[:, :n] = np.random.default_rng(0).integers(0, 4, (8, n))
    small = G.sim_batch(gs, torch_place(srows), arbitrated=True, queue_cap=3)
    full = G.sim_batch(gs, torch_place(srows), arbitrated=True)
    torch.cuda.synchronize()
    assert (small.to_numpy()["status"] == G.SIM_QUEUE).all()
    s, pk, _ = O.simulate_batch(star, srows, arbitrated=True)
    compare(full.to_numpy(), s, pk)
    empty = mk([], [], n_dev=3)
    ge = G.gmg_create(empty)
    out = G.sim_batch(ge, torch_place(np.zeros((4, 16), np.uint8)), arbitrated=True)
    torch.cuda.synchronize()
    e = out.to_numpy()
    assert (e["status"] == 0).all() and (e["score"] == 0).all() and (e["makespan"] == 0).all()
    # times so wide that an accelerator id no longer fits beside the key
    dw, rw = _case(11, 150, 4, None, dur_hi=1 << 40, link_hetero=False)
    with pytest.raises(G.GmgError) as ei:
        G.sim_batch(G.gmg_create(dw), torch_place(rw), arbitrated=True)
    assert ei.value.code == G.GMG_ERANGE
    # an arbitrated base snapshot also keeps the arbiter's checkpoints
    o = G._opts(arbitrated=True)
    import ctypes as C
    assert G.lib().inc_scratch_bytes(g.handle, 4, C.addressof(o)) > 0
    assert G.lib().base_workspace_bytes(g.handle, C.addressof(o)) > 0


def test_decode_memtight_full_size_sampled():
    """The memory-tight decode workload at full size (8 tenants x 64 steps x
    32 layers, N = 197,632 ops, D = 8, all 8,192 placements in one launch as
    bench.py runs it), arbitrated; 40 sampled candidates checked against the
    oracle one by one, every candidate's status checked."""
    wl = W.make_workload(4)
    rows = wl.all_full_rows()
    g = G.gmg_create(wl.desc)
    out = G.sim_batch(g, torch_place(rows), arbitrated=True)
    torch.cuda.synchronize()
    got = out.to_numpy()
    assert (got["status"] == G.SIM_OK).all()
    ks = np.unique(np.concatenate([[0, 1, rows.shape[0] - 1],
                                   np.random.default_rng(4).integers(0, rows.shape[0], 37)]))
    s, pk, _ = O.simulate_batch(wl.desc, rows[ks], arbitrated=True)
    compare({k: (None if v is None else v[ks]) for k, v in got.items()}, s, pk)


def _inc_compare(d, base_place, mv, **kw):
    g = G.gmg_create(d)
    b = G.base_create(g, torch.from_numpy(np.ascontiguousarray(base_place[:d.n_ops])).cuda())
    off, op, dv = G.moves_to_device(mv, "cuda")
    out = G.sim_incremental(g, b, off, op, dv, req_done=True, arbitrated=True, **kw)
    torch.cuda.synchronize()
    s, pk, rq = O.incremental_batch(d, base_place[:d.n_ops], mv, arbitrated=True)
    compare(out.to_numpy(), s, pk, rq)
    return out.to_numpy(), s


@pytest.mark.parametrize("seed,n,D,links", [(80, 60, 3, None), (81, 300, 8, "pair"), (82, 500, 16, "uplink"),
                                            (83, 200, 32, "random"), (85, 300, 48, "pair"), (86, 400, 256, None)])
def test_incremental_candidates_bit_exact(seed, n, D, links):
    """Move lists against a base placement, arbitrated: each candidate is the
    full arbitrated simulation of its moved placement (events = n), and
    malformed move lists get the same status codes as without arbitration."""
    d, rows = _case(seed, n, D, links)
    base = rows[0, :n].copy()
    mv = W.random_moves(seed, 64, base, D, max_moves=12)
    if D < 256:
        mv.dev[mv.off[3]] = D                       # a device out of range
    else:
        mv.op[mv.off[3]] = n                        # an op out of range
    if mv.off[8] - mv.off[7] > 1:
        mv.op[mv.off[7] + 1] = mv.op[mv.off[7]]     # an op moved twice
    got, s = _inc_compare(d, base, mv)
    assert got["status"][3] == G.SIM_MOVE_RANGE
    assert (got["events"][got["status"] == 0] == n).all()


def test_incremental_workload_moves_and_a_bad_base():
    """The incremental workload's 16,384 move lists (32 x 32-layer graph, 16
    accelerators) through sim_incremental, arbitrated, every candidate; then
    a base placement with a device out of range (every candidate BADBASE)."""
    wl = W.make_workload(3)
    _inc_compare(wl.desc, wl.base_place, wl.moves)
    d, rows = _case(84, 40, 3, None)
    bad = rows[0, :40].copy()
    bad[5] = 7
    mv = W.random_moves(84, 8, rows[0, :40].copy(), 3, max_moves=4)
    got, s = _inc_compare(d, bad, mv)
    assert (got["status"] == G.SIM_BADBASE).all()


def test_large_workload_subset_256_accelerators():
    """The first 256 placements of the 256-accelerator workload (128 tenants,
    N = 213,568 ops), arbitrated; 8 of them checked against the oracle."""
    wl = W.make_workload(5)
    rows = wl.full_rows(range(256))
    g = G.gmg_create(wl.desc)
    out = G.sim_batch(g, torch_place(rows), arbitrated=True)
    torch.cuda.synchronize()
    got = out.to_numpy()
    assert (got["status"] == G.SIM_OK).all()
    ks = np.array([0, 1, 37, 100, 128, 200, 254, 255])
    s, pk, _ = O.simulate_batch(wl.desc, rows[ks], arbitrated=True)
    compare({k: (None if v is None else v[ks]) for k, v in got.items()}, s, pk)


def test_incremental_arbitrated_ignores_a_base_queue_limit():
    """A base snapshot whose own pure-latency run stopped at a queue limit
    (queue_cap=2 on a graph with 120 successors of one op) cannot serve
    resumed candidates (pure latency: every candidate BADBASE), but the
    arbitrated candidates are full simulations of their moved rows and equal
    the oracle's."""
    n = 121
    d = mk([[]] + [[0]] * 120, [5] * n, [1 << 10] * n, n_dev=4, bw=100, lat=1)
    base = np.random.default_rng(3).integers(0, 4, n).astype(np.uint8)
    mv = W.random_moves(3, 16, base, 4, max_moves=6)
    g = G.gmg_create(d)
    b = G.base_create(g, torch.from_numpy(base).cuda(), queue_cap=2)
    off, op, dv = G.moves_to_device(mv, "cuda")
    lat = G.sim_incremental(g, b, off, op, dv)
    arb = G.sim_incremental(g, b, off, op, dv, req_done=True, arbitrated=True)
    torch.cuda.synchronize()
    st = lat.status.cpu().numpy()
    assert (st == G.SIM_BADBASE).all()
    s, pk, rq = O.incremental_batch(d, base, mv, arbitrated=True)
    compare(arb.to_numpy(), s, pk, rq)
    assert (arb.status.cpu().numpy() == 0).all()


# ---------------------------------------------------------------------------
# Incremental candidates resumed from an arbitrated base snapshot
# ---------------------------------------------------------------------------

def _resumed(d, base_place, mv, **kw):
    g = G.gmg_create(d)
    b = G.base_create(g, torch.from_numpy(np.ascontiguousarray(base_place[:d.n_ops])).cuda(), arbitrated=True)
    off, op, dv = G.moves_to_device(mv, "cuda")
    out = G.sim_incremental(g, b, off, op, dv, req_done=True, arbitrated=True, **kw)
    torch.cuda.synchronize()
    s, pk, rq = O.incremental_batch(d, base_place[:d.n_ops], mv, arbitrated=True, resumed=True)
    got = out.to_numpy()
    compare(got, s, pk, rq)
    return got, s


@pytest.mark.parametrize("seed,n,D,links,kw", [
    (90, 60, 3, None, {}),
    (91, 300, 8, "pair", {}),
    (92, 500, 16, "uplink", dict(explicit_cons=True)),
    (93, 400, 32, "random", {}),
    (94, 300, 6, None, dict(n_types=2)),
    (95, 300, 8, "pair", dict(dur_hi=1 << 31)),   # times beyond 2^31: 64-bit instances
    (96, 250, 5, None, dict(zero=True)),
])
def test_resumed_candidates_bit_exact(seed, n, D, links, kw):
    """Move lists against an arbitrated base snapshot: each candidate resumes
    at the latest checkpoint before its T0 -- the arbiter's queues, holds and
    FIFOs restored, a moved op's inputs recounted, its predecessors' remote
    sets, holds and FIFO places repaired -- and equals the full arbitrated
    simulation of its moved placement; events counts the ops with arbitrated
    base ready time >= T0."""
    zero = kw.pop("zero", False)
    d, rows = _case(seed, n, D, links, zero=zero, **kw)
    base = rows[0, :n].copy()
    mv = W.random_moves(seed, 96, base, D, max_moves=8)
    mv.dev[mv.off[3]] = D                            # a device out of range
    got, s = _resumed(d, base, mv)
    ok = got["status"] == 0
    assert got["status"][3] == G.SIM_MOVE_RANGE
    assert (got["events"][ok] < n).mean() > 0.5


def test_resumed_workload_every_candidate():
    """All 16,384 move lists of the incremental workload (32 x 32-layer
    graph, 16 accelerators) resumed from its arbitrated base."""
    wl = W.make_workload(3)
    got, s = _resumed(wl.desc, wl.base_place, wl.moves)
    assert (got["status"] == 0).all()
    assert got["events"].mean() < 0.9 * wl.desc.n_ops


def test_arbitrated_base_serves_arbitrated_candidates_only():
    d, rows = _case(97, 80, 4, None)
    base = rows[0, :80].copy()
    mv = W.random_moves(97, 8, base, 4, max_moves=3)
    g = G.gmg_create(d)
    b = G.base_create(g, torch.from_numpy(base).cuda(), arbitrated=True)
    off, op, dv = G.moves_to_device(mv, "cuda")
    with pytest.raises(G.GmgError) as e:
        G.sim_incremental(g, b, off, op, dv)
    assert e.value.code == G.GMG_EINVAL
    wide = W.random_desc(98, 60, 40)
    with pytest.raises(G.GmgError):
        G.base_create(G.gmg_create(wide), torch.zeros(64, dtype=torch.uint8, device="cuda"), arbitrated=True)
