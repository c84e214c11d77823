"""sim_batch_noalloc: the variant of sim_batch for callers that cannot
allocate device memory (its scratch is a fixed buffer inside the library).
Its results must equal sim_batch's on consecutive calls, which also shows
that leftovers of one call in the shared buffer do not leak into the next,
and the oracle's, bit for bit."""
import ctypes as C

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_common import compare  # noqa: E402
from oracle import oracle as O  # noqa: E402
from paper_2608_15762_gb300 import gmgsim as G  # noqa: E402
from paper_2608_15762_gb300 import workloads as W  # noqa: E402

pytestmark = pytest.mark.gpu

FIELDS = ("status", "makespan", "score", "viol_flag", "viol_op", "viol_dev", "viol_time", "peak",
          "sla_miss", "events", "req_done", "trace_start", "trace_finish")


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_15762_gb300 import build
    build.build()
    assert torch.cuda.is_available()


def _rows(seed, K, n, D):
    g = np.random.default_rng(seed)
    rows = np.zeros((K, W.placement_ld(n)), np.uint8)
    rows[:, :n] = g.integers(0, D, (K, n))
    return torch.from_numpy(rows).cuda()


@pytest.mark.parametrize("which", ["tiny", "random"])
def test_same_results_as_sim_batch_on_two_calls(which):
    if which == "tiny":
        wl = W.config1()
        desc = wl.desc
        batches = [torch.from_numpy(wl.all_full_rows()).cuda(), _rows(9, 300, desc.n_ops, desc.n_dev)]
    else:
        desc = W.random_desc(21, 700, 40, explicit_cons=True)
        batches = [_rows(1, 257, 700, 40), _rows(2, 128, 700, 40)]
    g = G.gmg_create(desc)
    for place in batches:
        tk = torch.tensor([0, place.shape[0] - 1], dtype=torch.int32, device="cuda")
        ref = G.sim_batch(g, place, req_done=True, trace_k=tk)
        got = G.sim_batch_noalloc(g, place, req_done=True, trace_k=tk)
        torch.cuda.synchronize()
        a, b = ref.to_numpy(), got.to_numpy()
        for f in FIELDS:
            assert np.array_equal(a[f], b[f]), f
        s, pk, rq = O.simulate_batch(desc, place.cpu().numpy())
        compare(b, s, pk, rq)


def _compare_calls(g, desc, batches, arbitrated=False, **kw):
    for place in batches:
        tk = torch.tensor([0, place.shape[0] - 1], dtype=torch.int32, device="cuda")
        ref = G.sim_batch(g, place, req_done=True, trace_k=tk, arbitrated=arbitrated, **kw)
        got = G.sim_batch_noalloc(g, place, req_done=True, trace_k=tk, arbitrated=arbitrated, **kw)
        torch.cuda.synchronize()
        a, b = ref.to_numpy(), got.to_numpy()
        for f in FIELDS:
            assert np.array_equal(a[f], b[f]), f
        s, pk, rq = O.simulate_batch(desc, place.cpu().numpy(), arbitrated=arbitrated)
        compare(b, s, pk, rq)


def test_arbitrated_transfers_on_two_calls():
    """Arbitrated transfers (Sec. 3.5.2) through the fixed buffer: on 8 and on
    40 accelerators (the two arbitrated kernels)."""
    for D in (8, 40):
        desc = W.random_desc(23 + D, 400, D)
        _compare_calls(G.gmg_create(desc), desc, [_rows(3, 97, 400, D), _rows(4, 33, 400, D)], arbitrated=True)


def _chain(n, D, seed):
    """A chain of n ops (each op feeds the next) with random sizes."""
    g = np.random.default_rng(seed)
    pred_off = np.arange(n + 1, dtype=np.int32) - 1
    pred_off[0] = 0
    return W.GmgDesc(n_dev=D, pred_off=pred_off, pred_idx=np.arange(n - 1, dtype=np.int32),
                     dur=g.integers(1, 50, n).astype(np.int64), out_bytes=g.integers(0, 1 << 12, n).astype(np.int64),
                     release=np.zeros(n, np.int64), req_id=np.full(n, -1, np.int32),
                     scored=np.ones(n, np.uint8), deadline=np.zeros(0, np.int64),
                     cap=np.full(D, 1 << 40, np.int64), base=np.zeros(D, np.int64),
                     avail0=np.zeros(D, np.int64), bw=np.full(D * D, 7, np.int64),
                     lat=np.full(D * D, 2, np.int64)).normalized()


def test_fewer_slots_than_the_grid():
    """A graph whose warp slot is about 1 MB: the fixed buffer holds a few
    dozen slots, fewer than sim_batch's grid, so each warp takes several
    candidates in turn."""
    n = 60_000
    desc = _chain(n, 3, 5)
    g = G.gmg_create(desc)
    slot = G.sim_scratch_bytes(g, 1) // 4          # one block of 4 warps for one candidate
    assert 4 * slot <= _noalloc_bytes() < G.sim_scratch_bytes(g, 4096)
    _compare_calls(g, desc, [_rows(5, 211, n, 3), _rows(6, 64, n, 3)])


def test_one_warp_blocks_when_four_slots_do_not_fit():
    """A graph whose warp slot is about 13 MB: fewer than four slots fit, so
    the call re-plans with one-warp blocks."""
    n = 800_000
    desc = _chain(n, 2, 7)
    g = G.gmg_create(desc)
    slot = G.sim_scratch_bytes(g, 1) // 4
    assert slot <= _noalloc_bytes() < 4 * slot
    _compare_calls(g, desc, [_rows(7, 6, n, 2), _rows(8, 3, n, 2)])


def _noalloc_bytes():
    """GMG_NOALLOC_SCRATCH_BYTES as include/gmgsim.h defines it."""
    import os
    import re
    hdr = os.path.join(os.path.dirname(__file__), "..", "include", "gmgsim.h")
    m = re.search(r"#define GMG_NOALLOC_SCRATCH_BYTES \(\(size_t\)(\d+) << (\d+)\)", open(hdr).read())
    return int(m.group(1)) << int(m.group(2))


def test_refuses_a_graph_whose_scratch_does_not_fit():
    n = 5 << 20   # a chain whose one-warp scratch (a finish time per op, ...) exceeds 32 MiB
    pred_off = np.arange(n + 1, dtype=np.int32) - 1
    pred_off[0] = 0
    desc = W.GmgDesc(n_dev=2, pred_off=pred_off, pred_idx=np.arange(n - 1, dtype=np.int32),
                     dur=np.ones(n, np.int64), out_bytes=np.ones(n, np.int64),
                     release=np.zeros(n, np.int64), req_id=np.full(n, -1, np.int32),
                     scored=np.ones(n, np.uint8), deadline=np.zeros(0, np.int64),
                     cap=np.full(2, 1 << 40, np.int64), base=np.zeros(2, np.int64),
                     avail0=np.zeros(2, np.int64), bw=np.ones(4, np.int64),
                     lat=np.zeros(4, np.int64)).normalized()
    g = G.gmg_create(desc)
    assert G.sim_scratch_bytes(g, 1) > _noalloc_bytes()
    place = torch.zeros((1, W.placement_ld(n)), dtype=torch.uint8, device="cuda")
    out = G.SimOut.empty(1, 2, 0, place.device)
    co = out._c()
    o = G._opts()
    rc = G.lib().sim_batch_noalloc(g.handle, place.data_ptr(), 1, place.shape[1], C.addressof(o),
                                   C.addressof(co), None)
    assert rc == G.GMG_EWS
