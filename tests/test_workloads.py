"""The seeded synthetic workloads have the stated shapes and are reproducible."""
import numpy as np
import pytest

from paper_2608_15762_gb300 import workloads as W


@pytest.mark.parametrize("c,n,e,d,r,k", [
    (1, 50, 57, 2, 1, 256),
    (2, 3088, 8 * (14 * 32 + 1), 8, 8, 4096),
])
def test_prefill_shapes(c, n, e, d, r, k):
    wl = W.make_workload(c)
    assert (wl.desc.n_ops, wl.desc.n_edges, wl.desc.n_dev, wl.desc.n_req, wl.n_full) == (n, e, d, r, k)
    rows = wl.full_rows([0, k - 1])
    assert rows.shape == (2, wl.ld) and wl.ld % 16 == 0
    assert rows[:, :n].max() < d


def test_topological_and_deterministic():
    a, b = W.config2(), W.config2()
    for f in ("pred_off", "pred_idx", "dur", "out_bytes", "deadline"):
        assert np.array_equal(getattr(a.desc, f), getattr(b.desc, f))
    n = a.desc.n_ops
    for i in range(n):
        ps = a.desc.pred_idx[a.desc.pred_off[i]:a.desc.pred_off[i + 1]]
        assert (ps < i).all() and (np.diff(ps) > 0).all()
    assert np.array_equal(a.full_rows([17]), b.full_rows([17]))
    assert not np.array_equal(a.full_rows([17]), a.full_rows([18]))
    assert a.desc.dur.min() >= 5 and a.desc.dur.max() <= 50000
    assert a.desc.out_bytes.min() >= W.MiB and a.desc.out_bytes.max() <= 256 * W.MiB


def test_incremental_workload():
    wl = W.config3(n_cand=64)
    d = wl.desc
    assert (d.n_ops, d.n_dev, d.n_req) == (12352, 16, 32)
    mv = wl.moves
    assert mv.n_cand == 64
    cnt = np.diff(mv.off)
    assert cnt.min() >= 1 and cnt.max() <= 16
    assert (mv.op >= 16 * 386).all()                    # only offline ops move
    assert (mv.dev != wl.base_place[mv.op]).all()
    for k in range(64):
        ops = mv.op[mv.off[k]:mv.off[k + 1]]
        assert len(set(ops.tolist())) == len(ops)
    assert (d.release > 0).sum() == 16 * 3             # 3 released segments per online request


def test_decode_workload_kv_growth():
    wl = W.config4(cap=1 << 40, n_cand=4)
    d = wl.desc
    assert (d.n_ops, d.n_dev, d.n_req) == (197632, 8, 8)
    t = W.decode_template(32, 64)
    kv = np.flatnonzero(t.kind == W.LAYER_OPS.index("kvw"))
    b = d.out_bytes[:t.n][kv]
    step = t.step[kv]
    assert (b % (step + 1) == 0).all() and len(set((b // (step + 1)).tolist())) == 1


def test_large_workload():
    wl = W.config5(n_cand=128)
    d = wl.desc
    assert d.n_dev == 256 and 150_000 < d.n_ops < 260_000
    assert wl.n_full == 64 and wl.moves.n_cand == 64
    cnt = np.diff(wl.moves.off)
    assert cnt.min() >= 1 and cnt.max() <= 64
    assert (wl.moves.dev != wl.base_place[wl.moves.op]).all()
    assert d.release.max() < 750_000
