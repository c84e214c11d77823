"""GPU parity of the online estimators (include/gmgest.h) against the oracle:
coefficients after every online batch (fp64 normal equations against
numpy's least squares: relative 1e-7), fitted flags exactly, integer
durations and link tables exactly (a rounding that falls within 1e-6 of a
half integer may differ by one: the two fits differ in the last bits)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_common import compare, oracle_rows, torch_place  # noqa: E402
from oracle import estimators as OE  # noqa: E402
from oracle import oracle as O  # noqa: E402
from paper_2608_15762_gb300 import gmgsim as G  # noqa: E402
from paper_2608_15762_gb300 import workloads as W  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_15762_gb300 import build
    build.build()
    assert torch.cuda.is_available()


def _batch(g, counts, F, beta_true):
    off = np.zeros(len(counts) + 1, np.int32)
    off[1:] = np.cumsum(counts)
    S = int(off[-1])
    x = g.uniform(0, 10, (S, F))
    if F > 1:
        x[:, -1] = 1.0                                       # constant term
    e_of = np.repeat(np.arange(len(counts)), counts)
    y = np.einsum("sf,sf->s", x, beta_true[e_of]) + g.normal(0, 1.0, S)
    return off, x, y


def _dev(a, dt):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=dt)).cuda()


def _close(got, want):
    return np.all(np.abs(got - want) <= 1e-7 * (np.abs(want) + 1e-3 * np.abs(want).max() + 1e-12))


@pytest.mark.parametrize("F", range(1, 9))
def test_online_batches_match_least_squares(F):
    g = np.random.default_rng(100 + F)
    E = 13
    beta_true = g.uniform(-5, 50, (E, F))
    est = G.Estimators(E, F)
    orc = OE.EstimatorsOracle(E, F)
    for b in range(3):
        counts = g.integers(0, 400, E)
        counts[0] = 0                                        # never any sample
        counts[1] = 1 if b == 0 else 0                       # fewer than F (for F > 1)
        counts[2] = 5000 if b == 1 else 3
        off, x, y = _batch(g, counts, F, beta_true)
        est.update(_dev(off, np.int32), _dev(x, np.float64), _dev(y, np.float64))
        orc.update(off, x, y)
        beta, fitted = est.coefficients()
        torch.cuda.synchronize()
        ob, of = orc.coefficients()
        assert fitted.cpu().numpy().tolist() == of.tolist(), b
        assert _close(beta.cpu().numpy(), ob), b


def test_rank_deficient_estimator_is_not_fitted():
    g = np.random.default_rng(7)
    off = np.array([0, 50, 100], np.int32)
    x = g.uniform(0, 10, (100, 4))
    x[50:, 3] = 3.0 * x[50:, 1]                              # estimator 1: dependent columns
    y = g.uniform(0, 100, 100)
    est = G.Estimators(2, 4)
    est.update(_dev(off, np.int32), _dev(x, np.float64), _dev(y, np.float64))
    _, fitted = est.coefficients()
    assert fitted.cpu().tolist() == [1, 0]


def test_updates_are_reproducible_bit_for_bit():
    g = np.random.default_rng(8)
    off, x, y = _batch(g, [3000, 17, 0, 800], 5, g.uniform(0, 9, (4, 5)))
    outs = []
    for _ in range(2):
        est = G.Estimators(4, 5)
        est.update(_dev(off, np.int32), _dev(x, np.float64), _dev(y, np.float64))
        outs.append(est.coefficients()[0].cpu().numpy())
    assert np.array_equal(outs[0], outs[1])


def _predict_both(est, orc, est_of, x, dflt):
    d = est.predict_durations(_dev(est_of, np.int32), _dev(x, np.float64), _dev(dflt, np.int64)).cpu().numpy()
    ob, of = orc.coefficients()
    od = OE.predict_durations(ob, of, est_of, x, dflt)
    return d, od, ob, of


def test_predicted_durations_and_links():
    g = np.random.default_rng(9)
    T, K, F = 2, 14, 5                                       # types x template operators
    E = T * K
    beta_true = g.uniform(1, 40, (E, F))
    est, orc = G.Estimators(E, F), OE.EstimatorsOracle(E, F)
    counts = g.integers(20, 300, E)
    counts[5] = 2                                            # not fitted: defaults
    off, x, y = _batch(g, counts, F, beta_true)
    est.update(_dev(off, np.int32), _dev(x, np.float64), _dev(y, np.float64))
    orc.update(off, x, y)
    n = 5000
    kind = g.integers(0, K, n)
    est_of = np.stack([t * K + kind for t in range(T)], axis=1)
    est_of[::97, 1] = -1                                     # no estimator
    xo = g.uniform(0, 10, (n, F))
    xo[:, -1] = 1.0
    dflt = g.integers(1, 1000, n)
    d, od, ob, of = _predict_both(est, orc, est_of, xo, dflt)
    bad = np.argwhere(d != od)
    for i, t in bad:
        v = float(np.dot(ob[est_of[i, t]], xo[i]))
        assert abs(abs(v - np.floor(v)) - 0.5) < 1e-6 and abs(int(d[i, t]) - int(od[i, t])) == 1
    assert (d[:, 1][::97] == dflt[::97]).all()
    # transfer estimators: features (size, 1)
    D = 6
    tr, to = G.Estimators(D * D, 2), OE.EstimatorsOracle(D * D, 2)
    counts = g.integers(30, 200, D * D)
    counts[7] = 0
    off = np.zeros(D * D + 1, np.int32)
    off[1:] = np.cumsum(counts)
    size = g.uniform(1e5, 3e8, off[-1])
    q = np.repeat(np.arange(D * D), counts)
    inv_bw = 1.0 / g.integers(50_000, 400_000, D * D)
    yy = size * inv_bw[q] + (5 + q % 7) + g.normal(0, 0.3, off[-1])
    xx = np.stack([size, np.ones_like(size)], axis=1)
    tr.update(_dev(off, np.int32), _dev(xx, np.float64), _dev(yy, np.float64))
    to.update(off, xx, yy)
    bwd, latd = np.full(D * D, 400_000), np.full(D * D, 10)
    bw, lat = tr.links(D, _dev(bwd, np.int64), _dev(latd, np.int64))
    ob, of = to.coefficients()
    obw, olat = OE.links(ob, of, D, bwd, latd)
    assert bw.cpu().numpy().tolist() == obw.tolist() and lat.cpu().numpy().tolist() == olat.tolist()


def test_fitted_durations_drive_the_simulation():
    """Feedback -> per-(type, operator) estimators -> durations -> the typed
    what-if simulation, against the oracle fed the oracle's durations."""
    g = np.random.default_rng(10)
    base = W.random_desc(31, 240, 6, dur_hi=300, n_types=2)
    K, F, T = 12, 3, 2
    kind = g.integers(0, K, base.n_ops)
    xo = np.stack([g.uniform(0, 10, base.n_ops), g.uniform(0, 10, base.n_ops), np.ones(base.n_ops)], axis=1)
    beta_true = g.uniform(2, 30, (T * K, F))
    est, orc = G.Estimators(T * K, F), OE.EstimatorsOracle(T * K, F)
    off, x, y = _batch(g, g.integers(10, 60, T * K), F, beta_true)
    est.update(_dev(off, np.int32), _dev(x, np.float64), _dev(y, np.float64))
    orc.update(off, x, y)
    est_of = np.stack([t * K + kind for t in range(T)], axis=1)
    d, od, _, _ = _predict_both(est, orc, est_of, xo, base.dur)
    assert np.array_equal(d, od)
    import dataclasses
    desc = dataclasses.replace(base, dur_by_type=d).normalized()
    rows = np.zeros((64, W.placement_ld(base.n_ops)), np.uint8)
    rows[:, :base.n_ops] = g.integers(0, 6, (64, base.n_ops))
    out = G.sim_batch(G.gmg_create(desc), torch_place(rows), req_done=True)
    torch.cuda.synchronize()
    s, pk, rq = oracle_rows(dataclasses.replace(base, dur_by_type=od).normalized(), rows)
    compare(out.to_numpy(), s, pk, rq)


def test_empty_batches_one_type_and_one_accelerator():
    est, orc = G.Estimators(3, 2), OE.EstimatorsOracle(3, 2)
    off = np.zeros(4, np.int32)
    est.update(_dev(off, np.int32), torch.zeros((0, 2), dtype=torch.float64, device="cuda"),
               torch.zeros(0, dtype=torch.float64, device="cuda"))
    beta, fitted = est.coefficients()
    assert fitted.cpu().tolist() == [0, 0, 0] and not beta.cpu().numpy().any()
    g = np.random.default_rng(12)
    o2, x, y = _batch(g, [40, 0, 9], 2, g.uniform(1, 9, (3, 2)))
    est.update(_dev(o2, np.int32), _dev(x, np.float64), _dev(y, np.float64))
    orc.update(o2, x, y)
    est_of = np.array([[0], [1], [2], [-1]], np.int32)         # one accelerator type
    xo = np.stack([g.uniform(0, 10, 4), np.ones(4)], axis=1)
    d, od, _, _ = _predict_both(est, orc, est_of, xo, np.array([5, 6, 7, 8]))
    assert np.array_equal(d, od) and d[1, 0] == 6 and d[3, 0] == 8
    tr = G.Estimators(1, 2)                                     # one accelerator: only the diagonal
    bw, lat = tr.links(1, _dev(np.array([9]), np.int64), _dev(np.array([4]), np.int64))
    assert bw.cpu().tolist() == [9] and lat.cpu().tolist() == [4]
