"""Pins of the estimator oracle (Sec. 3.3.1 linear transfer / operator
estimators fitted online by least squares) against what least squares and
the rounding rules fix."""
import numpy as np
import pytest

from oracle import estimators as E


def _csr(counts):
    off = np.zeros(len(counts) + 1, np.int32)
    off[1:] = np.cumsum(counts)
    return off


@pytest.mark.parametrize("F", [1, 2, 5, 8])
def test_noise_free_samples_recover_the_coefficients(F):
    g = np.random.default_rng(F)
    beta = g.uniform(-5, 50, F)
    x = g.uniform(0, 10, (60, F))
    est = E.EstimatorsOracle(1, F)
    est.update([0, 60], x, x @ beta)
    b, fitted = est.coefficients()
    assert fitted[0] == 1
    assert np.allclose(b[0], beta, rtol=1e-9, atol=1e-9)


def test_two_features_give_the_simple_regression_line():
    # features (size, 1): slope = cov(size, y) / var(size), intercept = mean(y) - slope mean(size)
    g = np.random.default_rng(3)
    size = g.uniform(0, 100, 40)
    y = 2.5 * size + 7 + g.normal(0, 3, 40)
    est = E.EstimatorsOracle(1, 2)
    est.update([0, 40], np.stack([size, np.ones(40)], axis=1), y)
    b, _ = est.coefficients()
    slope = ((size - size.mean()) * (y - y.mean())).sum() / ((size - size.mean()) ** 2).sum()
    assert np.isclose(b[0][0], slope, rtol=1e-12)
    assert np.isclose(b[0][1], y.mean() - slope * size.mean(), rtol=1e-12)


def test_residual_is_orthogonal_to_every_feature():
    g = np.random.default_rng(4)
    x = g.uniform(0, 10, (200, 5))
    y = x @ g.uniform(0, 9, 5) + g.normal(0, 2, 200)
    est = E.EstimatorsOracle(1, 5)
    est.update([0, 200], x, y)
    b, _ = est.coefficients()
    r = y - x @ b[0]
    assert np.abs(x.T @ r).max() < 1e-8 * np.abs(x.T @ y).max()


def test_batches_are_accumulated_per_estimator():
    g = np.random.default_rng(5)
    counts = [[3, 0, 9], [7, 4, 0], [0, 1, 2]]
    est = E.EstimatorsOracle(3, 2)
    allx = [[], [], []]
    ally = [[], [], []]
    for c in counts:
        x = g.uniform(0, 5, (sum(c), 2))
        y = g.uniform(0, 5, sum(c))
        est.update(_csr(c), x, y)
        off = _csr(c)
        for e in range(3):
            allx[e].append(x[off[e]:off[e + 1]])
            ally[e].append(y[off[e]:off[e + 1]])
    b, fitted = est.coefficients()
    for e in range(3):
        X, y = np.vstack(allx[e]), np.concatenate(ally[e])
        assert fitted[e] == 1
        assert np.allclose(b[e], np.linalg.lstsq(X, y, rcond=None)[0])


def test_too_few_samples_or_rank_deficient_is_not_fitted():
    g = np.random.default_rng(6)
    est = E.EstimatorsOracle(3, 3)
    x = g.uniform(0, 5, (2 + 10 + 10, 3))
    x[12:, 2] = x[12:, 0] * 2.0            # estimator 2: a column is a multiple of another
    est.update(_csr([2, 10, 10]), x, g.uniform(0, 9, 22))
    b, fitted = est.coefficients()
    assert fitted.tolist() == [0, 1, 0]
    assert not b[0].any() and not b[2].any()


def test_duration_rounding_and_fallbacks():
    beta = np.array([[1.0, 0.0], [1.0, 0.0]])
    fitted = np.array([1, 0])
    x = np.array([[2.5, 0], [3.5, 0], [-7.0, 0], [1e13, 0], [4.0, 0]])
    est_of = np.array([[0, 1], [0, -1], [0, 0], [0, 0], [1, 0]])
    d = E.predict_durations(beta, fitted, est_of, x, np.array([11, 12, 13, 14, 15]))
    # half to even; below 1 -> 1; above 2^40 -> 2^40; unfitted or -1 -> default
    assert d.tolist() == [[2, 11], [4, 12], [1, 1], [1 << 40, 1 << 40], [15, 4]]


def test_link_tables():
    D = 3
    beta = np.zeros((D * D, 2))
    fitted = np.zeros(D * D, np.int32)
    beta[1] = [1 / 400000, 10.4]      # 0 -> 1
    beta[5] = [0.0, -3.0]              # 1 -> 2: no size term, negative latency
    fitted[[1, 5, 4]] = 1              # 4 is the diagonal (1 -> 1): ignored
    bw, lat = E.links(beta, fitted, D, np.full(D * D, 7), np.full(D * D, 9))
    assert bw[1] == 400000 and lat[1] == 10
    assert bw[5] == 1 << 40 and lat[5] == 0
    assert bw[4] == 7 and lat[4] == 9 and bw[2] == 7 and lat[2] == 9
