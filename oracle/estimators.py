"""CPU oracle of the online linear estimators (Sec. 3.3.1).

TEST INFRASTRUCTURE ONLY: the plain definition the GPU estimators are
checked against.  Only the test suite, the smoke check and the benchmark's
CPU-baseline leg use it; the product never imports it.

What it computes:

* Transfer estimator per accelerator pair, t = alpha * size + c, and operator
  estimator per (accelerator type, template operator), t = sum_j beta_j x_j
  over shape-derived features (Sec. 3.3.1).  Both are linear models fitted
  to executor feedback.
* "Incorporated online": an estimator's coefficients are the least-squares
  fit over every sample it has received so far, beta = argmin ||X beta - y||^2
  (numpy.linalg.lstsq on the stacked samples).  An estimator is fitted once
  it has at least F samples and X has full column rank (numpy's matrix_rank);
  otherwise its coefficients are 0 and it is not used.
* Durations for the simulation: clamp(rint(beta_e . x_i), 1, 2^40) for op i on
  a type whose estimator e is fitted, else the op's default duration; rint
  rounds halves to even (numpy.rint).
* Link tables from transfer estimators with features (size, 1):
  bw = clamp(rint(1 / alpha), 1, 2^40) (2^40 when alpha <= 0),
  lat = clamp(rint(c), 0, 2^40); defaults where not fitted and on the diagonal.
"""
from __future__ import annotations

import numpy as np

MAX_TICKS = 1 << 40


class EstimatorsOracle:
    """n_est estimators of n_feat features; keeps every sample received."""

    def __init__(self, n_est: int, n_feat: int):
        self.n_est, self.n_feat = n_est, n_feat
        self.xs = [np.zeros((0, n_feat)) for _ in range(n_est)]
        self.ys = [np.zeros(0) for _ in range(n_est)]

    def update(self, off, x, y) -> None:
        """Samples in CSR form by estimator: rows off[e]..off[e+1] of x (S, F), y (S,)."""
        off = np.asarray(off)
        x = np.asarray(x, np.float64).reshape(-1, self.n_feat)
        y = np.asarray(y, np.float64)
        for e in range(self.n_est):
            a, b = int(off[e]), int(off[e + 1])
            if b > a:
                self.xs[e] = np.vstack([self.xs[e], x[a:b]])
                self.ys[e] = np.concatenate([self.ys[e], y[a:b]])

    def coefficients(self):
        beta = np.zeros((self.n_est, self.n_feat))
        fitted = np.zeros(self.n_est, np.int32)
        for e in range(self.n_est):
            X, y = self.xs[e], self.ys[e]
            if X.shape[0] >= self.n_feat and np.linalg.matrix_rank(X) == self.n_feat:
                beta[e] = np.linalg.lstsq(X, y, rcond=None)[0]
                fitted[e] = 1
        return beta, fitted


def clamp_rint(v: float, lo: int) -> int:
    r = np.rint(v)
    if not r >= lo:
        return lo
    if r >= MAX_TICKS:
        return MAX_TICKS
    return int(r)


def predict_durations(beta, fitted, est_of, x, dflt) -> np.ndarray:
    est_of = np.asarray(est_of)
    n_ops, n_types = est_of.shape
    out = np.zeros((n_ops, n_types), np.int64)
    for i in range(n_ops):
        for t in range(n_types):
            e = int(est_of[i, t])
            if e < 0 or not fitted[e]:
                out[i, t] = int(dflt[i])
            else:
                out[i, t] = clamp_rint(float(np.dot(beta[e], x[i])), 1)
    return out


def links(beta, fitted, n_dev, bw_dflt, lat_dflt):
    bw = np.array(bw_dflt, np.int64).copy()
    lat = np.array(lat_dflt, np.int64).copy()
    for d in range(n_dev):
        for e in range(n_dev):
            q = d * n_dev + e
            if d == e or not fitted[q]:
                continue
            alpha, c = float(beta[q][0]), float(beta[q][1])
            bw[q] = clamp_rint(1.0 / alpha, 1) if alpha > 0 else MAX_TICKS
            lat[q] = clamp_rint(c, 0)
    return bw, lat
