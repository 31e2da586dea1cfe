"""Pins of the oracle's least-squares calibration of the batch-time coefficients (Sec. 4.1)."""
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2607_18253_gb300 import workloads as W

COEF = np.array([[4e-3, 5e-5, 5e-5, 1.5e-7, 9e-9],
                 [8e-3, 1.2e-4, 1.2e-4, 3.7e-7, 2.3e-8],
                 [3e-3, 7e-5, 9e-5, 2e-7, 1e-8]])


def test_noiseless_logs_give_the_coefficients_back():
    F, m, t = W.batch_log(5000, 3, seed=1, coef=COEF, noise=0.0)
    got = oracle.calibrate(F, m, t, 3, shared_beta1=False)
    np.testing.assert_allclose(got, COEF, rtol=1e-7)
    # the four-coefficient form recovers models whose beta1p == beta1d
    got4 = oracle.calibrate(F, m, t, 3, shared_beta1=True)
    np.testing.assert_allclose(got4[:2], COEF[:2], rtol=1e-7)


def _exact_normal_equations(X, y):
    # Gaussian elimination in rationals on X^T X beta = X^T y
    n = X.shape[1]
    A = [[sum(Fraction(X[r, i]) * Fraction(X[r, j]) for r in range(X.shape[0])) for j in range(n)] for i in range(n)]
    b = [sum(Fraction(X[r, i]) * Fraction(y[r]) for r in range(X.shape[0])) for i in range(n)]
    for c in range(n):
        piv = next(r for r in range(c, n) if A[r][c] != 0)
        A[c], A[piv] = A[piv], A[c]
        b[c], b[piv] = b[piv], b[c]
        for r in range(n):
            if r != c and A[r][c] != 0:
                f = A[r][c] / A[c][c]
                A[r] = [a - f * cc for a, cc in zip(A[r], A[c])]
                b[r] -= f * b[c]
    return [float(b[i] / A[i][i]) for i in range(n)]


def test_matches_exact_rational_least_squares():
    F, m, t = W.batch_log(40, 1, seed=2, coef=COEF[:1], noise=0.05)
    got = oracle.calibrate(F, m, t, 1, shared_beta1=False)[0]
    exact = _exact_normal_equations(F.astype(np.float64), t)
    np.testing.assert_allclose(got, exact, rtol=1e-8)
    X = np.stack([F[:, 0], F[:, 1] + F[:, 2], F[:, 3], F[:, 4]], axis=1).astype(np.float64)
    got4 = oracle.calibrate(F, m, t, 1, shared_beta1=True)[0]
    exact4 = _exact_normal_equations(X, t)
    np.testing.assert_allclose(got4[[0, 1, 3, 4]], exact4, rtol=1e-8)
    assert got4[1] == got4[2]


def test_residual_is_orthogonal_to_the_regressors():
    F, m, t = W.batch_log(20000, 2, seed=3, coef=COEF[:2], noise=0.04)
    got = oracle.calibrate(F, m, t, 2, shared_beta1=False)
    for k in range(2):
        X = F[m == k].astype(np.float64)
        r = t[m == k] - X @ got[k]
        scale = np.abs(X).max(axis=0) * np.abs(t[m == k]).max() * X.shape[0]
        assert np.all(np.abs(X.T @ r) <= 1e-9 * scale)
    # with 4% noise the fitted batch times land near the generating model's
    for k in range(2):
        X = F[m == k].astype(np.float64)
        pred, true = X @ got[k], X @ COEF[k]
        assert np.sqrt(np.mean(((pred - true) / true) ** 2)) < 0.01


def test_underdetermined_models_are_nan():
    F, m, t = W.batch_log(100, 2, seed=4, coef=COEF[:2], noise=0.0)
    m = m.copy()
    m[:] = 0
    m[:3] = 1  # model 1: three rows for five unknowns
    got = oracle.calibrate(F, m, t, 3, shared_beta1=False)
    assert np.all(np.isfinite(got[0])) and np.all(np.isnan(got[1])) and np.all(np.isnan(got[2]))
