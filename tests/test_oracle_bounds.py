"""Pins for the oracle's error bounds (CPU only).

* gamma_n and u against the numbers the paper prints (golden fixture);
* Higham's dot-product bound and Thm. 4 must dominate the error of an
  actual binary32 evaluation (numpy float32 arithmetic, sequential order)
  on random and adversarial inputs;
* special cases where Thm. 4's right-hand side has a closed form
  (eta = 0; x = 0), which a dropped or swapped term fails.
"""

import math

import numpy as np
import pytest

from oracle import bounds, linear


def test_unit_roundoff_and_gamma_against_paper(golden):
    p32 = golden["binary32_precision"]["value"]
    p64 = golden["binary64_precision"]["value"]
    assert bounds.unit_roundoff(p32) == 2.0 ** -24
    d = 8192
    ratio = bounds.gamma(d, bounds.unit_roundoff(p32)) / bounds.gamma(d, bounds.unit_roundoff(p64))
    g = golden["gamma_ratio_fp32_over_fp64"]
    assert ratio == pytest.approx(g["value"], rel=g["rel_tol"])
    assert bounds.gamma(3, 0.1) == pytest.approx(0.3 / 0.7)
    with pytest.raises(ValueError):
        bounds.gamma(10, 0.1)
    assert bounds.log_index(3072) == 13 and bounds.log_index(4096) == 13 and bounds.log_index(2) == 2


def _exact_dots(W, X):
    return np.sum(W.astype(np.float64) * X.astype(np.float64), axis=1)  # exact enough: K*2^-53


@pytest.mark.parametrize("dot", [bounds.dot_fp32_sequential, bounds.dot_fp32_pairwise])
def test_higham_dot_bound_dominates_fp32(dot):
    rng = np.random.default_rng(0)
    T, d = 2000, 512
    W = rng.standard_normal((T, d)).astype(np.float32)
    X = rng.standard_normal((T, d)).astype(np.float32)
    # adversarial rows: huge cancelling terms
    X[:100, ::2] *= 1e6
    X[:100, 1::2] = -X[:100, ::2] * W[:100, ::2] / np.where(W[:100, 1::2] == 0, 1, W[:100, 1::2])
    fl = dot(W, X).astype(np.float64)
    S = np.sum(np.abs(W.astype(np.float64) * X.astype(np.float64)), axis=1)
    assert np.all(np.abs(fl - _exact_dots(W, X)) <= bounds.dot_bound(S, d))


@pytest.mark.parametrize("eps", [0.1, 1.0, 10.0, float("inf")])
def test_thm4_dominates_fp32_cancellation(eps):
    rng = np.random.default_rng(int(0 if math.isinf(eps) else eps * 10))
    T, d = 3000, 256
    W = (0.02 * rng.standard_normal((T, d))).astype(np.float32)
    X = rng.standard_normal((T, d))
    X = (X / np.sqrt(np.mean(X * X, axis=1, keepdims=True))).astype(np.float32)
    b = 0.0 if math.isinf(eps) else 2 * d ** 0.75 / eps
    Nz = (b * rng.laplace(size=(T, d))).astype(np.float32)
    err, Xt = bounds.cancellation_error_fp32(W, X, Nz)
    S_x, S_xt, S_n = bounds.rowwise_abs_sums(W, X, Xt, Nz)
    assert np.all(err <= bounds.thm4_bound(S_x, S_xt, S_n, d) + 1e-30)
    # against the exact <w, x> the mask rounding enters; hard_bound covers it
    exact = _exact_dots(W, X)
    rec = (bounds.dot_fp32_sequential(W, Xt) - bounds.dot_fp32_sequential(W, Nz)).astype(np.float64)
    assert np.all(np.abs(rec - exact) <= bounds.hard_bound(S_x, S_xt, S_n, d))


def test_thm4_closed_forms():
    u = 2.0 ** -24
    d = 100
    g = d * u / (1 - d * u)
    # eta = 0: x~ = x, S_xt = S_x, S_n = 0  ->  2 gamma_d S_x + u S_x
    assert bounds.thm4_bound(3.0, 3.0, 0.0, d) == pytest.approx(2 * g * 3.0 + u * 3.0, rel=1e-15)
    # x = 0: x~ = eta, S_x = 0, S_xt = S_n  ->  2 gamma_d S_n
    assert bounds.thm4_bound(0.0, 5.0, 5.0, d) == pytest.approx(2 * g * 5.0, rel=1e-15)
    # Eq. fp-log-bound uses gamma_{ceil(log2 d)+1} = gamma_8 for d = 100
    g8 = 8 * u / (1 - 8 * u)
    assert bounds.log_bound(1.0, 2.0, 4.0, d) == pytest.approx(g8 * 7.0 + u * 1.0, rel=1e-15)
    # hard bound: Thm 4 plus the mask rounding and the second-order term
    hb = bounds.hard_bound(1.0, 2.0, 4.0, d)
    assert hb == pytest.approx(g * 7.0 + u + u * 2.0 * (1 + u) / (1 - u) + u * g * 7.0, rel=1e-15)


def test_thm4_worked_integer_example():
    # w = (1, 2), x = (1, -1), eta = (0.5, 0.5): |x| = (1,1), |x+eta| = (1.5, 0.5), |eta| = (0.5, 0.5)
    W = np.array([[1.0, 2.0]], dtype=np.float32)
    X = np.array([[1.0, -1.0]], dtype=np.float32)
    Nz = np.array([[0.5, 0.5]], dtype=np.float32)
    S_x, S_xt, S_n = linear.abs_products(X, linear.mask(X, Nz), Nz, W)
    assert (S_x[0, 0], S_xt[0, 0], S_n[0, 0]) == (3.0, 2.5, 1.5)


def test_statistics_fields():
    st = bounds.bound_statistics([1.0, 2.0, 10.0], [4.0, 4.0, 4.0])
    assert st["mean_error"] == pytest.approx(13 / 3)
    assert st["violation_pct"] == pytest.approx(100 / 3)
    assert st["max_err_over_bound"] == pytest.approx(2.5)


def test_log_bound_pattern_on_synthetic_inputs():
    """Sec. 6.3.2 methodology on synthetic inputs: the log bound is an estimate, not a bound.

    The paper sees bound/error near 4.3 and about 10% violations on captured
    activations.  Here only the qualitative facts are asserted: errors and
    bounds scale like 1/eps, and most elements stay under the estimate.
    """
    rng = np.random.default_rng(7)
    T, d = 4000, 3072
    W = (0.02 * rng.standard_normal((T, d))).astype(np.float32)
    X = rng.standard_normal((T, d))
    X = (X / np.sqrt(np.mean(X * X, axis=1, keepdims=True))).astype(np.float32)
    G = rng.standard_normal((T, d))
    stats = {}
    for eps in (1.0, 10.0):
        Nz = (2 * d ** 0.75 / eps * G).astype(np.float32)
        err, Xt = bounds.cancellation_error_fp32(W, X, Nz, dot=bounds.dot_fp32_pairwise)
        S = bounds.rowwise_abs_sums(W, X, Xt, Nz)
        stats[eps] = bounds.bound_statistics(err, bounds.log_bound(*S, d))
        assert stats[eps]["violation_pct"] < 50.0
        assert stats[eps]["ratio"] > 1.0
    assert 5 < stats[1.0]["mean_error"] / stats[10.0]["mean_error"] < 20
    assert 8 < stats[1.0]["mean_bound"] / stats[10.0]["mean_bound"] < 12
