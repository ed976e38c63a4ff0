"""Pins for the oracle's mask / masked product / correction / unmask (CPU only).

* brute force with exact rationals on tiny shapes (non-square, so a
  transposed operand fails);
* the identity of Eq. add-and-then-subtract, exactly, on inputs whose
  masked sums are exact;
* zero noise reduces to the plain product;
* the two elementwise steps are correctly rounded binary32 operations.
"""

from fractions import Fraction

import numpy as np
import pytest

from oracle import linear


def _exact_matmul(A, W):
    M, K = A.shape
    N = W.shape[0]
    return [[sum(Fraction(float(A[m, k])) * Fraction(float(W[n, k])) for k in range(K)) for n in range(N)]
            for m in range(M)]


@pytest.mark.parametrize("M,K,N", [(1, 1, 1), (2, 3, 5), (3, 8, 2), (5, 7, 4)])
def test_product_brute_force(M, K, N):
    rng = np.random.default_rng(M * 100 + K * 10 + N)
    A = rng.standard_normal((M, K)).astype(np.float32)
    W = rng.standard_normal((N, K)).astype(np.float32)
    got = linear.masked_linear(A, W)
    assert got.shape == (M, N)
    exact = _exact_matmul(A, W)
    for m in range(M):
        for n in range(N):
            ref = float(exact[m][n])
            scale = float(sum(abs(Fraction(float(A[m, k])) * Fraction(float(W[n, k]))) for k in range(K)))
            assert abs(got[m, n] - ref) <= 4 * K * 2.0 ** -53 * scale


def test_add_then_subtract_identity_exact():
    # integer-valued fp32 operands: x + eta and every product/sum are exact
    rng = np.random.default_rng(3)
    X = rng.integers(-50, 50, (6, 12)).astype(np.float32)
    Nz = rng.integers(-1000, 1000, (6, 12)).astype(np.float32)
    W = rng.integers(-9, 9, (7, 12)).astype(np.float32)
    Xt = linear.mask(X, Nz)
    assert np.array_equal(Xt.astype(np.float64), X.astype(np.float64) + Nz.astype(np.float64))
    r = linear.masked_linear(Xt, W)
    C = linear.precompute_noise_product(Nz, W)
    np.testing.assert_array_equal(r - C, linear.reference_output(X, W))
    Y = linear.unmask(r.astype(np.float32), C.astype(np.float32))
    np.testing.assert_array_equal(Y.astype(np.float64), linear.reference_output(X, W))


def test_zero_noise_reduces_to_plain_product():
    rng = np.random.default_rng(4)
    X = rng.standard_normal((4, 33)).astype(np.float32)
    W = rng.standard_normal((9, 33)).astype(np.float32)
    Z = np.zeros_like(X)
    Xt = linear.mask(X, Z)
    assert np.array_equal(Xt, X)
    assert np.array_equal(linear.precompute_noise_product(Z, W), np.zeros((4, 9)))
    np.testing.assert_array_equal(linear.masked_linear(Xt, W), linear.reference_output(X, W))


def test_elementwise_steps_round_to_nearest_even():
    one = np.float32(1.0)
    # 1 + 2^-24 is a tie between 1 and 1 + 2^-23: even wins
    assert linear.mask(np.array([one]), np.array([np.float32(2.0 ** -24)]))[0] == one
    # 1 + 3*2^-24 is a tie between 1+2^-23 and 1+2^-22: the even one is 1 + 2^-22
    assert linear.mask(np.array([one]), np.array([np.float32(3 * 2.0 ** -24)]))[0] == np.float32(1 + 2.0 ** -22)
    # just above the tie rounds up
    v = linear.mask(np.array([one]), np.array([np.float32(2.0 ** -24 + 2.0 ** -40)]))[0]
    assert v == np.float32(1 + 2.0 ** -23)
    # unmask: 2^24 + 1 - 0 rounds (tie) to 2^24
    assert linear.unmask(np.array([16777216.0]), np.array([-1.0]))[0] == np.float32(16777216.0)
    assert linear.unmask(np.array([3.0]), np.array([3.0]))[0] == 0.0


def test_max_relative_error_definition():
    Y = np.array([[1.0, 2.0], [3.0, -4.0]])
    Yr = np.array([[1.0, 2.5], [3.0, -4.0]])
    assert linear.max_relative_error(Y, Yr) == pytest.approx(0.5 / 4.0)
    assert linear.max_relative_error(np.zeros((0, 3)), np.zeros((0, 3))) == 0.0


def test_binary64_mask_rounds_once():
    """The binary64 mask of Sec. 5.5 is x + eta rounded once to binary64 (within half an ulp of the
    exact rational sum), 2^29 times finer than the binary32 mask, which loses x almost entirely
    when eta is 10^8 times larger."""
    g = np.random.default_rng(5)
    x = g.standard_normal(2000).astype(np.float32)
    eta = (g.standard_normal(2000) * 2.6e8).astype(np.float32)
    xt = linear.mask_f64(x, eta)
    assert xt.dtype == np.float64
    for a, b, s in zip(x[:300], eta[:300], xt[:300]):
        exact = Fraction(float(a)) + Fraction(float(b))
        assert abs(Fraction(float(s)) - exact) <= Fraction(np.spacing(abs(float(s)))) / 2
    assert np.max(np.abs(xt - eta.astype(np.float64) - x)) <= 2.0 ** -53 * np.max(np.abs(xt))
    assert np.max(np.abs(linear.mask(x, eta).astype(np.float64) - eta.astype(np.float64) - x)) > 1.0
