"""Pins for the oracle's sensitivity bounds (CPU only).

* ||W||_2 by power iteration against numpy's SVD (a library routine);
* Prop. z-standard-norm: ||x^||_2 = sqrt(d) after RMS normalisation;
* Thm. 1 closed form for alpha = 1 (2 d^(3/4)) and the printed dimensions;
* Thms. 1-3 dominate ||f(x) - f(y)|| for random and adversarial pairs,
  with f written out from Eqs. ln, att-mech-normalized and
  activation-function.
"""

import numpy as np
import pytest

from oracle import sensitivity as sens


@pytest.mark.parametrize("shape", [(5, 5), (7, 3), (3, 11), (64, 200)])
def test_spectral_norm_matches_svd(shape):
    rng = np.random.default_rng(sum(shape))
    W = rng.standard_normal(shape)
    assert sens.spectral_norm(W, iters=2000) == pytest.approx(np.linalg.svd(W, compute_uv=False)[0], rel=1e-6)


def test_rms_norm_has_norm_sqrt_d():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((10, 300)) * 7 + 1
    np.testing.assert_allclose(np.linalg.norm(sens.rms_normalize(x), axis=1), np.sqrt(300), rtol=1e-12)
    assert np.all(np.linalg.norm(sens.rms_normalize(x, 1e-3), axis=1) <= np.sqrt(300))


def test_thm1_closed_form_alpha_one():
    for d in (256, 2560, 3072):
        assert sens.delta_layernorm(np.ones(d)) == pytest.approx(2 * d ** 0.75, rel=1e-12)
    assert sens.delta_layernorm(np.ones(3072)) == pytest.approx(825.3, abs=0.05)
    assert sens.norm4([1.0, -1.0, 2.0]) == pytest.approx(18 ** 0.25)


def test_thm1_dominates_layernorm_differences():
    rng = np.random.default_rng(2)
    d = 64
    alpha = rng.standard_normal(d)
    beta = rng.standard_normal(d)
    bound = sens.delta_layernorm(alpha)
    worst = 0.0
    for _ in range(300):
        x, y = rng.standard_normal(d) * 10, rng.standard_normal(d)
        for yy in (y, -x):
            diff = np.linalg.norm(sens.layernorm(x, alpha, beta) - sens.layernorm(yy, alpha, beta))
            worst = max(worst, diff)
    assert worst <= bound
    # the bound is attained up to Cauchy-Schwarz slack: alpha = 1, y = -x gives 2 sqrt(d) vs 2 d^(3/4)
    x = rng.standard_normal(d)
    one = np.ones(d)
    diff = np.linalg.norm(sens.layernorm(x, one, None) - sens.layernorm(-x, one, None))
    assert diff == pytest.approx(2 * np.sqrt(d), rel=1e-12) and diff <= sens.delta_layernorm(one)


def _attention(x_seq, W_val, alpha, beta, probs):
    """Eq. att-mech-normalized: W_val beta + sum_i p_i W_val (alpha (.) x^_i)."""
    xh = sens.rms_normalize(x_seq)
    return W_val @ beta + sum(p * (W_val @ (alpha * xi)) for p, xi in zip(probs, xh))


def test_thm2_dominates_attention_differences():
    rng = np.random.default_rng(3)
    d, n = 48, 6
    alpha, beta = rng.standard_normal(d), rng.standard_normal(d)
    W_val = rng.standard_normal((d, d)) * 0.3
    bound = sens.delta_attention(alpha, sens.spectral_norm(W_val, iters=3000))
    for _ in range(200):
        xs, ys = rng.standard_normal((n, d)), rng.standard_normal((n, d))
        ys[1:] = xs[1:]  # neighbouring: one token differs
        p = rng.dirichlet(np.ones(n))
        q = rng.dirichlet(np.ones(n))
        diff = np.linalg.norm(_attention(xs, W_val, alpha, beta, p) - _attention(ys, W_val, alpha, beta, q))
        assert diff <= bound


def _activation(x, W_up, W_gate, alpha, beta):
    """Eq. activation-function: W_up LN(x) (.) W_gate LN(x) (.) sig(W_gate LN(x))."""
    ln = sens.layernorm(x, alpha, beta)
    g = W_gate @ ln
    return (W_up @ ln) * g / (1.0 + np.exp(-g))


def test_thm3_dominates_activation_differences_with_dff_reading():
    rng = np.random.default_rng(4)
    d, d_ff = 16, 40
    alpha, beta = rng.standard_normal(d), 0.1 * rng.standard_normal(d)
    W_up = rng.standard_normal((d_ff, d)) * 0.2
    W_gate = rng.standard_normal((d_ff, d)) * 0.2
    bound = sens.delta_activation(alpha, beta, d_ff, sens.spectral_norm(W_up, iters=3000),
                                  sens.spectral_norm(W_gate, iters=3000))
    worst = 0.0
    for _ in range(500):
        x, y = rng.standard_normal(d), rng.standard_normal(d)
        worst = max(worst, np.linalg.norm(_activation(x, W_up, W_gate, alpha, beta)
                                          - _activation(y, W_up, W_gate, alpha, beta)))
    assert worst <= bound
    # d_ff enters as sqrt(d_ff): doubling d_ff scales the bound by sqrt(2)
    b2 = sens.delta_activation(alpha, beta, 2 * d_ff, 1.0, 1.0)
    b1 = sens.delta_activation(alpha, beta, d_ff, 1.0, 1.0)
    assert b2 / b1 == pytest.approx(np.sqrt(2), rel=1e-12)
