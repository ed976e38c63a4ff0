"""Pins for the oracle's noise law (CPU only).

The mechanism fixes the law: N(0, (Delta f/eps)^2) for the Gaussian
mechanism (Prop. eps-GDP mechanism, Sec. 4.4) and Laplace(0, Delta f/eps)
for the configured alternative.  Checked with a KS test on 10^6 samples
against the closed-form CDFs, the moments, and closed-form quantiles.
"""

import math

import numpy as np
import pytest

from oracle import philox, stats

N_KS = 10 ** 6


@pytest.mark.parametrize("sens,eps", [(2.0, 1.0), (825.3, 0.5), (1.0, 10.0)])
def test_laplace_law(sens, eps):
    eta = philox.noise((N_KS,), sens, eps, "laplace", seed=11, stream_id=3).astype(np.float64)
    b = float(np.float32(sens / eps))
    d = stats.ks_statistic(eta, lambda x: stats.laplace_cdf(x, b))
    assert d <= stats.ks_critical(N_KS, 0.001), d
    assert abs(eta.var() / (2 * b * b) - 1) < 0.01
    assert abs(eta.mean()) < 5 * math.sqrt(2) * b / math.sqrt(N_KS)
    # median of |eta| of Laplace(0, b) is b ln 2
    assert abs(np.median(np.abs(eta)) / (b * math.log(2)) - 1) < 0.01


@pytest.mark.parametrize("sens,eps", [(2.0, 1.0), (719.8, 0.1)])
def test_gaussian_law(sens, eps):
    eta = philox.noise((N_KS,), sens, eps, "gaussian", seed=5, stream_id=1).astype(np.float64)
    s = float(np.float32(sens / eps))
    d = stats.ks_statistic(eta, lambda x: stats.normal_cdf(x, s))
    assert d <= stats.ks_critical(N_KS, 0.001), d
    assert abs(eta.var() / (s * s) - 1) < 0.01
    assert abs(eta.mean()) < 5 * s / math.sqrt(N_KS)
    # the pair (a, b) of one Box-Muller draw lies on the circle of radius s R
    r = philox.radius_fp64((N_KS,), 5, 1)
    e64 = philox.noise((N_KS,), sens, eps, "gaussian", seed=5, stream_id=1, as_fp64=True)
    pairs = e64.reshape(-1, 2)
    np.testing.assert_allclose(np.hypot(pairs[:, 0], pairs[:, 1]), s * r.reshape(-1, 2)[:, 0], rtol=1e-12)


def test_gaussian_pairs_are_uncorrelated():
    e = philox.noise((400000,), 1.0, 1.0, "gaussian", seed=8, as_fp64=True).reshape(-1, 2)
    assert abs(np.corrcoef(e[:, 0], e[:, 1])[0, 1]) < 0.01
    q = philox.noise((400000,), 1.0, 1.0, "gaussian", seed=8, as_fp64=True).reshape(-1, 4)
    assert abs(np.corrcoef(q[:, 1], q[:, 2])[0, 1]) < 0.01


def test_ks_statistic_matches_scipy():
    scipy_stats = pytest.importorskip("scipy.stats")
    rng = np.random.default_rng(0)
    x = rng.laplace(0.0, 3.0, 5000)
    ours = stats.ks_statistic(x, lambda t: stats.laplace_cdf(t, 3.0))
    ref = scipy_stats.kstest(x, scipy_stats.laplace(scale=3.0).cdf).statistic
    assert abs(ours - ref) < 1e-12
    y = rng.normal(0.0, 2.0, 5000)
    ours = stats.ks_statistic(y, lambda t: stats.normal_cdf(t, 2.0))
    ref = scipy_stats.kstest(y, scipy_stats.norm(scale=2.0).cdf).statistic
    assert abs(ours - ref) < 1e-12


def test_ks_detects_wrong_scale():
    eta = philox.noise((200000,), 2.0, 1.0, "laplace", seed=1).astype(np.float64)
    d = stats.ks_statistic(eta, lambda x: stats.laplace_cdf(x, 2.0 * 1.05))
    assert d > stats.ks_critical(200000, 0.001)


def test_eps_infinity_gives_exact_zeros_and_bad_eps_rejected():
    for mech in ("laplace", "gaussian"):
        z = philox.noise((7, 9), 3.0, float("inf"), mech, seed=1)
        assert z.dtype == np.float32 and np.all(z == 0)
    for bad in (0.0, -1.0, float("nan")):
        with pytest.raises(ValueError):
            philox.noise((4,), 1.0, bad, "laplace", seed=0)
    with pytest.raises(ValueError):
        philox.noise((4,), -1.0, 1.0, "laplace", seed=0)


def test_laplace_extremes_closed_form():
    b = 2.0
    # m = 0xFFFFFF -> u = 1 -> eta = 0 ; m = 0 -> u = 2^-24 -> |eta| = 24 b ln 2; bit 31 is the sign
    words = np.array([0x00FFFFFF, 0x00000000, 0x80000000, 0x7F000000], dtype=np.uint32)
    eta = philox.laplace_from_words(words, b)
    assert eta[0] == 0.0
    assert eta[1] == pytest.approx(24 * b * math.log(2), rel=1e-15)
    assert eta[2] == pytest.approx(-24 * b * math.log(2), rel=1e-15)
    assert eta[3] == pytest.approx(24 * b * math.log(2), rel=1e-15)  # bits 24..30 are unused


def test_box_muller_closed_form():
    # r_a >> 8 = 2^24 - 1 -> u1 = 1 -> R = 0 ; r_b >> 8 = 2^22 -> u2 = 1/4 -> angle pi/2
    blk = np.array([[0xFFFFFFFF, 0x40000000, 0x00000000, 0x00000000]], dtype=np.uint32)
    g = philox.gaussian_from_blocks(blk, 3.0)
    assert g[0, 0] == 0.0 and g[0, 1] == 0.0
    R = math.sqrt(-2 * math.log(2.0 ** -24))
    assert g[0, 2] == pytest.approx(3.0 * R, rel=1e-15)  # u2 = 0 -> cos 0 = 1
    assert g[0, 3] == 0.0
