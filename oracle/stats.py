"""Kolmogorov-Smirnov statistic against the closed-form noise CDFs.

Used to check that the noise has the law the mechanism prescribes: the
Gaussian N(0, sigma^2) with sigma = Delta f / eps (Prop. eps-GDP mechanism,
Sec. 4.4) or the Laplace alternative with scale b = Delta f / eps.
"""

import math

import numpy as np


def laplace_cdf(x, b):
    """F(x) = 1/2 e^{x/b} for x < 0 and 1 - 1/2 e^{-x/b} for x >= 0."""
    x = np.asarray(x, dtype=np.float64)
    return np.where(x < 0, 0.5 * np.exp(np.minimum(x, 0.0) / b), 1.0 - 0.5 * np.exp(-np.maximum(x, 0.0) / b))


def normal_cdf(x, sigma):
    """F(x) = 1/2 erfc(-x / (sigma sqrt 2))."""
    x = np.asarray(x, dtype=np.float64)
    return 0.5 * np.vectorize(math.erfc)(-x / (sigma * math.sqrt(2.0)))


def ks_statistic(samples, cdf):
    """D_n = sup_x |F_n(x) - F(x)| for the empirical CDF F_n of ``samples``."""
    x = np.sort(np.asarray(samples, dtype=np.float64).ravel())
    n = x.size
    F = cdf(x)
    i = np.arange(1, n + 1, dtype=np.float64)
    return float(max(np.max(i / n - F), np.max(F - (i - 1) / n)))


def ks_critical(n, alpha=0.001):
    """Large-n critical value c(alpha)/sqrt(n), c(alpha) = sqrt(-ln(alpha/2)/2)."""
    return math.sqrt(-math.log(alpha / 2.0) / 2.0) / math.sqrt(n)
