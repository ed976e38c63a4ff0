"""Floating-point cancellation bounds (Sec. 4.5) and fp32 dot-product emulation.

Notation follows Sec. 4.5: binary32 has precision p = 24 and unit round-off
u = 2^-p (Eq. ulp); gamma_d = d u / (1 - d u) (Def. u-and-theta); Higham's
dot-product bound |<w,x> - fl(<w,x>)| <= gamma_d <|w|,|x|> (Eq.
dot-product-bound).  Thm. 4 bounds the error of recovering <w,x> from the
masked product:

    |fl(<w,x>) - fl(fl(<w,x+eta>) - fl(<w,eta>))|
        <= gamma_d <|w|, |x| + |x+eta| + |eta|> + u <|w|,|x|> + O(d u^2),

and Eq. fp-log-bound replaces gamma_d by gamma_{ceil(log2 d)+1} (pairwise
summation, Higham Sec. 3.1 p. 64) as an empirical, tighter estimate.

Readings taken here (the paper treats x + eta as exact):
* S_xt uses the masked input actually sent, x~ = fl(x + eta).
* ``hard_bound`` adds the rounding of the mask itself (<= u <|w|,|x~|>) and
  writes the second-order term out instead of dropping it, so it bounds the
  recovered value against both the exact <w,x> and fl(<w,x>).
"""

import math

import numpy as np

P_BINARY32 = 24
P_BINARY64 = 53


def unit_roundoff(p=P_BINARY32):
    """u = 2^-p (Eq. ulp)."""
    return 2.0 ** (-p)


def gamma(n, u=None):
    """gamma_n = n u / (1 - n u) (Def. u-and-theta); requires n u < 1."""
    u = unit_roundoff() if u is None else u
    nu = n * u
    if nu >= 1.0:
        raise ValueError("gamma_n needs n*u < 1")
    return nu / (1.0 - nu)


def log_index(d):
    """ceil(log2 d) + 1, the gamma index of Eq. fp-log-bound."""
    return int(math.ceil(math.log2(d))) + 1


def thm4_bound(S_x, S_xt, S_n, d, u=None):
    """Right-hand side of Thm. 4 without the O(d u^2) term."""
    u = unit_roundoff() if u is None else u
    g = gamma(d, u)
    return g * (S_x + S_xt + S_n) + u * S_x


def hard_bound(S_x, S_xt, S_n, d, u=None):
    """Thm. 4 plus the mask rounding and the written-out second-order term.

    gamma_d (S_x + S_xt + S_n) + u S_x + u S_xt (1+u)/(1-u) + u gamma_d (S_x + S_xt + S_n).
    """
    u = unit_roundoff() if u is None else u
    g = gamma(d, u)
    return (thm4_bound(S_x, S_xt, S_n, d, u) + u * S_xt * (1.0 + u) / (1.0 - u)
            + u * g * (S_x + S_xt + S_n))


def log_bound(S_x, S_xt, S_n, d, u=None):
    """Eq. fp-log-bound: gamma_{ceil(log2 d)+1} (S_x + S_xt + S_n) + u S_x."""
    u = unit_roundoff() if u is None else u
    g = gamma(log_index(d), u)
    return g * (S_x + S_xt + S_n) + u * S_x


def dot_bound(S, d, u=None):
    """Higham's bound gamma_d <|w|,|x|> (Eq. dot-product-bound)."""
    return gamma(d, unit_roundoff() if u is None else u) * S


def dot_fp32_sequential(W, X):
    """fl(<w,x>) in binary32 with left-to-right recursive summation.

    W and X are [T, d] (T independent dot products).  Each product and each
    partial sum is rounded to fp32, i.e. the order the standard model of
    Eq. std-model is applied to in Higham's proof.
    """
    W = np.asarray(W, dtype=np.float32)
    X = np.asarray(X, dtype=np.float32)
    acc = np.zeros(W.shape[0], dtype=np.float32)
    for k in range(W.shape[1]):
        acc = acc + W[:, k] * X[:, k]  # both ops in float32 with RN
    return acc


def dot_fp32_pairwise(W, X):
    """fl(<w,x>) in binary32 with pairwise (cascade) summation of the fp32 products."""
    terms = np.asarray(W, dtype=np.float32) * np.asarray(X, dtype=np.float32)
    while terms.shape[1] > 1:
        if terms.shape[1] % 2:
            terms = np.concatenate([terms, np.zeros((terms.shape[0], 1), np.float32)], axis=1)
        terms = terms[:, 0::2] + terms[:, 1::2]
    return terms[:, 0]


def cancellation_error_fp32(W, X, N, dot=dot_fp32_sequential):
    """The quantity of Eq. fp-error, evaluated in binary32.

    |fl(<w,x>) - fl(fl(<w,x~>) - fl(<w,eta>))| for rows of W, X, N ([T, d]),
    with x~ = fl(x + eta).  The outer difference is exact (fp64), as the
    paper notes it is not a floating-point operation.
    """
    X = np.asarray(X, dtype=np.float32)
    N = np.asarray(N, dtype=np.float32)
    Xt = X + N
    A = dot(W, X)
    B = dot(W, Xt)
    C = dot(W, N)
    recovered = B - C  # one fp32 subtraction
    return np.abs(A.astype(np.float64) - recovered.astype(np.float64)), Xt


def rowwise_abs_sums(W, X, Xt, N):
    """Per-row S_x, S_xt, S_n for [T, d] operands (fp64)."""
    Wa = np.abs(np.asarray(W, dtype=np.float64))
    return (np.sum(Wa * np.abs(np.asarray(X, dtype=np.float64)), axis=1),
            np.sum(Wa * np.abs(np.asarray(Xt, dtype=np.float64)), axis=1),
            np.sum(Wa * np.abs(np.asarray(N, dtype=np.float64)), axis=1))


def bound_statistics(err, bound):
    """Mean error, mean bound, their ratio and the violation rate (Table numerical-error)."""
    err = np.asarray(err, dtype=np.float64).ravel()
    bound = np.asarray(bound, dtype=np.float64).ravel()
    me, mb = float(err.mean()), float(bound.mean())
    return {
        "mean_error": me,
        "mean_bound": mb,
        "ratio": (mb / me) if me > 0 else float("inf"),
        "violation_pct": 100.0 * float(np.mean(err > bound)),
        "max_err_over_bound": float(np.max(err / np.where(bound > 0, bound, np.inf))) if err.size else 0.0,
    }
