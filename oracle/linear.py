"""Masking, masked product, correction and unmask (oracle side).

Sec. 3.3.1 ("Offloading Linear Operations") and Eq. add-and-then-subtract:
the TEE forms the masked input x~ = x + eta, the GPU returns r = W x~, and
the TEE recovers W x = r - W eta, where W eta (the "correction") is
precomputed (Sec. 5.2).  In exact arithmetic the result is exactly W x.

Conventions: rows are tokens.  X is [M, K], W is [N, K] (the nn.Linear
layout, footnote on PyTorch's transposed storage in Sec. 2.2.3), results
are [M, N]; the paper's column-vector W x is the same product transposed.
Products are evaluated in fp64 from fp32 inputs (every product of two fp32
numbers is exact in fp64), which is the plain definition to within
K * 2^-53 relative to sum |w||x|.  The two elementwise steps (mask and
unmask) are single fp32 operations in the paper's working precision
(binary32, Sec. 4.5.1); evaluating them in fp64 and rounding once to fp32
gives the correctly rounded fp32 result, because 53 >= 2*24 + 2 makes the
double rounding innocuous (Figueroa, "When is double rounding innocuous?",
SIGNUM 1995).
"""

import numpy as np


def _f64(a):
    return np.asarray(a, dtype=np.float32).astype(np.float64)


def mask(X, N):
    """x~ = fl32(x + eta) elementwise (Sec. 3.3.1)."""
    return (_f64(X) + _f64(N)).astype(np.float32)


def mask_f64(X, N):
    """x~ = fl64(x + eta), the mask in binary64 (Sec. 5.5): one rounding of at most 2^-53 |x~|."""
    return _f64(X) + _f64(N)


def matmul_exact(A, W):
    """A W^T in fp64 for fp32 A [M, K] and W [N, K] (the plain definition of the product)."""
    return _f64(A) @ _f64(W).T


def masked_linear(Xt, W):
    """r = W x~ for every row of X~ (what the GPU computes, Sec. 5.1), in fp64."""
    return matmul_exact(Xt, W)


def precompute_noise_product(N, W):
    """The correction W eta for every row of N (Sec. 5.2), in fp64.

    Rows of N may stack several independent noise draws; each row is
    handled independently, so a batch [draws*M, K] is the same definition.
    """
    return matmul_exact(N, W)


def unmask(Yt, C):
    """W x = r - W eta (Eq. add-and-then-subtract), one fp32 subtraction per element."""
    return (_f64(Yt) - _f64(C)).astype(np.float32)


def reference_output(X, W):
    """The unmasked target W x (exact, fp64): what unmask(masked_linear) reaches in R."""
    return matmul_exact(X, W)


def abs_products(X, Xt, N, W):
    """The three |w|-weighted sums of Thm. 4 for every output element.

    S_x = <|w|, |x|>, S_xt = <|w|, |x~|>, S_n = <|w|, |eta|>, each [M, N] fp64.
    """
    Wa = np.abs(_f64(W))
    return (np.abs(_f64(X)) @ Wa.T, np.abs(_f64(Xt)) @ Wa.T, np.abs(_f64(N)) @ Wa.T)


def max_relative_error(Y, Yref):
    """max |Y - Yref| / max |Yref| (matrix max-norm relative error)."""
    Y = np.asarray(Y, dtype=np.float64)
    Yref = np.asarray(Yref, dtype=np.float64)
    denom = np.max(np.abs(Yref)) if Yref.size else 0.0
    if denom == 0.0:
        return float(np.max(np.abs(Y))) if Y.size else 0.0
    return float(np.max(np.abs(Y - Yref)) / denom)
