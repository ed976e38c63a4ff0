"""Shared helpers of the GPU parity tests (tolerances written out here)."""

import numpy as np

from oracle import bounds, linear

U = 2.0 ** -24  # binary32 unit round-off (Eq. ulp)
# Per-term error of the three-product TF32 split: two truncated residual
# terms (2^-21 each) plus the dropped lo*lo term (2^-22), rounded up.
TF32X3_TERM = 3 * 2.0 ** -21
# Per-term error of the fp16 split (each operand row scaled by a power of two, hi and lo
# binary16 with 11 significant bits each): the residual of each operand is rounded once
# (2^-22 relative each) and lo*lo is dropped (2^-22), so 3 * 2^-22, rounded up to 2^-20.
# A residual below fp16's normal range is rounded to an absolute 2^-25 in the scaled
# units, at most 2^-39 of the row's largest entry: FP16X3_ABS.
FP16X3_TERM = 2.0 ** -20
FP16X3_ABS = 2.0 ** -38


def product_tolerance(S, K, path, A=None, W=None):
    """Max |GPU - exact| allowed for a K-term product with sum |a||w| = S.

    fp32: Higham's bound gamma_K S (Eq. dot-product-bound), valid for any
    summation order and for split-K partials summed afterwards.
    tf32x3 / fp16x3: the same plus the per-term split error; fp16x3 also the
    absolute term of residuals below fp16's normal range (needs A and W).
    """
    g = bounds.gamma(max(K, 1), U)
    if path == "fp32":
        return g * S
    if path == "tf32x3":
        return (g + TF32X3_TERM) * S
    a = np.abs(np.asarray(A, dtype=np.float64))
    w = np.abs(np.asarray(W, dtype=np.float64))
    floor = FP16X3_ABS * (a.max(axis=1)[:, None] * w.sum(axis=1)[None, :] +
                          a.sum(axis=1)[:, None] * w.max(axis=1)[None, :])
    return (g + FP16X3_TERM) * S + floor


def f64(t):
    return t.detach().double().cpu().numpy()


def f32(t):
    return t.detach().float().cpu().numpy()


def ulp32(x):
    x = np.abs(np.asarray(x, dtype=np.float32))
    return np.spacing(np.maximum(x, np.float32(np.finfo(np.float32).tiny))).astype(np.float64)


def assert_product_close(got, A, W, path, C=None, what=""):
    """got ~ A W^T (- C) within the product tolerance (elementwise)."""
    ref = linear.matmul_exact(A, W)
    S = np.abs(A.astype(np.float64)) @ np.abs(W.astype(np.float64)).T
    tol = product_tolerance(S, A.shape[1], path, A, W)
    if C is not None:
        ref = ref - C.astype(np.float64)
        tol = tol * (1 + 2 * U) + 2 * U * np.abs(ref)
    err = np.abs(got.astype(np.float64) - ref)
    bad = err > tol
    assert not bad.any(), (f"{what}: {int(bad.sum())} of {bad.size} outside tolerance; "
                           f"worst err/tol {float(np.max(err / np.maximum(tol, 1e-300))):.3g}")
    return float(np.max(err / np.maximum(tol, 1e-300))) if err.size else 0.0
