"""Global l2 sensitivities of the functions feeding each offloaded projection.

Sec. 4.3 bounds Delta f (Def. global-sensitivity) for:

* Thm. 1 (input of Q, K, V, Gate, Up and the LM head, after LayerNorm or
  RMSNorm):           Delta LN  <= 2 sqrt(d) ||alpha||_4
* Thm. 2 (input of O, after attention):
                      Delta att <= 2 sqrt(d) ||W_val||_2 ||alpha||_4
* Thm. 3 (input of Down, after the SiLU-gated activation):
                      Delta act <= 2 sqrt(d) (sqrt(d) ||alpha||_4 + ||beta||_2)^2
                                   ||W_up||_2 ||W_gate||_2

||W||_2 is the spectral norm (largest singular value, Eq. matrix-norm).
Sec. 4.3 says to substitute the dimension that applies to each operation.
Reading taken for Thm. 3: the leading sqrt(d) comes from ||sig(g(x))||_2 <=
sqrt(dim g(x)), so it is sqrt(d_ff); the inner sqrt(d) ||alpha||_4 bounds
||LN(x)||_2 and uses the model dimension d.
"""

import numpy as np


def norm4(alpha):
    """||alpha||_4 = (sum alpha_i^4)^(1/4)."""
    a = np.asarray(alpha, dtype=np.float64)
    return float(np.sum(a ** 4) ** 0.25)


def delta_layernorm(alpha):
    """Thm. 1: 2 sqrt(d) ||alpha||_4 with d = len(alpha)."""
    d = np.asarray(alpha).size
    return 2.0 * np.sqrt(d) * norm4(alpha)


def delta_attention(alpha, wval_norm2):
    """Thm. 2: 2 sqrt(d) ||W_val||_2 ||alpha||_4."""
    d = np.asarray(alpha).size
    return 2.0 * np.sqrt(d) * float(wval_norm2) * norm4(alpha)


def delta_activation(alpha, beta, d_ff, wup_norm2, wgate_norm2):
    """Thm. 3 with the dimension reading above: 2 sqrt(d_ff) (sqrt(d)||alpha||_4 + ||beta||_2)^2 ||W_up|| ||W_gate||."""
    d = np.asarray(alpha).size
    beta_norm = float(np.linalg.norm(np.asarray(beta, dtype=np.float64))) if beta is not None else 0.0
    ln_bound = np.sqrt(d) * norm4(alpha) + beta_norm
    return 2.0 * np.sqrt(d_ff) * ln_bound ** 2 * float(wup_norm2) * float(wgate_norm2)


def spectral_norm(W, iters=200, seed=0, tol=1e-12):
    """||W||_2 by power iteration on W^T W in fp64 (returns sqrt of the top eigenvalue)."""
    W = np.asarray(W, dtype=np.float64)
    rng = np.random.default_rng(seed)
    v = rng.standard_normal(W.shape[1])
    v /= np.linalg.norm(v)
    sigma = 0.0
    for _ in range(iters):
        u = W @ v
        s_new = np.linalg.norm(u)
        if s_new == 0.0:
            return 0.0
        v = W.T @ (u / s_new)
        v /= np.linalg.norm(v)
        if abs(s_new - sigma) <= tol * s_new:
            sigma = s_new
            break
        sigma = s_new
    return float(np.linalg.norm(W @ v))


def rms_normalize(x, gamma_eps=0.0):
    """RMS normalisation of each row (Def. normalization with mu = 0)."""
    x = np.asarray(x, dtype=np.float64)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + gamma_eps)


def layernorm(x, alpha, beta, gamma_eps=0.0, rms=True):
    """LN(x) = alpha (.) x^ + beta (Eq. ln) with x^ z-score or RMS normalised."""
    x = np.asarray(x, dtype=np.float64)
    if not rms:
        x = x - x.mean(axis=-1, keepdims=True)
    return np.asarray(alpha) * rms_normalize(x, gamma_eps) + (0.0 if beta is None else np.asarray(beta))
