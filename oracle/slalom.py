"""The Slalom comparator (Sec. 6.2), oracle side: exact integer arithmetic in numpy int64.

The paper compares its noise masking with Slalom's: inputs and weights are quantized to fixed
point with 8 fractional bits, the input is masked with a uniform element of the prime field
Z_q, q = 2^23 + 2^21 + 7, the GPU computes W_qt (x_qt + eta) mod q, the TEE subtracts the
precomputed W_qt eta mod q and de-quantizes the result (Sec. 6.2).  Readings (the paper names
the parameters, not the encoding):

* quantize: v_qt = rint(v 2^8), rounding half to even;
* mask element e: Philox block e // 2 + offset, words (2 (e % 2), 2 (e % 2) + 1) as the 64-bit
  integer lo + 2^32 hi, eta = that mod q (bias below q / 2^64);
* x~_qt = (x_qt mod q + eta) mod q in [0, q);
* recovered y_qt = (W_qt x~_qt - W_qt eta) mod q, taken in (-q/2, q/2], and y = y_qt 2^-16.

Oracle: test infrastructure only; the CUDA path does not use it.
"""

import numpy as np

from . import philox

Q = 2 ** 23 + 2 ** 21 + 7  # Sec. 6.2
FRAC_BITS = 8


def quantize(v):
    """v_qt = rint(v 2^8) as int64 (round half to even)."""
    return np.rint(np.asarray(v, dtype=np.float64) * 2.0 ** FRAC_BITS).astype(np.int64)


def mask_noise(shape, seed, stream_id=0, offset=0):
    """Uniform elements of Z_q from the Philox stream (two words per element)."""
    n = int(np.prod(shape))
    blocks = philox.philox_blocks((n + 1) // 2, seed, stream_id, offset)  # [nb, 4] uint32
    words = blocks.reshape(-1, 2)[:n]                                      # (lo, hi) pairs in stream order
    v = words[:, 0].astype(object) + (words[:, 1].astype(object) << 32)
    return np.array([int(x) % Q for x in v], dtype=np.int64).reshape(shape)


def mask(X, eta):
    """x~_qt = (x_qt mod q + eta) mod q."""
    return (np.mod(quantize(X), Q) + eta) % Q


def product(A_qt, W_qt):
    """The exact integer product A_qt W_qt^T (int64; inputs below 2^24 and 2^8, K below 2^13)."""
    return A_qt.astype(np.int64) @ W_qt.astype(np.int64).T


def unmask(r, c):
    """y = ((r - c) mod q) in (-q/2, q/2], de-quantized by 2^-16."""
    y = np.mod(r - c, Q)
    y = np.where(y > (Q - 1) // 2, y - Q, y)
    return y.astype(np.float64) * 2.0 ** (-2 * FRAC_BITS)


def masked_linear(X, W, eta):
    """The whole comparator: quantize, mask, product, correction, unmask, de-quantize."""
    W_qt = quantize(W)
    r = product(mask(X, eta), W_qt) % Q
    c = product(eta, W_qt) % Q
    return unmask(r, c)
