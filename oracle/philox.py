"""Philox4x32-10 and the noise transforms (oracle side, fp64).

The paper masks each offloaded input with noise drawn from the Gaussian
mechanism N(0, (Delta f / eps)^2 I) (Prop. "eps-GDP mechanism", Sec. 2.3;
Sec. 4.4 "Making the Process Differentially Private").  It does not say how
the random numbers are produced.  Both sides of this repository draw them
from the same published counter-based generator, Philox4x32 with 10 rounds
(Salmon, Moraes, Dror, Shaw, "Parallel Random Numbers: As Easy as 1, 2, 3",
SC'11, Sec. 3.3), each side from its own implementation.

Stream layout (shared definition, not shared code):

* element ``e`` of a flat tensor belongs to Philox block ``j = e // 4 + offset``
  (64-bit, wrapping) and uses lane ``e % 4`` of that block;
* the 128-bit counter is ``(lo32(j), hi32(j), lo32(stream_id), hi32(stream_id))``;
* the 64-bit key is ``(lo32(seed), hi32(seed))``.

Transforms (scale ``b = fl32(Delta / eps)``, rounded once on the host):

* Laplace (a configured alternative to the paper's Gaussian): one 32-bit word
  ``r`` per element; bit 31 is the sign, the low 24 bits ``m`` give
  ``u = (m + 1) 2^-24`` in ``(0, 1]`` and ``eta = +-b * (-ln u)``.  This is the
  inverse CDF of Laplace(0, b) split into its independent sign and magnitude.
* Gaussian (the paper's mechanism): Box-Muller on the word pairs (0, 1) and
  (2, 3) of a block: ``u1 = ((r_a >> 8) + 1) 2^-24`` in ``(0, 1]``,
  ``u2 = (r_b >> 8) 2^-24`` in ``[0, 1)``, ``R = sqrt(-2 ln u1)``; lane a gets
  ``b R cos(2 pi u2)`` and lane b gets ``b R sin(2 pi u2)``.
* ``eps = +inf`` gives ``b = 0`` and therefore ``eta = 0`` (the paper's
  noise-free T3 configuration, Table "configurations").
"""

import numpy as np

# Philox4x32 constants as published by Salmon et al. (SC'11, Sec. 3.3):
# the two round multipliers and the two Weyl key increments.
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
ROUNDS = 10
_MASK32 = np.uint64(0xFFFFFFFF)
TWO_M24 = 2.0 ** -24


def philox4x32_10(c0, c1, c2, c3, k0, k1):
    """Apply Philox4x32-10 to counter words (c0..c3) under key (k0, k1).

    One round multiplies counter word 0 by M0 and word 2 by M1 (full 64-bit
    products split into hi/lo halves) and forms the new state
    (hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0); the key is bumped by (W0, W1)
    between rounds.  Inputs are array-likes of integers < 2^32; the four
    outputs are uint32 arrays.
    """
    c0, c1, c2, c3 = (np.asarray(c, dtype=np.uint64) & _MASK32 for c in (c0, c1, c2, c3))
    k0 = np.asarray(k0, dtype=np.uint64) & _MASK32
    k1 = np.asarray(k1, dtype=np.uint64) & _MASK32
    m0, m1 = np.uint64(PHILOX_M0), np.uint64(PHILOX_M1)
    for rnd in range(ROUNDS):
        if rnd > 0:
            k0 = (k0 + np.uint64(PHILOX_W0)) & _MASK32
            k1 = (k1 + np.uint64(PHILOX_W1)) & _MASK32
        p0 = m0 * c0  # < 2^64, no wrap
        p1 = m1 * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & _MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & _MASK32
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return tuple(c.astype(np.uint32) for c in (c0, c1, c2, c3))


def philox_blocks(nblocks, seed, stream_id, offset):
    """Return the uint32 words of Philox blocks offset .. offset+nblocks-1 as [nblocks, 4]."""
    j = (np.arange(nblocks, dtype=np.uint64) + np.uint64(offset % 2**64))  # wraps mod 2^64
    seed = int(seed) % 2**64
    stream_id = int(stream_id) % 2**64
    w = philox4x32_10(j & _MASK32, j >> np.uint64(32),
                      np.full(nblocks, stream_id & 0xFFFFFFFF, dtype=np.uint64),
                      np.full(nblocks, stream_id >> 32, dtype=np.uint64),
                      seed & 0xFFFFFFFF, seed >> 32)
    return np.stack(w, axis=1)


def philox_stream(n, seed, stream_id=0, offset=0):
    """The uint32 word used by each of the n elements of a flat tensor."""
    nblocks = (n + 3) // 4
    return philox_blocks(nblocks, seed, stream_id, offset).reshape(-1)[:n]


def scale_fp32(sensitivity, eps):
    """Noise scale b = Delta f / eps (Sec. 4.4), evaluated in fp64 and rounded once to fp32."""
    if not (eps > 0):
        raise ValueError("eps must be > 0")
    if sensitivity < 0 or not np.isfinite(sensitivity):
        raise ValueError("sensitivity must be finite and >= 0")
    if np.isinf(eps):
        return np.float32(0.0)
    return np.float32(float(sensitivity) / float(eps))


def laplace_from_words(words, b):
    """Laplace(0, b) samples (fp64) from uint32 words: sign from bit 31, magnitude -b ln u."""
    words = np.asarray(words, dtype=np.uint32)
    neg = (words >> np.uint32(31)).astype(bool)
    m = (words & np.uint32(0xFFFFFF)).astype(np.float64)
    u = (m + 1.0) * TWO_M24
    mag = float(b) * (-np.log(u))
    return np.where(neg, -mag, mag)


def gaussian_from_blocks(blocks, sigma):
    """N(0, sigma^2) samples (fp64) from Philox blocks [n, 4] by Box-Muller on word pairs."""
    blocks = np.asarray(blocks, dtype=np.uint32)
    out = np.empty(blocks.shape, dtype=np.float64)
    for a, bb in ((0, 1), (2, 3)):
        u1 = ((blocks[:, a] >> np.uint32(8)).astype(np.float64) + 1.0) * TWO_M24
        u2 = (blocks[:, bb] >> np.uint32(8)).astype(np.float64) * TWO_M24
        r = np.sqrt(-2.0 * np.log(u1))
        out[:, a] = float(sigma) * r * np.cos(2.0 * np.pi * u2)
        out[:, bb] = float(sigma) * r * np.sin(2.0 * np.pi * u2)
    return out


def noise(shape, sensitivity, eps, mech, seed, stream_id=0, offset=0, as_fp64=False):
    """The noise tensor eta of the given shape (fp32 unless as_fp64).

    ``mech`` is "laplace" or "gaussian".  eps = +inf yields zeros exactly.
    """
    shape = tuple(int(s) for s in shape)
    n = int(np.prod(shape)) if shape else 1
    b = scale_fp32(sensitivity, eps)
    nblocks = (n + 3) // 4
    blocks = philox_blocks(nblocks, seed, stream_id, offset)
    if mech == "laplace":
        eta = laplace_from_words(blocks.reshape(-1)[:n], np.float64(b))
    elif mech == "gaussian":
        eta = gaussian_from_blocks(blocks, np.float64(b)).reshape(-1)[:n]
    else:
        raise ValueError(f"unknown mechanism {mech!r}")
    eta = eta.reshape(shape)
    return eta if as_fp64 else eta.astype(np.float32)


def radius_fp64(shape, seed, stream_id=0, offset=0):
    """Box-Muller radius R = sqrt(-2 ln u1) behind each Gaussian element (for tolerances)."""
    shape = tuple(int(s) for s in shape)
    n = int(np.prod(shape))
    blocks = philox_blocks((n + 3) // 4, seed, stream_id, offset)
    r = np.empty(blocks.shape, dtype=np.float64)
    for a, bb in ((0, 1), (2, 3)):
        u1 = ((blocks[:, a] >> np.uint32(8)).astype(np.float64) + 1.0) * TWO_M24
        r[:, a] = r[:, bb] = np.sqrt(-2.0 * np.log(u1))
    return r.reshape(-1)[:n].reshape(shape)
