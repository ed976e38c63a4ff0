"""Pins of the Slalom comparator oracle (Sec. 6.2)."""

import numpy as np

from oracle import slalom


def test_modulus_is_the_papers_prime(golden):
    q = golden["slalom"]["modulus"]
    assert slalom.Q == q == 2 ** 23 + 2 ** 21 + 7
    assert all(q % p for p in range(2, int(q ** 0.5) + 1))  # prime by trial division
    assert slalom.FRAC_BITS == golden["slalom"]["fraction_bits"]


def test_quantize_rounds_half_to_even():
    v = np.array([0.5 / 256, 1.5 / 256, -0.5 / 256, 2.5 / 256, 1.0, -0.02])
    np.testing.assert_array_equal(slalom.quantize(v), [0, 2, 0, 2, 256, -5])


def test_mask_noise_is_uniform_and_deterministic():
    eta = slalom.mask_noise((4000,), seed=3, stream_id=1)
    assert eta.min() >= 0 and eta.max() < slalom.Q
    np.testing.assert_array_equal(eta, slalom.mask_noise((4000,), seed=3, stream_id=1))
    # ten equal bins of Z_q: chi-square well inside the 0.1% critical value for 9 dof (27.9)
    counts = np.bincount(eta * 10 // slalom.Q, minlength=10)
    assert np.sum((counts - 400) ** 2 / 400) < 27.9
    # two words per element: element 1 of block 0 uses words 2 and 3
    from oracle import philox
    w = philox.philox_blocks(1, 3, 1, 0)[0]
    assert eta[1] == (int(w[2]) + (int(w[3]) << 32)) % slalom.Q


def test_unmask_recovers_the_quantized_product_exactly():
    """(W x~ - W eta) mod q == W_qt x_qt whenever |W_qt x_qt| < q/2: the one-time pad cancels."""
    g = np.random.default_rng(7)
    X = g.standard_normal((5, 300))
    W = g.standard_normal((40, 300)) * 0.02
    eta = slalom.mask_noise(X.shape, seed=11)
    y = slalom.masked_linear(X, W, eta)
    exact_qt = slalom.product(slalom.quantize(X), slalom.quantize(W))
    assert np.max(np.abs(exact_qt)) < slalom.Q // 2
    np.testing.assert_array_equal(y, exact_qt.astype(np.float64) * 2.0 ** -16)
    # brute force on a tiny case with Python integers
    Xs, Ws, es = X[:1, :3], W[:2, :3], eta[:1, :3]
    xq = [round(v * 256) for v in Xs[0]]  # Python round is also half to even
    wq = [[round(v * 256) for v in row] for row in Ws]
    for n in range(2):
        r = sum(((xq[k] % slalom.Q + int(es[0, k])) % slalom.Q) * wq[n][k] for k in range(3))
        c = sum(int(es[0, k]) * wq[n][k] for k in range(3))
        t = (r - c) % slalom.Q
        t = t - slalom.Q if t > (slalom.Q - 1) // 2 else t
        assert slalom.masked_linear(Xs, Ws, es)[0, n] == t / 65536.0


def test_quantization_error_bound():
    """The recovered product differs from the float product by at most the quantization error:
    sum_k |x_k| |dw_k| + |w_k| |dx_k| + |dx_k| |dw_k| with |dv| <= 2^-9."""
    g = np.random.default_rng(9)
    X = g.standard_normal((6, 512))
    W = g.standard_normal((30, 512)) * 0.02
    eta = slalom.mask_noise(X.shape, seed=12)
    y = slalom.masked_linear(X, W, eta)
    h = 2.0 ** -9
    bound = np.abs(X) @ (np.full(W.shape, h)).T + h * (np.ones(X.shape) @ np.abs(W).T) + h * h * X.shape[1]
    assert np.all(np.abs(y - X @ W.T) <= bound)
