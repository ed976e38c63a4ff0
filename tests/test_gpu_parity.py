"""GPU parity: every entry point of the C ABI against the fp64 oracle.

Inputs are seeded (paper_2609_15039_gb300.workloads) and go to both sides;
expected values come only from ``oracle``.  Integer work (the Philox
stream) is compared bit for bit; floating point within tolerances derived
from the arithmetic (see _util.py and each test).
"""

import math

import numpy as np
import pytest
import torch

from oracle import bounds, linear, philox, slalom, stats
from paper_2609_15039_gb300 import workloads as wl
from _util import U, assert_product_close, f32, f64, ulp32

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def spl():
    from paper_2609_15039_gb300 import spl as binding
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    binding.lib()
    return binding


def dev(a):
    return torch.as_tensor(np.ascontiguousarray(a)).cuda()


# ---------------------------------------------------------------- a2: Philox
@pytest.mark.parametrize("n,seed,sid,off", [
    (1, 0, 0, 0), (5, 1, 0, 0), (4099, 0xDEADBEEFCAFEF00D, 7, 3), (1 << 20, 42, 2**40 + 5, 2**33),
    (1003, 9, 1, 2**64 - 100),
])
def test_random_bits_bit_exact(spl, n, seed, sid, off):
    out = torch.empty(n, dtype=torch.int32, device="cuda")
    spl.spl_random_bits(out, seed, sid, off)
    got = out.cpu().numpy().view(np.uint32)
    np.testing.assert_array_equal(got, philox.philox_stream(n, seed, sid, off))


def test_random_bits_large_stream_sampled(spl):
    n = 1 << 28  # 2.7e8 words on the GPU
    out = torch.empty(n, dtype=torch.int32, device="cuda")
    spl.spl_random_bits(out, 123456789, 3, 11)
    idx = np.random.default_rng(0).integers(0, n, 20000)
    got = out[torch.as_tensor(idx, device="cuda")].cpu().numpy().view(np.uint32)
    blocks = philox.philox_blocks(1, 0, 0, 0)  # warm
    exp = np.empty(idx.size, dtype=np.uint32)
    j = idx // 4 + 11
    w = philox.philox4x32_10(j & 0xFFFFFFFF, j >> 32, 3, 0, 123456789 & 0xFFFFFFFF, 123456789 >> 32)
    for lane in range(4):
        sel = idx % 4 == lane
        exp[sel] = w[lane][sel]
    del blocks
    np.testing.assert_array_equal(got, exp)
    # first 2^24 words in full
    np.testing.assert_array_equal(out[: 1 << 24].cpu().numpy().view(np.uint32),
                                  philox.philox_stream(1 << 24, 123456789, 3, 11))


# ----------------------------------------------------------- a2: noise values
@pytest.mark.parametrize("shape", [(1, 1), (3, 5), (37, 53), (128, 3072)])
@pytest.mark.parametrize("mech", ["laplace", "gaussian"])
def test_noise_matches_oracle(spl, shape, mech):
    sens, eps, seed, sid, off = 825.3, 0.5, 77, 4, 9
    N = torch.empty(shape, dtype=torch.float32, device="cuda")
    spl.spl_noise(N, sens, eps, mech, seed, sid, off)
    got = f64(N)
    exp = philox.noise(shape, sens, eps, mech, seed, sid, off).astype(np.float64)
    if mech == "laplace":
        tol = 4 * ulp32(exp)  # logf within 1 ulp, one product rounding
    else:
        b = float(np.float32(sens / eps))
        R = philox.radius_fp64(shape, seed, sid, off)
        # radius b sqrt(-2 ln u): ln u 1.6 ulp (1.6 U after the root), sqrt.approx 1.68 U, x b 1 U;
        # sin/cos 1.7 ulp (3.4 U): 7.7 U b R, plus the last rounding
        tol = 8 * U * b * R + 2 * ulp32(exp)
    assert np.all(np.abs(got - exp) <= tol)


def test_noise_eps_infinity_is_zero(spl):
    N = torch.full((7, 9), 5.0, device="cuda")
    spl.spl_noise(N, 3.0, None, "gaussian", 1)
    assert torch.count_nonzero(N).item() == 0


@pytest.mark.parametrize("mech", ["laplace", "gaussian"])
def test_gpu_noise_law_ks(spl, mech):
    n = 10 ** 6
    sens, eps = 2.0, 1.0
    N = torch.empty(n, device="cuda")
    spl.spl_noise(N, sens, eps, mech, seed=2024, stream_id=1)
    x = f64(N)
    b = float(np.float32(sens / eps))
    cdf = (lambda t: stats.laplace_cdf(t, b)) if mech == "laplace" else (lambda t: stats.normal_cdf(t, b))
    assert stats.ks_statistic(x, cdf) <= stats.ks_critical(n, 0.001)
    var = 2 * b * b if mech == "laplace" else b * b
    assert abs(x.var() / var - 1) < 0.01


# ------------------------------------------------------ a3 mask, a6 unmask
@pytest.mark.parametrize("shape", [(1, 3), (17, 33), (128, 3072)])
def test_mask_and_unmask_bit_exact(spl, shape):
    g = np.random.default_rng(sum(shape))
    X = g.standard_normal(shape).astype(np.float32)
    Nz = (700 * g.standard_normal(shape)).astype(np.float32)
    Xt = torch.empty(shape, device="cuda")
    spl.spl_mask(Xt, dev(X), dev(Nz))
    np.testing.assert_array_equal(f32(Xt), linear.mask(X, Nz))
    Y = torch.empty(shape, device="cuda")
    spl.spl_unmask(Y, dev(Nz), dev(X))
    np.testing.assert_array_equal(f32(Y), linear.unmask(Nz, X))
    # in place
    Xd = dev(X)
    spl.spl_mask(Xd, Xd, dev(Nz))
    np.testing.assert_array_equal(f32(Xd), linear.mask(X, Nz))


@pytest.mark.parametrize("mech", ["laplace", "gaussian"])
@pytest.mark.parametrize("shape", [(16, 256), (5, 7)])
def test_noise_mask_fused(spl, mech, shape):
    X = wl.activations(*shape, seed=3, norm="unit").numpy()
    Xt = torch.empty(shape, device="cuda")
    N = torch.empty(shape, device="cuda")
    spl.spl_noise_mask(Xt, N, dev(X), 2.0, 1.0, mech, seed=0)
    n_exp = philox.noise(shape, 2.0, 1.0, mech, 0).astype(np.float64)
    xt_exp = linear.mask(X, n_exp.astype(np.float32)).astype(np.float64)
    # the GPU's eta differs from the oracle's by a few ulps (transcendentals); X~ by that plus one rounding
    dn = np.abs(f64(N) - n_exp)
    assert np.all(np.abs(f64(Xt) - xt_exp) <= dn + ulp32(xt_exp) + ulp32(n_exp) * 8)
    # property: the eta written out is exactly the eta that was added
    assert torch.equal(Xt.cpu(), (torch.as_tensor(X) + N.cpu()))
    # without N_out, in place, same X~
    Xd = dev(X)
    spl.spl_noise_mask(Xd, None, Xd, 2.0, 1.0, mech, seed=0)
    assert torch.equal(Xd, Xt)
    # eps = inf: X~ == X bit for bit
    spl.spl_noise_mask(Xt, N, dev(X), 2.0, None, mech, seed=0)
    np.testing.assert_array_equal(f32(Xt), X)
    assert torch.count_nonzero(N).item() == 0


def test_split_tf32_properties(spl):
    W = wl.weight(257, 1028, seed=5).numpy()
    # ties: 1 + 2^-11 sits halfway between 1 and 1 + 2^-10 (TF32 ulp at 1)
    W[0, :4] = [0.0, -0.0, 1.0 + 2.0 ** -11, -(1.0 + 3 * 2.0 ** -11)]
    hi = torch.empty_like(dev(W))
    lo = torch.empty_like(hi)
    spl.spl_split_tf32(hi, lo, dev(W))
    h, l = f32(hi), f32(lo)
    assert np.all(h.astype(np.float64) + l.astype(np.float64) == W.astype(np.float64))
    assert np.all(h.view(np.uint32) & 0x1FFF == 0)  # 10 explicit mantissa bits
    assert np.all(np.abs(l.astype(np.float64)) <= 2.0 ** -11 * np.abs(W.astype(np.float64)) * (1 + 2 ** -10))
    assert h[0, 2] == np.float32(1.0 + 2.0 ** -10)  # tie rounds away from zero
    assert h[0, 3] == np.float32(-(1.0 + 2 * 2.0 ** -10))


# ------------------------------------------------ a4/a5/a6: products
def _weights(spl, N, K, seed):
    """Host W and the device Weight with both splits (the fp16 one when K % 8 == 0)."""
    W = wl.weight(N, K, seed=seed).numpy()
    return W, spl.Weight.prepare(dev(W))


def _fp16_bits(x):
    return np.asarray(x, dtype=np.float16).view(np.int16)


@pytest.mark.parametrize("cols", [1032, 16448])  # rows held in registers; longer rows take the two-pass kernel
def test_split_fp16_properties(spl, cols):
    """hi = fp16(w 2^e), lo = fp16(w 2^e - hi) per row; e puts the row's largest |w| in [2^14, 2^15)."""
    W = wl.weight(37, cols, seed=6).numpy()
    W[1] = 0.0                                  # all-zero row: e = 0, hi = lo = 0
    W[2] *= np.float32(1e-30)                   # tiny row (residuals below fp16's normal range)
    W[3] *= np.float32(1e30)                    # huge row
    W[4, :4] = [1.0, 1.0 + 2.0 ** -11, -(1.0 + 3 * 2.0 ** -11), 2.0 ** -30]  # fp16 ties at 1 (ulp 2^-10)
    W[4, 4:] = 0.0
    hi = torch.empty(W.shape, dtype=torch.int16, device="cuda")
    lo = torch.empty_like(hi)
    ex = torch.empty(W.shape[0], dtype=torch.int32, device="cuda")
    spl.spl_split_fp16(hi, lo, ex, dev(W))
    e = ex.cpu().numpy()
    h = hi.cpu().numpy().view(np.float16).astype(np.float64)
    l = lo.cpu().numpy().view(np.float16).astype(np.float64)
    amax = np.abs(W.astype(np.float64)).max(axis=1)
    assert e[1] == 0 and not h[1].any() and not l[1].any()
    nz = amax > 0
    scaled_max = amax[nz] * np.exp2(e[nz].astype(np.float64))
    assert np.all((scaled_max >= 2.0 ** 14) & (scaled_max < 2.0 ** 15))
    Ws = W.astype(np.float64) * np.exp2(e.astype(np.float64))[:, None]  # exact: power-of-two scaling
    # numpy's float16 cast rounds to nearest even, the kernel's __float2half_rn too
    np.testing.assert_array_equal(hi.cpu().numpy(), _fp16_bits(Ws))
    np.testing.assert_array_equal(lo.cpu().numpy(), _fp16_bits(Ws - h))
    assert np.all(np.abs(Ws - h - l) <= 2.0 ** -22 * np.abs(Ws) + 2.0 ** -25)
    assert e[4] == 14 and h[4, 1] == 2.0 ** 14  # 2^14 (1 + 2^-11) ties to even (2^14)


SHAPES = [(1, 4, 1), (3, 8, 5), (1, 256, 512), (16, 256, 512), (7, 3072, 1024), (17, 260, 300),
          (130, 1028, 600), (128, 3072, 1024), (300, 64, 257), (130, 1032, 600), (17, 264, 300),
          (257, 2056, 520)]


def _skip(path, K):
    if path != "fp32" and K < 64:
        pytest.skip("the three-product split is not within gamma_K below K = 64 (the AUTO path picks FP32)")
    if path == "fp16x3" and K % 8:
        pytest.skip("FP16X3 needs K % 8 == 0 (whole 16-byte rows of fp16)")


@pytest.mark.parametrize("M,K,N", SHAPES)
@pytest.mark.parametrize("path", ["fp32", "tf32x3", "fp16x3"])
def test_products_match_oracle(spl, M, K, N, path):
    _skip(path, K)
    W, Wt = _weights(spl, N, K, seed=M + K + N)
    A = (wl.activations(M, K, seed=M * 7 + 1).numpy() * 300).astype(np.float32)
    C = wl.activations(M, N, seed=11).numpy()
    ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N, path))
    Yt = torch.empty((M, N), device="cuda")
    for _ in range(2):  # twice: the workspace must be reusable (counters reset)
        spl.spl_masked_linear(Yt, dev(A), Wt, path=path, workspace=ws)
        assert_product_close(f32(Yt), A, W, path, what="masked_linear")
    Cp = torch.empty((M, N), device="cuda")
    spl.spl_precompute_noise_product(Cp, dev(A), Wt, path=path, workspace=ws)
    assert_product_close(f32(Cp), A, W, path, what="precompute")
    Y = torch.empty((M, N), device="cuda")
    spl.spl_masked_linear_unmask(Y, dev(A), Wt, dev(C), path=path, workspace=ws)
    assert_product_close(f32(Y), A, W, path, C=C, what="masked_linear_unmask")
    assert spl.spl_get_device_status() == 0


TC_VARIANTS = [(256, 192), (128, 224), (128, 96), (160, 224), (192, 224), (224, 224)]


def test_long_row_products_back_to_back_share_a_workspace(spl):
    """FP16X3 products with K > 16384 (the left operand split by the two-pass kernel) issued back to
    back on one stream with one workspace: each split waits for the product before it, which may
    still be reading the previous split, so every result equals the same call made alone."""
    M, K, N = 130, 16448, 384
    Ws = [spl.Weight.prepare(wl.weight(N, K, seed=60 + i, device="cuda")) for i in range(2)]
    Xs = [wl.activations(M, K, seed=70 + i, device="cuda") * (1 + 40 * i) for i in range(2)]
    Cs = [wl.activations(M, N, seed=80 + i, device="cuda") for i in range(2)]
    refs = []
    for X, W, C in zip(Xs, Ws, Cs):
        Y = torch.empty((M, N), device="cuda")
        spl.spl_masked_linear_unmask(Y, X, W, C, path="fp16x3",
                                     workspace=spl.workspace(spl.spl_linear_workspace_bytes(M, K, N, "fp16x3")))
        torch.cuda.synchronize()
        refs.append(Y)
    ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N, "fp16x3"))
    outs = [[torch.empty((M, N), device="cuda") for _ in range(2)] for _ in range(4)]
    for rep in range(4):
        for i in range(2):
            spl.spl_masked_linear_unmask(outs[rep][i], Xs[i], Ws[i], Cs[i], path="fp16x3", workspace=ws)
    torch.cuda.synchronize()
    for rep in range(4):
        for i in range(2):
            assert torch.equal(outs[rep][i], refs[i]), (rep, i)
    ref64 = Xs[0].double() @ Ws[0].w.double().T - Cs[0].double()
    assert float((refs[0].double() - ref64).abs().max()) <= 1e-5 * float(ref64.abs().max())


@pytest.mark.parametrize("splits", [1, 3, 8])
@pytest.mark.parametrize("path", ["tf32x3", "fp16x3"])
@pytest.mark.parametrize("tile_n,ring_kb", TC_VARIANTS)
def test_tc_every_launch_shape(spl, path, tile_n, ring_kb, splits):
    """Each kernel instance (encoding x tile width x ring) with each cluster K-split, on a ragged
    problem: M, N and K not multiples of the tile, and at 8 splits an empty last K range."""
    M, K, N = 130, 1032, 600
    W, Wt = _weights(spl, N, K, seed=41)
    A = (wl.activations(M, K, seed=42).numpy() * 300).astype(np.float32)
    C = wl.activations(M, N, seed=43).numpy()
    Y = torch.empty((M, N), device="cuda")
    spl.spl_test_tc_product(Y, dev(A), Wt, dev(C), path=path, tile_n=tile_n, ring_kb=ring_kb, splits=splits)
    assert_product_close(f32(Y), A, W, path, C=C, what=f"{path} tile {tile_n} split {splits}")
    Y2 = torch.empty((M, N), device="cuda")
    spl.spl_test_tc_product(Y2, dev(A), Wt, None, path=path, tile_n=tile_n, ring_kb=ring_kb, splits=splits)
    assert_product_close(f32(Y2), A, W, path, what="without C")
    # the first tiles unsplit in a launch of their own, the rest split
    tiles = -(-M // 128) * -(-N // tile_n)
    Y3 = torch.empty((M, N), device="cuda")
    spl.spl_test_tc_product(Y3, dev(A), Wt, dev(C), path=path, tile_n=tile_n, ring_kb=ring_kb, splits=splits,
                            full_tiles=tiles // 2 + 1)
    assert_product_close(f32(Y3), A, W, path, C=C, what=f"{path} tile {tile_n} split {splits}, two launches")
    assert spl.spl_get_device_status() == 0


SWAP_WIDTHS = [16, 32, 64, 128]


@pytest.mark.parametrize("M", [9, 16, 33, 64])
@pytest.mark.parametrize("ctas", [0, 1, 7, 40])
def test_swap_every_width_and_run_length(spl, M, ctas):
    """The swapped kernel (weight rows in the MMA's 128 rows, tokens in its N) at every token-tile
    width and run length (1 CTA: one run over every tile, whole tiles straight out; 7 and 40: runs
    that cut tiles into pieces summed through the workspace), ragged M, K and N (tokens past M are
    the copy's zero rows): within the product tolerance of the oracle, with and without C, and the
    same bits at every width -- an output's sum does not depend on the other columns of its MMA,
    which the bank relies on."""
    K, N = 1032, 600
    W, Wt = _weights(spl, N, K, seed=81)
    A = (wl.activations(M, K, seed=82 + M).numpy() * 300).astype(np.float32)
    C = wl.activations(M, N, seed=83).numpy()
    ws = spl.workspace(max(spl.spl_test_tc_swap_workspace_bytes(M, K, N, tn, ctas) for tn in SWAP_WIDTHS))
    first = None
    for tn in SWAP_WIDTHS:
        Y = torch.full((M, N), float("nan"), device="cuda")
        spl.spl_test_tc_swap_product(Y, dev(A), Wt, dev(C), tile_tokens=tn, ctas=ctas, workspace=ws)
        assert_product_close(f32(Y), A, W, "fp16x3", C=C, what=f"swap {tn} ctas {ctas}")
        if first is None:
            first = Y
        assert torch.equal(Y, first), (tn, float((Y - first).abs().max()))
    Y2 = torch.full((M, N), float("nan"), device="cuda")
    spl.spl_test_tc_swap_product(Y2, dev(A), Wt, None, tile_tokens=16 if M <= 16 else 64, ctas=ctas, workspace=ws)
    assert_product_close(f32(Y2), A, W, "fp16x3", what="swap without C")
    assert spl.spl_get_device_status() == 0


def test_library_takes_the_swapped_kernel_for_few_rows(spl):
    """AUTO runs 9-16 rows on the swapped kernel: the library's product equals the swapped kernel's
    bit for bit (at the width of the rows and the library's run length), also on the operand split
    beforehand (the layers' form); from 17 rows on it takes the 128-row tiles."""
    K, N = 3072, 5120
    W, Wt = _weights(spl, N, K, seed=91)
    for M in (9, 16, 17):
        A = wl.activations(M, K, seed=92 + M).numpy()
        ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N))
        Y = torch.empty((M, N), device="cuda")
        spl.spl_masked_linear(Y, dev(A), Wt, workspace=ws)
        tn = next(t for t in SWAP_WIDTHS if M <= t)
        Ys = torch.empty((M, N), device="cuda")
        spl.spl_test_tc_swap_product(Ys, dev(A), Wt, None, tile_tokens=tn, ctas=0,
                                     workspace=spl.workspace(spl.spl_test_tc_swap_workspace_bytes(M, K, N, tn, 0)))
        assert torch.equal(Y, Ys) == (M <= 16), M
        if M <= 16:  # the pre-split operand
            hi = torch.empty((M, K), dtype=torch.int16, device="cuda")
            lo, ex = torch.empty_like(hi), torch.empty(M, dtype=torch.int32, device="cuda")
            spl.spl_split_fp16(hi, lo, ex, dev(A))
            Yp = torch.empty((M, N), device="cuda")
            spl.spl_masked_linear_unmask_split(Yp, spl.Weight(None, f16_hi=hi, f16_lo=lo, f16_exp=ex), Wt,
                                               torch.zeros((M, N), device="cuda"), workspace=ws)
            assert torch.equal(Yp, Y)
    assert spl.spl_get_device_status() == 0


@pytest.mark.parametrize("path", ["fp16x3", "tf32x3"])
@pytest.mark.parametrize("M,M_bank,K,N", [(128, 128, 3072, 5120), (130, 70, 1032, 600), (0, 40, 264, 300),
                                          (40, 0, 264, 300), (12, 12, 2056, 700)])
def test_precompute_beside_masked_rows(spl, path, M, M_bank, K, N):
    """spl_masked_linear_unmask_precompute: the first M output rows are the masked product with its unmask,
    the others the corrections of the noise rows, each within the product tolerance of the oracle, and
    every row summed as the same row of a plain product of M + M_bank rows (bit for bit: launch forms
    are uniform over the rows)."""
    W, Wt = _weights(spl, N, K, seed=K + N + 5)
    rows = M + M_bank
    A = (wl.activations(rows, K, seed=rows + 3).numpy() * 300).astype(np.float32)
    C = wl.activations(M, N, seed=9).numpy()
    ws = spl.workspace(spl.spl_linear_workspace_bytes(rows, K, N, path))
    YC = torch.full((rows, N), float("nan"), device="cuda")
    spl.spl_masked_linear_unmask_precompute(YC, dev(A), Wt, dev(C) if M else None, M, path=path, workspace=ws)
    if M:
        assert_product_close(f32(YC[:M]), A[:M], W, path, C=C, what="masked rows")
    if M_bank:
        assert_product_close(f32(YC[M:]), A[M:], W, path, what="correction rows")
    P = torch.empty((rows, N), device="cuda")
    spl.spl_masked_linear(P, dev(A), Wt, path=path, workspace=ws)
    assert torch.equal(YC[M:], P[M:])  # the correction rows: no C subtracted, the same sums
    if M:
        Yu = torch.empty((M, N), device="cuda")
        spl.spl_unmask(Yu, P[:M].contiguous(), dev(C))
        assert torch.equal(YC[:M], Yu)  # fused unmask = the plain product then one subtraction
    assert spl.spl_get_device_status() == 0


@pytest.mark.parametrize("path", ["tf32x3", "fp16x3"])
def test_products_with_extreme_row_scales(spl, path):
    """Rows of A and W spread over 60 orders of magnitude, zero rows included: the power-of-two
    row scaling of FP16X3 keeps every row inside fp16's range."""
    M, K, N = 160, 1024, 300
    A = wl.activations(M, K, seed=31).numpy().astype(np.float64)
    A *= np.array([0.0, 1e-20, 1e-5, 1.0, 1e5, 1e20])[np.arange(M) % 6][:, None]
    W = wl.weight(N, K, seed=32).numpy().astype(np.float64)
    W *= np.array([1e-10, 1.0, 1e10])[np.arange(N) % 3][:, None]
    A, W = A.astype(np.float32), W.astype(np.float32)
    Wt = spl.Weight.prepare(dev(W))
    Y = torch.empty((M, N), device="cuda")
    spl.spl_masked_linear(Y, dev(A), Wt, path=path, workspace=spl.workspace(spl.spl_linear_workspace_bytes(M, K, N)))
    assert_product_close(f32(Y), A, W, path, what=path)
    assert not torch.any(Y[0::6]).item()  # zero rows give exact zeros


def test_one_workspace_serves_every_shape_and_path(spl):
    """Decode counters sit at a fixed place, so partials of other calls never land on them."""
    cases = [(130, 1028, 600, "tf32x3"), (1, 3072, 3072, "fp32"), (17, 260, 300, "fp32"), (4, 8192, 1024, "fp32"),
             (1, 3072, 3072, "fp32"), (1000, 1024, 256, "fp16x3"), (300, 64, 257, "fp32"), (16, 2560, 3000, "fp32"),
             (1, 3072, 3072, "fp32")]
    need = max(spl.spl_linear_workspace_bytes(M, K, N, path) for M, K, N, path in cases)
    ws = spl.workspace(need)
    for i, (M, K, N, path) in enumerate(cases):
        W, Wt = _weights(spl, N, K, seed=50 + i)
        A = (wl.activations(M, K, seed=60 + i).numpy() * 300).astype(np.float32)
        C = wl.activations(M, N, seed=70 + i).numpy()
        Y = torch.empty((M, N), device="cuda")
        spl.spl_masked_linear_unmask(Y, dev(A), Wt, dev(C), path=path, workspace=ws)
        assert_product_close(f32(Y), A, W, path, C=C, what=f"case {i}")
    # the counter region is back to zero after every call
    assert torch.count_nonzero(ws[: 64 * 1024]).item() == 0


def test_workspace_errors(spl):
    M, K, N = 4, 3072, 3072
    W, Wt = _weights(spl, N, K, seed=1)
    Wd = Wt.w
    A = dev(wl.activations(M, K, seed=2).numpy())
    Y = torch.empty((M, N), device="cuda")
    need = spl.spl_linear_workspace_bytes(M, K, N, "fp32")
    assert need > 0
    with pytest.raises(spl.SplError) as e:
        spl.spl_masked_linear(Y, A, Wd, path="fp32", workspace=spl.workspace(16))
    assert e.value.status == spl.SPL_EWORKSPACE
    A130, Y130 = dev(np.zeros((130, K), np.float32)), torch.empty((130, N), device="cuda")
    for path in ("tf32x3", "fp16x3"):
        with pytest.raises(spl.SplError) as e:
            spl.spl_masked_linear(Y130, A130, Wd, path=path,
                                  workspace=spl.workspace(spl.spl_linear_workspace_bytes(130, K, N)))
        assert e.value.status == spl.SPL_EUNSUPPORTED  # no weight split given
    with pytest.raises(spl.SplError) as e:  # FP16X3 keeps its row exponents in the workspace
        spl.spl_masked_linear(Y130, A130, Wt, path="fp16x3", workspace=None)
    assert e.value.status == spl.SPL_EWORKSPACE
    misaligned = torch.empty(M * K + 1, device="cuda")[1:].view(M, K)
    with pytest.raises(spl.SplError) as e:
        spl.spl_masked_linear(Y, misaligned, Wd, path="fp32", workspace=spl.workspace(need))
    assert e.value.status == spl.SPL_EALIGN
    # K % 8 != 0: no fp16 split is made, AUTO takes TF32X3, explicit FP16X3 is refused
    K4 = 1028
    W4 = spl.Weight.prepare(dev(wl.weight(64, K4, seed=3).numpy()))
    assert W4.f16_hi is None
    W4.f16_hi, W4.f16_lo = torch.zeros((64, K4), dtype=torch.int16, device="cuda"), torch.zeros(
        (64, K4), dtype=torch.int16, device="cuda")
    W4.f16_exp = torch.zeros(64, dtype=torch.int32, device="cuda")
    with pytest.raises(spl.SplError) as e:
        spl.spl_masked_linear(torch.empty((130, 64), device="cuda"), dev(np.zeros((130, K4), np.float32)), W4,
                              path="fp16x3", workspace=spl.workspace(spl.spl_linear_workspace_bytes(130, K4, 64)))
    assert e.value.status == spl.SPL_EALIGN


def test_empty_reduction(spl):
    C = torch.arange(6, dtype=torch.float32, device="cuda").view(2, 3)
    Y = torch.full((2, 3), 9.0, device="cuda")
    spl.spl_masked_linear_unmask(Y, torch.empty((2, 0), device="cuda"), torch.empty((3, 0), device="cuda"), C)
    assert torch.equal(Y, -C)


@pytest.mark.parametrize("M,K,N,path", [(128, 3072, 3072, "tf32x3"), (128, 3072, 3072, "fp32"),
                                         (1, 3072, 3072, "fp32"), (128, 8192, 3072, "tf32x3"),
                                         (128, 3072, 3072, "fp16x3"), (128, 8192, 3072, "fp16x3")])
def test_matched_correction_cancels_rounding(spl, M, K, N, path):
    """A bank of 8 corrections summed in the online product's order: the same values up to
    rounding, every recovered output inside the hard bound, and a recovered error no larger than
    with a correction computed with its own plan for 8 x M rows."""
    draws, b = 8, 1443.0
    W, Wt = _weights(spl, N, K, seed=K + N)
    X = wl.activations(M, K, seed=21).numpy()
    eta = philox.noise((draws * M, K), b, 1.0, "gaussian", seed=22)
    Nd = dev(eta)
    C_plain, C_matched = torch.empty((draws * M, N), device="cuda"), torch.empty((draws * M, N), device="cuda")
    ws = spl.workspace(max(spl.spl_linear_workspace_bytes(draws * M, K, N, path),
                           spl.spl_precompute_matched_workspace_bytes(draws * M, K, N, M, path),
                           spl.spl_linear_workspace_bytes(M, K, N, path)))
    spl.spl_precompute_noise_product(C_plain, Nd, Wt, path=path, workspace=ws)
    spl.spl_precompute_noise_product_matched(C_matched, Nd, Wt, M, path=path, workspace=ws)
    assert_product_close(f32(C_matched), eta, W, path, what="matched correction")
    d = draws - 1
    Xt = linear.mask(X, eta[d * M:(d + 1) * M])
    errs = {}
    for name, Cb in (("plain", C_plain), ("matched", C_matched)):
        Y = torch.empty((M, N), device="cuda")
        spl.spl_masked_linear_unmask(Y, dev(Xt), Wt, Cb[d * M:(d + 1) * M].contiguous(), path=path, workspace=ws)
        err = np.abs(f64(Y) - linear.reference_output(X, W))
        S = linear.abs_products(X, Xt, eta[d * M:(d + 1) * M], W)
        assert np.all(err <= bounds.hard_bound(*S, K)), name
        errs[name] = float(err.mean())
    # Matching never hurts.  How much it helps depends on how far the plain plan's order is from the
    # online one: FMA chains in ascending k already keep the two roundings correlated, and on the
    # tensor cores the dominant error -- the truncation bias of each accumulation chain -- is the same
    # in both wherever their chains are cut at the same K boundaries (every chain of an unsplit tile
    # starts at a multiple of 32 k-blocks), so only the round-to-nearest folds differ.
    assert errs["matched"] <= errs["plain"] * 1.1, errs


@pytest.mark.parametrize("M,K,N,path", [(128, 3072, 3072, "fp16x3"), (128, 3072, 5120, "fp16x3"),
                                         (128, 8192, 3072, "fp16x3"), (128, 3072, 16384, "fp16x3"),
                                         (128, 3072, 3072, "tf32x3"), (100, 1032, 600, "fp16x3"),
                                         (128, 3072, 3072, "fp32"), (1, 3072, 3072, "fp32"), (512, 3072, 3072, "fp16x3"),
                                         (1, 3072, 5120, "fp32"), (1, 3072, 16384, "fp32"), (1, 8192, 3072, "fp32"),
                                         (4, 3072, 5120, "fp32"), (3, 1028, 600, "fp32"),
                                         (16, 3072, 5120, "fp16x3"), (16, 9728, 2560, "fp16x3"),
                                         (16, 3072, 16384, "fp16x3"), (32, 2560, 19456, "fp16x3"),
                                         (12, 1032, 600, "fp16x3")])
@pytest.mark.parametrize("draws", [4, 8])
def test_matched_correction_is_the_online_order_bitwise(spl, M, K, N, path, draws):
    """The bank's correction of draw d is, bit for bit, what the online product computes when
    its input is that draw's noise: the same K ranges, partials summed in the same order (with 8
    draws of 128 rows the bank mixes whole waves of tiles that fold the K ranges in TMEM and
    tiles split over a cluster)."""
    W, Wt = _weights(spl, N, K, seed=K + N + 1)
    eta = torch.empty((draws * M, K), device="cuda")
    spl.spl_noise(eta, 1443.0, 1.0, "gaussian", seed=23)
    C = torch.empty((draws * M, N), device="cuda")
    ws = spl.workspace(max(spl.spl_precompute_matched_workspace_bytes(draws * M, K, N, M, path),
                           spl.spl_linear_workspace_bytes(M, K, N, path)))
    spl.spl_precompute_noise_product_matched(C, eta, Wt, M, path=path, workspace=ws)
    for d in range(draws):
        Y = torch.empty((M, N), device="cuda")
        spl.spl_masked_linear(Y, eta[d * M:(d + 1) * M].contiguous(), Wt, path=path, workspace=ws)
        assert torch.equal(Y, C[d * M:(d + 1) * M]), (d, float((Y - C[d * M:(d + 1) * M]).abs().max()))
    assert spl.spl_get_device_status() == 0


@pytest.mark.parametrize("tile_n,ring_kb", [(256, 192), (224, 224), (128, 96)])
@pytest.mark.parametrize("N", [600, 601])
def test_tc_unsplit_epilogue_on_ragged_rows(spl, tile_n, ring_kb, N):
    """Unsplit tiles store through TMA when an output row is a whole number of 16-byte units
    (N = 600) and through the thread loop otherwise (N = 601): in segmented mode (the K ranges of a
    2-way split folded in order) both give the 2-way cluster-split product bit for bit, whose
    reduction always stores through the thread loop; with and without C, ragged M and N."""
    M, K = 131, 1040
    W, Wt = _weights(spl, N, K, seed=53)
    A = wl.activations(M, K, seed=54).numpy()
    C = dev(wl.activations(M, N, seed=55).numpy())
    ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N, "fp16x3"))
    for Cx in (C, None):
        ref = torch.empty((M, N), device="cuda")
        spl.spl_test_tc_product(ref, dev(A), Wt, Cx, tile_n=tile_n, ring_kb=ring_kb, splits=2, workspace=ws)
        assert_product_close(f32(ref), A, W, "fp16x3", C=None if Cx is None else C.cpu().numpy(),
                             what=f"N {N} split 2")
        Y = torch.full((M, N), float("nan"), device="cuda")
        spl.spl_test_tc_product(Y, dev(A), Wt, Cx, tile_n=tile_n, ring_kb=ring_kb, splits=1, seg_splits=2,
                                workspace=ws)
        assert torch.equal(Y, ref), float((Y - ref).abs().max())
    assert spl.spl_get_device_status() == 0


@pytest.mark.parametrize("path", ["tf32x3", "fp16x3"])
@pytest.mark.parametrize("tile_n,ring_kb", [v for v in TC_VARIANTS if v != (128, 96)])
@pytest.mark.parametrize("K", [264, 3080])
def test_tc_persistent_equals_unsplit_product(spl, path, tile_n, ring_kb, K):
    """The persistent kernel (one CTA per SM looping over tiles, two TMEM buffers, the epilogue of
    one tile beside the mainloop of the next) gives the unsplit product bit for bit, with and
    without C, on a problem of 2 to 4 tiles per CTA with ragged M, N and K -- at K = 3080 with every
    tile's K range cut into accumulation chains that are folded in TMEM (4 for FP16X3, 7 for TF32X3)."""
    M, N = 2600, 4000
    W, Wt = _weights(spl, N, K, seed=61)
    A = wl.activations(M, K, seed=62).numpy()
    C = dev(wl.activations(M, N, seed=63).numpy())
    ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N, path))
    assert -(-M // 128) * -(-N // tile_n) > spl.spl_test_tc_capacity(tile_n, ring_kb, 1)
    for Cx in (C, None):
        ref = torch.empty((M, N), device="cuda")
        spl.spl_test_tc_product(ref, dev(A), Wt, Cx, path=path, tile_n=tile_n, ring_kb=ring_kb, splits=1, workspace=ws)
        Y = torch.full((M, N), float("nan"), device="cuda")
        spl.spl_test_tc_product(Y, dev(A), Wt, Cx, path=path, tile_n=tile_n, ring_kb=ring_kb, splits=1, workspace=ws,
                                persistent=True)
        assert torch.equal(Y, ref), float((Y - ref).abs().max())
    rows = np.arange(0, M, 97)
    assert_product_close(f32(ref[torch.as_tensor(rows, device="cuda")]), A[rows], W, path, what="persistent, no C")
    assert spl.spl_get_device_status() == 0


def test_library_picks_persistent_for_many_waves(spl):
    """The launch model takes the persistent kernel for a product of many waves of unsplit tiles
    (Qwen Gate|Up at 2048 rows) and not for one wave (128 rows, cluster split); the product the
    library runs equals the forced persistent launch bit for bit."""
    M, K, N = 2048, 2560, 19456
    shape = spl.spl_test_tc_shape(M, K, N)
    assert shape[5] == 1 and shape[4] == 1 and shape[2] == 0
    assert spl.spl_test_tc_shape(128, K, N)[5] == 0
    W = wl.weight(N, K, seed=71, device="cuda")
    Wt = spl.Weight.prepare(W)
    X = wl.activations(M, K, seed=72, device="cuda")
    C = wl.activations(M, N, seed=73, device="cuda")
    ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N, "fp16x3"))
    Y = torch.empty((M, N), device="cuda")
    spl.spl_masked_linear_unmask(Y, X, Wt, C, path="fp16x3", workspace=ws)
    Yp = torch.full((M, N), float("nan"), device="cuda")
    spl.spl_test_tc_product(Yp, X, Wt, C, path="fp16x3", tile_n=shape[0], ring_kb=shape[1], splits=1,
                            workspace=ws, persistent=True)
    assert torch.equal(Y, Yp)
    assert spl.spl_get_device_status() == 0


@pytest.mark.parametrize("path", ["tf32x3", "fp16x3"])
@pytest.mark.parametrize("tile_n,ring_kb", TC_VARIANTS)
@pytest.mark.parametrize("K,s", [(2056, 3), (3080, 2), (3080, 1)])
def test_tc_segmented_equals_split_product(spl, path, tile_n, ring_kb, K, s):
    """Every kernel instance in the bank's form (seg_splits = s) gives the online product of the
    same K-split bit for bit, alone and with the tiles after the first half+1 split over a cluster;
    ragged M, N and K.  Where a rank's K range is one accumulation chain (2056 / 3 on FP16X3) one CTA
    over all of K folds the ranks' partial sums in TMEM in rank order; where the ranks fold chains of
    their own (3080 / 2, and 2056 / 3 on TF32X3) the tiles run as the same cluster split; an unsplit
    product (s = 1) is folded at the same chain boundaries."""
    M, N = 300, 700
    W, Wt = _weights(spl, N, K, seed=47)
    A = (wl.activations(M, K, seed=48).numpy() * 30).astype(np.float32)
    C = dev(wl.activations(M, N, seed=49).numpy())
    tiles = -(-M // 128) * -(-N // tile_n)
    ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N, path))
    ref = torch.empty((M, N), device="cuda")
    spl.spl_test_tc_product(ref, dev(A), Wt, C, path=path, tile_n=tile_n, ring_kb=ring_kb, splits=s, workspace=ws)
    assert_product_close(f32(ref), A, W, path, C=C.cpu().numpy(), what=f"{path} tile {tile_n} split {s}")
    for full, splits in ((0, 1), (tiles // 2 + 1, s), (tiles, 1)):
        Y = torch.full((M, N), float("nan"), device="cuda")
        spl.spl_test_tc_product(Y, dev(A), Wt, C, path=path, tile_n=tile_n, ring_kb=ring_kb, splits=splits,
                                full_tiles=full, seg_splits=s, workspace=ws)
        assert torch.equal(Y, ref), (full, splits, float((Y - ref).abs().max()))
    assert spl.spl_get_device_status() == 0


def test_bank_shape_mixes_folded_and_split_tiles(spl):
    """A correction of 8 x 128 rows for the Llama Q|K|V shape: its tiles cover the output once,
    a whole wave of them folded in TMEM and the rest (if any) split over a cluster the way the
    online product splits K."""
    online = spl.spl_test_tc_shape(128, 3072, 5120)
    assert online[2] == 0  # the online product is one split launch
    bank = spl.spl_test_tc_shape(1024, 3072, 5120, seg_splits=online[4])
    assert bank[2] + bank[3] == (1024 // 128) * -(-5120 // bank[0])
    assert bank[3] == 0 or bank[4] == online[4]
    assert bank[2] % spl.spl_test_tc_capacity(bank[0], bank[1], 1) == 0


# ------------------------------------------------ a2 + a3 fused with the split of X~
@pytest.mark.parametrize("rows,cols,mech,eps", [(5, 8, "laplace", 1.0), (130, 3072, "gaussian", 0.5),
                                                (3, 16384, "laplace", 2.0), (17, 1032, "gaussian", None)])
def test_noise_mask_split_equals_separate_calls(spl, rows, cols, mech, eps):
    X = dev(wl.activations(rows, cols, seed=rows + cols).numpy())
    base = torch.tensor([3000], dtype=torch.int64, device="cuda")
    xt_ref = torch.empty_like(X)
    spl.spl_noise_mask(xt_ref, None, X, 825.3, eps, mech, seed=19, stream_id=2, offset=3000 + 40)
    hi_ref = torch.empty(X.shape, dtype=torch.int16, device="cuda")
    lo_ref, ex_ref = torch.empty_like(hi_ref), torch.empty(rows, dtype=torch.int32, device="cuda")
    spl.spl_split_fp16(hi_ref, lo_ref, ex_ref, xt_ref)
    xt = torch.empty_like(X)
    hi, lo, ex = torch.empty_like(hi_ref), torch.empty_like(lo_ref), torch.empty_like(ex_ref)
    spl.spl_noise_mask_split(xt, hi, lo, ex, X, 825.3, eps, mech, seed=19, stream_id=2, offset=40, offset_dev=base)
    assert torch.equal(xt, xt_ref) and torch.equal(hi, hi_ref) and torch.equal(lo, lo_ref) and torch.equal(ex, ex_ref)
    spl.spl_noise_mask_split(None, hi, lo, ex, X, 825.3, eps, mech, seed=19, stream_id=2, offset=3040)  # no X~ out
    assert torch.equal(hi, hi_ref) and torch.equal(ex, ex_ref)


@pytest.mark.parametrize("x_rows,noise_rows,cols,mech,eps", [(512, 512, 3072, "laplace", 1.0), (5, 3, 8, "gaussian", 0.5),
                                                               (3, 7, 16384, "laplace", 2.0), (0, 4, 1032, "gaussian", 1.0),
                                                               (6, 0, 1032, "laplace", None)])
def test_stacked_split_equals_two_calls(spl, x_rows, noise_rows, cols, mech, eps):
    """The left operand of the stacked product in one launch is, bit for bit, the mask + split of X's
    rows and the split of the noise rows drawn further on, as two separate calls make them."""
    eps = float("inf") if eps is None else eps
    X = dev(wl.activations(x_rows, cols, seed=x_rows + cols + 1).numpy())
    rows = x_rows + noise_rows
    base = torch.tensor([777], dtype=torch.int64, device="cuda")
    delta = 8 * 512 * cols // 4
    hi_ref = torch.zeros((rows, cols), dtype=torch.int16, device="cuda")
    lo_ref, ex_ref = torch.zeros_like(hi_ref), torch.zeros(rows, dtype=torch.int32, device="cuda")
    if x_rows:
        spl.spl_noise_mask_split(None, hi_ref[:x_rows], lo_ref[:x_rows], ex_ref[:x_rows], X, 825.3, eps, mech, seed=5,
                                 stream_id=1, offset=13, offset_dev=base)
    if noise_rows:
        spl.spl_noise_mask_split(None, hi_ref[x_rows:], lo_ref[x_rows:], ex_ref[x_rows:], None, 825.3, eps, mech,
                                 seed=5, stream_id=1, offset=13 + delta, offset_dev=base)
    hi, lo, ex = torch.full_like(hi_ref, 7), torch.full_like(lo_ref, 7), torch.full_like(ex_ref, 7)
    spl.spl_noise_mask_split_stacked(hi, lo, ex, X, 825.3, eps, mech, 5, noise_rows, delta, stream_id=1, offset=13,
                                     offset_dev=base)
    assert torch.equal(hi, hi_ref) and torch.equal(lo, lo_ref) and torch.equal(ex, ex_ref)


@pytest.mark.parametrize("rows,cols,mech", [(5, 8, "laplace"), (130, 3072, "gaussian"), (3, 16384, "laplace")])
def test_mask_split_with_stored_noise_equals_drawn(spl, rows, cols, mech):
    """The mask with a noise drawn earlier (as a bank refill keeps it) gives the X~ and the fp16
    split that drawing the noise in the same pass gives, bit for bit."""
    X = dev(wl.activations(rows, cols, seed=rows + 7 * cols).numpy())
    N = torch.empty_like(X)
    spl.spl_noise(N, 825.3, 0.5, mech, seed=23, stream_id=1, offset=77)
    ref_xt = torch.empty_like(X)
    hi_ref = torch.empty(X.shape, dtype=torch.int16, device="cuda")
    lo_ref, ex_ref = torch.empty_like(hi_ref), torch.empty(rows, dtype=torch.int32, device="cuda")
    spl.spl_noise_mask_split(ref_xt, hi_ref, lo_ref, ex_ref, X, 825.3, 0.5, mech, seed=23, stream_id=1, offset=77)
    xt = torch.empty_like(X)
    hi, lo, ex = torch.empty_like(hi_ref), torch.empty_like(lo_ref), torch.empty_like(ex_ref)
    spl.spl_mask_split(xt, hi, lo, ex, X, N)
    assert torch.equal(xt, ref_xt) and torch.equal(hi, hi_ref) and torch.equal(lo, lo_ref) and torch.equal(ex, ex_ref)
    spl.spl_mask_split(None, hi, lo, ex, X, N)  # no X~ out
    assert torch.equal(hi, hi_ref) and torch.equal(ex, ex_ref)
    # the noise a bank keeps: spl_noise_mask_split with X NULL writes it to Xt
    keep = torch.empty_like(X)
    spl.spl_noise_mask_split(keep, hi, lo, ex, None, 825.3, 0.5, mech, seed=23, stream_id=1, offset=77)
    assert torch.equal(keep, N)


@pytest.mark.parametrize("M,K,N,mech,eps", [(1, 3072, 3072, "laplace", 1.0), (2, 1028, 600, "gaussian", 0.5),
                                             (3, 8192, 520, "laplace", None), (4, 2560, 2056, "gaussian", 1.0),
                                             (5, 516, 300, "laplace", 1.0), (16, 3072, 512, "gaussian", 1.0)])
def test_noise_mask_linear_unmask_equals_separate_calls(spl, M, K, N, mech, eps):
    """The decode call with the mask drawn inside the product (M <= 4; two launches beyond) gives
    the X~ of spl_noise_mask and the Y of spl_masked_linear_unmask bit for bit, and both match the
    oracle: X~ within the noise tolerance, Y within the FP32 product bound of that X~."""
    W, Wt = _weights(spl, N, K, seed=N + K)
    X = wl.activations(M, K, seed=M + 21).numpy()
    C = dev(wl.activations(M, N, seed=M + 22).numpy())
    base = torch.tensor([500], dtype=torch.int64, device="cuda")
    ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N, "fp32"))
    xt_ref, Y_ref = torch.empty((M, K), device="cuda"), torch.empty((M, N), device="cuda")
    spl.spl_noise_mask(xt_ref, None, dev(X), 825.3, eps, mech, seed=23, stream_id=1, offset=500 + 12)
    spl.spl_masked_linear_unmask(Y_ref, xt_ref, Wt, C, path="fp32", workspace=ws)
    xt, Y = torch.full((M, K), 7.0, device="cuda"), torch.full((M, N), 7.0, device="cuda")
    n0 = spl.spl_launch_count()
    spl.spl_noise_mask_linear_unmask(Y, xt, dev(X), Wt, C, 825.3, eps, mech, seed=23, stream_id=1, offset=12,
                                     path="fp32", workspace=ws, offset_dev=base)
    torch.cuda.synchronize()
    assert spl.spl_launch_count() - n0 == (1 if M <= 4 else 2)
    assert torch.equal(xt, xt_ref) and torch.equal(Y, Y_ref)
    # against the oracle: X~ = fl32(X + eta) with the oracle's eta (a few ulps of the transcendentals)
    n_exp = philox.noise((M, K), 825.3, math.inf if eps is None else eps, mech, 23, 1, 512).astype(np.float64)
    xt_exp = linear.mask(X, n_exp.astype(np.float32)).astype(np.float64)
    tol = 2 * ulp32(xt_exp) + 8 * ulp32(n_exp)
    if mech == "gaussian" and eps is not None:
        tol = tol + 8 * U * float(np.float32(825.3 / eps)) * philox.radius_fp64((M, K), 23, 1, 512)
    assert np.all(np.abs(f64(xt) - xt_exp) <= tol)
    assert_product_close(f32(Y), f32(xt), W, "fp32", C=f32(C), what="fused decode call")
    Xd = dev(X)
    with pytest.raises(spl.SplError) as e:  # X~ may not overwrite X: other blocks still read it
        spl.spl_noise_mask_linear_unmask(Y, Xd, Xd, Wt, C, 825.3, eps, mech, seed=23, path="fp32", workspace=ws)
    assert e.value.status == spl.SPL_EINVAL


@pytest.mark.parametrize("M,M_bank,K,N,mech,eps", [(1, 1, 3072, 5120, "laplace", 1.0), (2, 2, 8192, 3072, "gaussian", 1.0),
                                                  (1, 3, 1032, 600, "laplace", None), (0, 2, 3072, 1000, "gaussian", 0.5),
                                                  (3, 0, 264, 300, "laplace", 0.5), (1, 1, 9728, 3072, "gaussian", 1.0)])
def test_stacked_decode_call_equals_separate_calls(spl, M, M_bank, K, N, mech, eps):
    """The stacked decode step in one launch: the X~ rows of spl_noise_mask, the noise rows of spl_noise
    drawn noise_block_delta blocks further on, and the product of spl_masked_linear_unmask_precompute on
    that operand, bit for bit; X~ and the noise against the oracle's draw, every output row within the
    FP32 product bound of the operand the kernel wrote."""
    W, Wt = _weights(spl, N, K, seed=N + K + 1)
    rows = M + M_bank
    X = wl.activations(max(M, 1), K, seed=M + 31).numpy()[:M]
    C = dev(wl.activations(max(M, 1), N, seed=M + 32).numpy()[:M]) if M else None
    base = torch.tensor([300], dtype=torch.int64, device="cuda")
    delta = 8 * K // 4 + 5
    ws = spl.workspace(spl.spl_linear_workspace_bytes(rows, K, N, "fp32"))
    xt_ref, YC_ref = torch.zeros((rows, K), device="cuda"), torch.empty((rows, N), device="cuda")
    if M:
        spl.spl_noise_mask(xt_ref[:M], None, dev(X), 825.3, eps, mech, seed=23, stream_id=2, offset=300 + 9)
    if M_bank:
        spl.spl_noise(xt_ref[M:], 825.3, eps, mech, seed=23, stream_id=2, offset=300 + 9 + delta)
    spl.spl_masked_linear_unmask_precompute(YC_ref, spl.Weight(xt_ref), Wt, C, M, path="fp32", workspace=ws)
    xt, YC = torch.full((rows, K), 7.0, device="cuda"), torch.full((rows, N), 7.0, device="cuda")
    n0 = spl.spl_launch_count()
    spl.spl_noise_mask_linear_unmask_precompute(YC, xt, dev(X) if M else None, Wt, C, 825.3, eps, mech, 23, M_bank,
                                                delta, stream_id=2, offset=9, path="fp32", workspace=ws,
                                                offset_dev=base)
    torch.cuda.synchronize()
    assert spl.spl_launch_count() - n0 == 1
    assert torch.equal(xt, xt_ref) and torch.equal(YC, YC_ref)
    e = math.inf if eps is None else eps
    n_exp = np.zeros((rows, K))
    if M:
        n_exp[:M] = philox.noise((M, K), 825.3, e, mech, 23, 2, 309)
    if M_bank:
        n_exp[M:] = philox.noise((M_bank, K), 825.3, e, mech, 23, 2, 309 + delta)
    xt_exp = n_exp.copy()
    if M:
        xt_exp[:M] = linear.mask(X, n_exp[:M].astype(np.float32))
    tol = 2 * ulp32(xt_exp) + 8 * ulp32(n_exp)
    if mech == "gaussian" and eps is not None:
        r = np.zeros((rows, K))
        if M:
            r[:M] = philox.radius_fp64((M, K), 23, 2, 309)
        if M_bank:
            r[M:] = philox.radius_fp64((M_bank, K), 23, 2, 309 + delta)
        tol = tol + 8 * U * float(np.float32(825.3 / eps)) * r
    assert np.all(np.abs(f64(xt) - xt_exp) <= tol)
    if M:
        assert_product_close(f32(YC[:M]), f32(xt[:M]), W, "fp32", C=f32(C), what="masked rows")
    if M_bank:
        assert_product_close(f32(YC[M:]), f32(xt[M:]), W, "fp32", what="correction rows")
    assert spl.spl_get_device_status() == 0


@pytest.mark.parametrize("M,M_bank,K,N", [(1, 1, 3072, 5120), (8, 8, 8192, 3072), (0, 5, 1032, 600), (4, 0, 264, 300),
                                          (3, 9, 9728, 3072)])
def test_precompute_on_the_decode_kernel(spl, M, M_bank, K, N):
    """spl_masked_linear_unmask_precompute at up to 16 rows on FP32 runs the decode kernel: every row
    summed as the same row of a plain product of M + M_bank rows, C subtracted from the first M only."""
    W, Wt = _weights(spl, N, K, seed=K + N + 7)
    rows = M + M_bank
    A = (wl.activations(rows, K, seed=rows + 5).numpy() * 300).astype(np.float32)
    C = wl.activations(max(M, 1), N, seed=11).numpy()[:M]
    ws = spl.workspace(spl.spl_linear_workspace_bytes(rows, K, N, "fp32"))
    YC = torch.full((rows, N), float("nan"), device="cuda")
    spl.spl_masked_linear_unmask_precompute(YC, spl.Weight(dev(A)), Wt, dev(C) if M else None, M, path="fp32",
                                            workspace=ws)
    if M:
        assert_product_close(f32(YC[:M]), A[:M], W, "fp32", C=C, what="masked rows")
    if M_bank:
        assert_product_close(f32(YC[M:]), A[M:], W, "fp32", what="correction rows")
    P = torch.empty((rows, N), device="cuda")
    spl.spl_masked_linear(P, dev(A), Wt, path="fp32", workspace=ws)
    assert torch.equal(YC[M:], P[M:])
    if M:
        Yu = torch.empty((M, N), device="cuda")
        spl.spl_unmask(Yu, P[:M].contiguous(), dev(C))
        assert torch.equal(YC[:M], Yu)
    assert spl.spl_get_device_status() == 0


@pytest.mark.parametrize("rows,cols,mech,eps", [(1024, 3072, "gaussian", 1.0), (37, 1032, "laplace", 0.5),
                                                (8, 8192, "laplace", None)])
def test_noise_split_is_the_split_of_the_noise(spl, rows, cols, mech, eps):
    """With no input the fused kernel splits the noise itself: the same bits as spl_noise then
    spl_split_fp16 (eps = inf: the split of zeros)."""
    eta = torch.empty((rows, cols), device="cuda")
    spl.spl_noise(eta, 825.3, eps, mech, seed=5, stream_id=3, offset=77)
    hi_ref = torch.empty((rows, cols), dtype=torch.int16, device="cuda")
    lo_ref, ex_ref = torch.empty_like(hi_ref), torch.empty(rows, dtype=torch.int32, device="cuda")
    spl.spl_split_fp16(hi_ref, lo_ref, ex_ref, eta)
    hi, lo, ex = torch.empty_like(hi_ref), torch.empty_like(lo_ref), torch.empty_like(ex_ref)
    xt = torch.full((rows, cols), 3.0, device="cuda")
    spl.spl_noise_mask_split(xt, hi, lo, ex, None, 825.3, eps, mech, seed=5, stream_id=3, offset=77)
    assert torch.equal(hi, hi_ref) and torch.equal(lo, lo_ref) and torch.equal(ex, ex_ref)
    assert torch.equal(xt, eta)  # X~ of no input is the noise


@pytest.mark.parametrize("M,K,N,order", [(1024, 3072, 5120, 128), (1024, 8192, 3072, 128), (400, 1032, 600, 100),
                                         (4096, 3072, 3072, 512)])
def test_matched_correction_from_the_split_noise(spl, M, K, N, order):
    """The bank's correction from the noise split as drawn equals the one from the fp32 noise, bit
    for bit, and so the online order."""
    W, Wt = _weights(spl, N, K, seed=K + N + 5)
    eta = torch.empty((M, K), device="cuda")
    spl.spl_noise(eta, 1443.0, 1.0, "gaussian", seed=29)
    hi = torch.empty((M, K), dtype=torch.int16, device="cuda")
    lo, ex = torch.empty_like(hi), torch.empty(M, dtype=torch.int32, device="cuda")
    spl.spl_noise_mask_split(None, hi, lo, ex, None, 1443.0, 1.0, "gaussian", seed=29)
    ws = spl.workspace(spl.spl_precompute_matched_workspace_bytes(M, K, N, order, "fp16x3"))
    C_ref, C, C_w = (torch.empty((M, N), device="cuda") for _ in range(3))
    spl.spl_precompute_noise_product_matched(C_ref, eta, Wt, order, path="fp16x3", workspace=ws)
    spl.spl_precompute_noise_product_matched_split(C, spl.Weight(None, f16_hi=hi, f16_lo=lo, f16_exp=ex), Wt, order,
                                                   path="fp16x3", workspace=ws)
    assert torch.equal(C, C_ref)
    # the FP32 path reads the fp32 noise of the descriptor
    ws32 = spl.workspace(spl.spl_precompute_matched_workspace_bytes(M, K, N, 1, "fp32"))
    C32_ref = torch.empty((M, N), device="cuda")
    spl.spl_precompute_noise_product_matched(C32_ref, eta, Wt, 1, path="fp32", workspace=ws32)
    spl.spl_precompute_noise_product_matched_split(C_w, spl.Weight(eta, f16_hi=hi, f16_lo=lo, f16_exp=ex), Wt, 1,
                                                   path="fp32", workspace=ws32)
    assert torch.equal(C_w, C32_ref)
    with pytest.raises(spl.SplError) as e:  # ... and refuses a descriptor without it
        spl.spl_precompute_noise_product_matched_split(C_w, spl.Weight(None, f16_hi=hi, f16_lo=lo, f16_exp=ex), Wt, 1,
                                                       path="fp32", workspace=ws32)
    assert e.value.status == spl.SPL_EINVAL
    assert spl.spl_get_device_status() == 0


@pytest.mark.parametrize("M,K,N", [(128, 3072, 3072), (130, 1032, 600), (512, 3072, 5120), (9, 256, 512)])
def test_presplit_product_equals_plain(spl, M, K, N):
    W, Wt = _weights(spl, N, K, seed=N + 3)
    X = dev(wl.activations(M, K, seed=M + 4).numpy())
    C = dev(wl.activations(M, N, seed=5).numpy())
    xt = torch.empty_like(X)
    hi = torch.empty(X.shape, dtype=torch.int16, device="cuda")
    lo, ex = torch.empty_like(hi), torch.empty(M, dtype=torch.int32, device="cuda")
    spl.spl_noise_mask_split(xt, hi, lo, ex, X, 825.3, 1.0, "gaussian", seed=7)
    ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N))
    Y_plain, Y_split, Y_none = (torch.empty((M, N), device="cuda") for _ in range(3))
    spl.spl_masked_linear_unmask(Y_plain, xt, Wt, C, path="fp16x3", workspace=ws)
    spl.spl_masked_linear_unmask_split(Y_split, spl.Weight(xt, f16_hi=hi, f16_lo=lo, f16_exp=ex), Wt, C,
                                       path="fp16x3", workspace=ws)
    # the split operand needs no room for its split: the kernels that reduce on chip take no workspace,
    # the swapped kernel of 9-16 rows only its counters and partial tiles
    need = spl.spl_split_workspace_bytes(M, K, N, path="fp16x3")
    assert (need > 0) == (M <= 16)
    assert need < spl.spl_linear_workspace_bytes(M, K, N, "fp16x3") or need == 0
    spl.spl_masked_linear_unmask_split(Y_none, spl.Weight(None, f16_hi=hi, f16_lo=lo, f16_exp=ex), Wt, C,
                                       path="fp16x3", workspace=spl.workspace(need) if need else None)
    assert torch.equal(Y_plain, Y_split) and torch.equal(Y_plain, Y_none)
    if need:
        with pytest.raises(spl.SplError) as e:  # the partial tiles need their room
            spl.spl_masked_linear_unmask_split(Y_none, spl.Weight(None, f16_hi=hi, f16_lo=lo, f16_exp=ex), Wt, C,
                                               path="fp16x3", workspace=None)
        assert e.value.status == spl.SPL_EWORKSPACE
    with pytest.raises(spl.SplError) as e:  # FP32 reads the fp32 X~, which is absent
        spl.spl_masked_linear_unmask_split(Y_none, spl.Weight(None, f16_hi=hi, f16_lo=lo, f16_exp=ex), Wt, C,
                                           path="fp32", workspace=ws)
    assert e.value.status == spl.SPL_EINVAL


# ------------------------------------------------ binary64 path (Sec. 5.5, the Down projection)
U53 = 2.0 ** -53


def test_noise_mask_f64_matches_oracle(spl):
    X = dev(wl.activations(37, 1028, seed=61).numpy())
    eta = torch.empty_like(X)
    spl.spl_noise(eta, 2.6e8, 1.0, "laplace", seed=62, stream_id=3, offset=17)
    Xt = torch.empty(X.shape, dtype=torch.float64, device="cuda")
    spl.spl_noise_mask_f64(Xt, X, 2.6e8, 1.0, "laplace", seed=62, stream_id=3, offset=17)
    np.testing.assert_array_equal(Xt.cpu().numpy(), linear.mask_f64(f32(X), f32(eta)))


@pytest.mark.parametrize("M,K,N", [(1, 256, 64), (3, 1028, 300), (8, 8192, 512), (13, 3072, 700), (128, 3072, 256)])
def test_f64_products_match_oracle(spl, M, K, N):
    """C = eta W^T and Y = fl32(X~ W^T - C) in binary64 against the exact products (oracle)."""
    W = wl.weight(N, K, seed=M + K).numpy()
    X = wl.activations(M, K, seed=M + 1).numpy()
    eta = philox.noise((M, K), 2.6e8, 1.0, "gaussian", seed=M + 2)
    Wd = dev(W)
    C = torch.empty((M, N), dtype=torch.float64, device="cuda")
    ws = spl.workspace(spl.spl_f64_workspace_bytes(M, K, N) + 64 * 1024)
    spl.spl_precompute_noise_product_f64(C, dev(eta), Wd, workspace=ws)
    Cref = linear.precompute_noise_product(eta, W)
    S_n = np.abs(eta.astype(np.float64)) @ np.abs(W.astype(np.float64)).T
    assert np.all(np.abs(C.cpu().numpy() - Cref) <= 2 * bounds.gamma(K, U53) * S_n)
    Xt = dev(linear.mask_f64(X, eta))
    Y = torch.empty((M, N), device="cuda")
    spl.spl_masked_linear_unmask_f64(Y, Xt, Wd, C, workspace=ws)
    ref = linear.reference_output(X, W)
    S = linear.abs_products(X, linear.mask_f64(X, eta), eta, W)
    tol = bounds.hard_bound(*S, K, u=U53) + bounds.gamma(K, U53) * S[0] + 2.0 ** -24 * np.abs(ref) * (1 + 2.0 ** -20)
    assert np.all(np.abs(f64(Y) - ref) <= tol)
    assert torch.count_nonzero(ws[: 64 * 1024]).item() == 0  # the decode counters stay untouched
    assert spl.spl_get_device_status() == 0


def test_f64_down_recovers_what_binary32_cannot(spl):
    """Llama Down shapes, Delta from Thm. 3 (~2.6e8): in binary32 the mask alone rounds away the
    input; the binary64 path recovers X W^T to a few ulps of fp32."""
    M, K, N = 4, 8192, 512
    W = wl.weight(N, K, seed=71).numpy()
    X = wl.activations(M, K, seed=72).numpy()
    delta, eps = 2.6e8, 1.0
    eta = torch.empty((M, K), device="cuda")
    spl.spl_noise(eta, delta, eps, "laplace", seed=73)
    Xd, Wd = dev(X), dev(W)
    ref = linear.reference_output(X, W)
    # binary64
    C64 = torch.empty((M, N), dtype=torch.float64, device="cuda")
    Xt64 = torch.empty((M, K), dtype=torch.float64, device="cuda")
    spl.spl_precompute_noise_product_f64(C64, eta, Wd)
    spl.spl_noise_mask_f64(Xt64, Xd, delta, eps, "laplace", seed=73)
    Y64 = torch.empty((M, N), device="cuda")
    spl.spl_masked_linear_unmask_f64(Y64, Xt64, Wd, C64)
    err64 = np.abs(f64(Y64) - ref)
    assert np.max(err64) <= 4 * 2.0 ** -24 * np.max(np.abs(ref))
    # binary32, same noise
    Wt = spl.Weight.prepare(Wd)
    C32 = torch.empty((M, N), device="cuda")
    Xt32 = torch.empty((M, K), device="cuda")
    ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N, "fp32"))
    spl.spl_precompute_noise_product(C32, eta, Wt, path="fp32", workspace=ws)
    spl.spl_noise_mask(Xt32, None, Xd, delta, eps, "laplace", seed=73)
    Y32 = torch.empty((M, N), device="cuda")
    spl.spl_masked_linear_unmask(Y32, Xt32, Wt, C32, path="fp32", workspace=ws)
    err32 = np.abs(f64(Y32) - ref)
    assert np.mean(err32) > 1e4 * np.mean(err64)


# ------------------------------------------------ Slalom comparator (Sec. 6.2)
@pytest.mark.parametrize("M,K,N", [(1, 256, 64), (5, 1028, 300), (16, 3072, 512), (128, 8192, 256)])
def test_slalom_matches_oracle_bitwise(spl, M, K, N):
    """Integer work end to end: quantized weights, the masked field elements, the exact
    correction and the de-quantized result all equal the oracle's bit for bit."""
    W = wl.weight(N, K, seed=K + 5).numpy()
    X = wl.activations(M, K, seed=M + 6).numpy()
    Wq = torch.empty((N, K), device="cuda")
    spl.spl_slalom_quantize(Wq, dev(W))
    np.testing.assert_array_equal(f64(Wq), slalom.quantize(W).astype(np.float64))
    Xt = torch.empty((M, K), device="cuda")
    eta = torch.empty((M, K), device="cuda")
    spl.spl_slalom_mask(Xt, eta, dev(X), seed=77, stream_id=2, offset=5)
    eta_or = slalom.mask_noise((M, K), seed=77, stream_id=2, offset=5)
    np.testing.assert_array_equal(f64(eta), eta_or.astype(np.float64))
    np.testing.assert_array_equal(f64(Xt), slalom.mask(X, eta_or).astype(np.float64))
    ws = spl.workspace(spl.spl_f64_workspace_bytes(M, K, N) + 64 * 1024)
    C = torch.empty((M, N), dtype=torch.float64, device="cuda")
    spl.spl_precompute_noise_product_f64(C, eta, Wq, workspace=ws)
    np.testing.assert_array_equal(C.cpu().numpy(), slalom.product(eta_or, slalom.quantize(W)).astype(np.float64))
    Y = torch.empty((M, N), device="cuda")
    spl.spl_slalom_linear_unmask(Y, Xt, Wq, C, workspace=ws)
    np.testing.assert_array_equal(f64(Y), slalom.masked_linear(X, W, eta_or))


# ---------------------------------------------------------- a8: bound on the GPU, path choice
def test_bound_check_matches_oracle(spl):
    M, K, N = 24, 1028, 300
    X = wl.activations(M, K, seed=3).numpy()
    eta = philox.noise((M, K), 50.0, 1.0, "gaussian", 9)
    Xt = linear.mask(X, eta)
    W, Wt = _weights(spl, N, K, seed=4)
    Wd = Wt.w
    C = torch.empty((M, N), device="cuda")
    Y = torch.empty((M, N), device="cuda")
    ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N, "fp32"))
    spl.spl_precompute_noise_product(C, dev(eta), Wd, path="fp32", workspace=ws)
    spl.spl_masked_linear_unmask(Y, dev(Xt), Wd, C, path="fp32", workspace=ws)
    got = spl.spl_bound_check(Y, dev(X), dev(Xt), dev(eta), Wd)
    S = linear.abs_products(X, Xt, eta, W)
    err = np.abs(f64(Y) - linear.reference_output(X, W))
    hard, logb = bounds.hard_bound(*S, K), bounds.log_bound(*S, K)
    assert got["elements"] == M * N
    assert got["max_err_over_hard"] == pytest.approx(float(np.max(err / hard)), rel=1e-9)
    assert got["max_err_over_log"] == pytest.approx(float(np.max(err / logb)), rel=1e-9)
    assert abs(got["log_violations"] - float(np.sum(err > logb))) <= 1
    assert got["sum_err"] == pytest.approx(float(err.sum()), rel=1e-9)
    assert got["sum_log_bound"] == pytest.approx(float(logb.sum()), rel=1e-12)
    assert got["sum_hard_bound"] == pytest.approx(float(hard.sum()), rel=1e-12)
    assert got["max_abs_ref"] == pytest.approx(float(np.max(np.abs(linear.reference_output(X, W)))), rel=1e-12)


@pytest.mark.parametrize("K,N", [(3072, 3072), (8, 64), (1028, 512)])
def test_choose_path_follows_its_rule(spl, K, N):
    rows = 128
    X = dev(wl.activations(rows, K, seed=5).numpy())
    eta = torch.empty((rows, K), device="cuda")
    spl.spl_noise(eta, 2 * 3072 ** 0.75, 1.0, "gaussian", seed=6)
    W, Wt = _weights(spl, N, K, seed=7)
    name, st = spl.spl_choose_path(X, eta, Wt)
    fp = st["fp32"]

    def ok(s):
        return (s["max_err_over_hard"] <= 1.0 and s["log_violations"] <= fp["log_violations"] + 0.01 * s["elements"]
                and s["sum_err"] <= 1.5 * fp["sum_err"] + 1e-300)

    expect = "fp16x3" if ok(st["fp16x3"]) else ("tf32x3" if ok(st["tf32x3"]) else "fp32")
    assert name == expect
    assert fp["max_err_over_hard"] <= 1.0 and fp["elements"] == rows * N
    if K % 8:
        assert st["fp16x3"]["max_err_over_hard"] == float("inf")  # no fp16 split for K % 8 != 0
    if K >= 64:
        assert st["tf32x3"]["max_err_over_hard"] <= 1.0
        assert name == ("fp16x3" if K % 8 == 0 else "tf32x3")  # the split paths stay inside the bound at Llama sizes


# ---------------------------------------------------------- a1: ||W||_2
def test_spectral_norm_matches_svd(spl):
    W = wl.weight(300, 200, seed=9).numpy()
    got = spl.spl_spectral_norm(dev(W), iters=300)
    assert got == pytest.approx(np.linalg.svd(W.astype(np.float64), compute_uv=False)[0], rel=2e-4)


# --------------------------------------------------- end to end, config "single"
def _run_path(spl, X, W, Wt, sens, eps, mech, seed, path):
    M, K = X.shape
    N = W.shape[0]
    Xt = torch.empty((M, K), device="cuda")
    Nz = torch.empty((M, K), device="cuda")
    spl.spl_noise_mask(Xt, Nz, dev(X), sens, eps, mech, seed=seed)
    ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N, path))
    C = torch.empty((M, N), device="cuda")
    spl.spl_precompute_noise_product(C, Nz, Wt, path=path, workspace=ws)
    Y = torch.empty((M, N), device="cuda")
    spl.spl_masked_linear_unmask(Y, Xt, Wt, C, path=path, workspace=ws)
    return Y


def _hard_check(Y, X, W, sens, eps, mech, seed):
    """|Y - X W^T| within the hard bound built from the oracle's own eta."""
    n_or = philox.noise(X.shape, sens, eps, mech, seed)
    xt_or = linear.mask(X, n_or)
    S_x, S_xt, S_n = linear.abs_products(X, xt_or, n_or, W)
    K = X.shape[1]
    hb = bounds.hard_bound(S_x, S_xt, S_n, K) * (1 + 1e-5)
    err = np.abs(f64(Y) - linear.reference_output(X, W))
    assert np.all(err <= hb), float(np.max(err / hb))
    return err, (S_x, S_xt, S_n)


@pytest.mark.parametrize("path", ["fp32", "tf32x3", "fp16x3"])
def test_config_single_masked_linear(spl, path):
    cfg = wl.CONFIGS["single"]
    M, K, N = cfg["M"], cfg["K"], cfg["N"]
    X = wl.activations(M, K, seed=cfg["seed"], norm="unit").numpy()
    W, Wt = _weights(spl, N, K, seed=cfg["seed"] + 1)
    for eps in cfg["eps"]:
        Y = _run_path(spl, X, W, Wt, cfg["sensitivity"], eps, cfg["mech"], cfg["seed"], path)
        _hard_check(Y, X, W, cfg["sensitivity"], eps, cfg["mech"], cfg["seed"])
        if math.isinf(eps):
            Yref = linear.reference_output(X, W)
            assert linear.max_relative_error(f64(Y), Yref) <= 1e-5
            plain = torch.empty((M, N), device="cuda")
            spl.spl_masked_linear(plain, dev(X), Wt, path=path,
                                  workspace=spl.workspace(spl.spl_linear_workspace_bytes(M, K, N, path)))
            assert torch.equal(plain, Y)  # zero noise: C = 0 and X~ = X, so unmask(r) is the plain product


# ------------------------------------------- end to end, one Llama layer (M=128)
@pytest.fixture(scope="module")
def llama_layer(spl):
    from paper_2609_15039_gb300.layer import MaskedLayer
    from oracle import sensitivity as osens
    model = wl.LLAMA_3_2_3B
    weights = {name: wl.weight(N, K, seed=200 + pi) for pi, (name, K, N, g) in enumerate(model.projections())}
    layer = MaskedLayer.from_weights(model, weights)
    ones = np.ones(model.d_model)
    # ||W||_2 from LAPACK's singular values (a library routine), exact to rounding
    norms = {n: float(np.linalg.svd(weights[n].double().numpy(), compute_uv=False)[0]) for n in ("v", "up", "gate")}
    deltas = {  # noise scales from the oracle: an input both sides get
        "qkv": osens.delta_layernorm(ones),
        "gateup": osens.delta_layernorm(ones),
        "o": osens.delta_attention(ones, norms["v"]),
        "down": osens.delta_activation(ones, None, model.d_ff, norms["up"], norms["gate"]),
    }
    return layer, weights, deltas, norms


def test_layer_sensitivities_match_oracle(llama_layer):
    layer, _weights_, deltas, norms = llama_layer
    # power iteration approaches ||W||_2 from below; 1000 steps bring it within 1e-5 on these
    # Gaussian matrices, whose top singular values are close together
    got = layer.sensitivities(power_iters=1000)
    for g in deltas:
        assert got[g] <= deltas[g] * (1 + 1e-5), g
        assert got[g] == pytest.approx(deltas[g], rel=1e-4), g
    assert got["qkv"] == pytest.approx(2 * 3072 ** 0.75, rel=1e-9)


@pytest.mark.parametrize("eps", [0.5, 1.0, 4.0])
def test_config_llama_layer(spl, llama_layer, eps):
    from paper_2609_15039_gb300.layer import split_outputs
    layer, weights, deltas, _norms = llama_layer
    layer.deltas = dict(deltas)
    model, M, mech, seed, draws = layer.model, wl.CONFIGS["llama_layer"]["M"], "gaussian", 31, 2
    layer.allocate(M, draws)
    inputs_np = {g: wl.activations(M, K, seed=100 + gi).numpy() for gi, (g, K, _n) in enumerate(model.input_groups())}
    inputs = {g: dev(x) for g, x in inputs_np.items()}
    layer.refill(eps, mech, seed, cycle=3)
    # the bank keeps the noise (or, for an FP16X3 group, only its fp16 split)
    bank = {g.name: (layer.bank[g.name]["es"].f16_hi.clone() if "es" in layer.bank[g.name]
                     else layer.bank[g.name]["eta"].clone()) for g in layer.groups}
    for d in range(draws):
        outs = split_outputs(layer, layer.online(inputs, eps, mech, seed, cycle=3, d=d))
        torch.cuda.synchronize()
        for gi, g in enumerate(layer.groups):
            # the online step regenerates exactly the bank's mask of draw d
            regen = torch.empty((M, g.K), device="cuda")
            xt = torch.empty((M, g.K), device="cuda")
            spl.spl_noise_mask(xt, regen, inputs[g.name], deltas[g.name], eps, mech, seed, stream_id=gi,
                                   offset=layer.block_offset(g, 3, d))
            if "es" in layer.bank[g.name]:
                hi, lo = torch.empty((M, g.K), dtype=torch.int16, device="cuda"), None
                lo, ex = torch.empty_like(hi), torch.empty(M, dtype=torch.int32, device="cuda")
                spl.spl_split_fp16(hi, lo, ex, regen)
                assert torch.equal(hi, bank[g.name][d * M:(d + 1) * M])
            else:
                assert torch.equal(regen, bank[g.name][d * M:(d + 1) * M])
            X = inputs_np[g.name]
            n_or = philox.noise((M, g.K), deltas[g.name], eps, mech, seed, stream_id=gi,
                                offset=layer.block_offset(g, 3, d))
            xt_or = linear.mask(X, n_or)
            for name in g.names:
                W = weights[name].numpy()
                S = linear.abs_products(X, xt_or, n_or, W)
                err = np.abs(f64(outs[name]) - linear.reference_output(X, W))
                hb = bounds.hard_bound(*S, g.K) * (1 + 1e-5)
                assert np.all(err <= hb), (name, d, float(np.max(err / hb)))
                st = bounds.bound_statistics(err, bounds.log_bound(*S, g.K))
                assert st["ratio"] > 1.0, (name, st)
