"""Zero-noise parity at the stacks' full reduction lengths (the noise-free configuration, eps = inf).

With eps = inf the noise is exactly zero (Sec. 4.4's scale Delta/eps is 0), so x~ = x, the correction
is 0 and the recovered output is the plain product X W^T: every launch form must reach it within a
max-norm relative error of 1e-5 (max |Y - Y*| / max |Y*|, Y* the exact product from the oracle).

That tolerance, unlike the worst-case bound gamma_K S, tells the split arithmetic apart from a
downgraded one.  With a = a_hi + a_lo (11 + 11 significant bits), dropping a cross product a_lo w_hi
leaves a per-term error uniform in +-2^-12 |a w|, whose sum over K terms has a standard deviation of
2^-12/sqrt(3) tau = 296 x 2^-21 tau, tau = sqrt(sum_k (a_k w_k)^2) the root sum of squares of the
terms; with random-signed terms |Y*| is of order tau too, so that is ~1.4e-4 relative -- fourteen times
the tolerance -- and dropping all of a_lo is worse still.

The per-element check below is mean |Y - Y*| / (2^-21 tau) <= 16.  A correct three-product split
contributes ~0.2; what dominates is the tensor core's accumulation, which truncates: on GB300 one
unbroken chain of FP16X3 MMAs leaves a bias toward zero of 0.0059 per element of K in these units
(TF32X3: 0.0117), which is why the kernels cut every chain at 1024 (FP16X3) or 512 (TF32X3) elements
of K and fold the pieces with round-to-nearest adds -- at most ~6 whatever K is.  The FP32 FMA path
(sequential round-to-nearest) stays near 0.5.  A split that lost a cross product reads ~236, fifteen
times the limit.

Launch forms covered: every tile width / ring of the tensor-core kernel, cluster K-splits 1..8, the
two-launch shape (whole waves unsplit + the rest split), the persistent kernel, the segmented (bank)
form, and the decode kernel; then the production paths of the Llama and Qwen layers at their own
sizes through MaskedLayer (noise + mask + split, bank, product with fused unmask), on sampled
outputs.  Reduction lengths: 2560 and 9728 (Qwen), 3072 and 8192 (Llama).
"""

import numpy as np
import pytest
import torch

from oracle import bounds, linear
from paper_2609_15039_gb300 import workloads as wl
from _util import f32

pytestmark = pytest.mark.gpu

REL_TOL = 1e-5
TC_VARIANTS = [(256, 192), (128, 224), (128, 96), (160, 224), (192, 224), (224, 224)]
FULL_K = [2560, 3072, 8192, 9728]


STAT_LIMIT = 16.0


@pytest.fixture(scope="module")
def spl():
    from paper_2609_15039_gb300 import spl as binding
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    binding.lib()
    return binding


def dev(a):
    return torch.as_tensor(np.ascontiguousarray(a)).cuda()


def zero_noise_errors(Y, A, W):
    """(max-norm relative error, mean |err| / (2^-21 tau)) of Y against the exact A W^T."""
    ref = linear.reference_output(A, W)
    A64, W64 = A.astype(np.float64), W.astype(np.float64)
    tau = np.sqrt((A64 * A64) @ (W64 * W64).T)
    err = np.abs(np.asarray(Y, dtype=np.float64) - ref)
    rel = linear.max_relative_error(Y, ref)
    return rel, float(np.mean(err / np.maximum(tau * 2.0 ** -21, 1e-300)))


def check(Y, A, W, K, what):
    rel, stat = zero_noise_errors(Y, A, W)
    assert rel <= REL_TOL, f"{what}: max-norm relative error {rel:.3g} > {REL_TOL}"
    assert stat <= STAT_LIMIT, f"{what}: mean err / (2^-21 tau) = {stat:.3g} > {STAT_LIMIT}"
    return rel, stat


@pytest.fixture(scope="module")
def problems(spl):
    """Per K: A [200, K] (two row tiles, the second ragged), W [600, K] (ragged for every tile width)."""
    out = {}
    for K in FULL_K:
        A = wl.activations(200, K, seed=K + 1).numpy()
        W = wl.weight(600, K, seed=K + 2).numpy()
        out[K] = (A, W, spl.Weight.prepare(dev(W)))
    return out


@pytest.mark.parametrize("path", ["fp16x3", "tf32x3"])
@pytest.mark.parametrize("tile_n,ring_kb", TC_VARIANTS)
@pytest.mark.parametrize("K", FULL_K)
def test_every_tc_launch_form_at_full_k(spl, problems, K, path, tile_n, ring_kb):
    A, W, Wt = problems[K]
    M, N = A.shape[0], W.shape[0]
    Ad, Cd = dev(A), torch.zeros((M, N), device="cuda")
    tiles = -(-M // 128) * -(-N // tile_n)
    forms = [dict(splits=s) for s in range(1, 9)]
    forms.append(dict(splits=3, full_tiles=tiles // 2 + 1))  # two launches: unsplit tiles, then split ones
    forms += [dict(splits=1, seg_splits=s) for s in (2, 5, 8)]  # the bank's segmented form
    if ring_kb != 96:
        forms.append(dict(splits=1, persistent=True))
    worst = [0.0, 0.0]
    for form in forms:
        for C in (None, Cd):  # C = 0: the correction at eps = inf, subtracted in the epilogue
            Y = torch.full((M, N), float("nan"), device="cuda")
            spl.spl_test_tc_product(Y, Ad, Wt, C, path=path, tile_n=tile_n, ring_kb=ring_kb, **form)
            rel, stat = check(f32(Y), A, W, K, f"{path} {tile_n}/{ring_kb} {form} C={'0' if C is not None else 'none'}")
            worst = [max(worst[0], rel), max(worst[1], stat)]
    assert spl.spl_get_device_status() == 0


@pytest.mark.parametrize("K", FULL_K)
@pytest.mark.parametrize("tn", [16, 64, 128])
@pytest.mark.parametrize("ctas", [0, 1, 57])
def test_swap_forms_at_full_k(spl, problems, K, tn, ctas):
    """The swapped kernel of few rows (weight in the MMA's rows, tokens in its columns) at 40 tokens:
    the library's run length, one run over all of K (chains folded over whole tiles), and runs
    cutting tiles into pieces summed through the workspace."""
    A, W, Wt = problems[K]
    A = np.ascontiguousarray(A[:40])
    Y = torch.full((40, W.shape[0]), float("nan"), device="cuda")
    spl.spl_test_tc_swap_product(Y, dev(A), Wt, None, tile_tokens=tn, ctas=ctas)
    check(f32(Y), A, W, K, f"swap {tn} ctas {ctas}")


@pytest.mark.parametrize("K", FULL_K)
@pytest.mark.parametrize("M", [1, 4, 16, 200])
def test_fp32_paths_at_full_k(spl, problems, K, M):
    """The FP32 paths: the streaming decode kernel (M <= 16) and the FMA kernel (M = 200)."""
    A, W, Wt = problems[K]
    A = A[:M]
    N = W.shape[0]
    ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N, "fp32"))
    Y = torch.full((M, N), float("nan"), device="cuda")
    spl.spl_masked_linear_unmask(Y, dev(A), Wt, torch.zeros((M, N), device="cuda"), path="fp32", workspace=ws)
    check(f32(Y), A, W, K, f"fp32 M={M}")
    Y2 = torch.full((M, N), float("nan"), device="cuda")
    spl.spl_masked_linear(Y2, dev(A), Wt, path="fp32", workspace=ws)
    check(f32(Y2), A, W, K, f"fp32 masked_linear M={M}")


@pytest.mark.parametrize("M", [1, 4, 16, 64, 130])
@pytest.mark.parametrize("K", FULL_K)
def test_noise_free_call_chain(spl, problems, K, M):
    """eps = inf through the boundary's call chain: spl_noise_mask (zero noise, x~ = x bit for bit),
    the correction of the zero noise (exactly 0), the masked product with fused unmask (AUTO)."""
    A, W, Wt = problems[K]
    A = np.ascontiguousarray(A[:M])
    N = W.shape[0]
    Xd = dev(A)
    Xt, Nz = torch.empty_like(Xd), torch.empty_like(Xd)
    spl.spl_noise_mask(Xt, Nz, Xd, 825.3, float("inf"), "laplace", 3)
    assert torch.equal(Xt, Xd) and not torch.any(Nz).item()
    ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N))
    C = torch.full((M, N), float("nan"), device="cuda")
    spl.spl_precompute_noise_product(C, Nz, Wt, workspace=ws)
    assert not torch.any(C).item()
    Y = torch.full((M, N), float("nan"), device="cuda")
    spl.spl_masked_linear_unmask(Y, Xt, Wt, C, workspace=ws)
    check(f32(Y), A, W, K, f"AUTO M={M}")


def _layer(model, M, draws, seed):
    from paper_2609_15039_gb300.layer import MaskedLayer
    weights = {name: wl.weight(N, K, seed=wl.layer_seed(seed, 0, pi), device="cuda")
               for pi, (name, K, N, g) in enumerate(model.projections())}
    layer = MaskedLayer.from_weights(model, weights)
    layer.deltas = {g: 825.3 for g, _k, _n in model.input_groups()}  # any scale: eps = inf zeroes it
    layer.allocate(M, draws)
    inputs = {g: wl.activations(M, K, seed=wl.layer_seed(seed, 0, 50 + gi), device="cuda")
              for gi, (g, K, _n) in enumerate(model.input_groups())}
    return layer, inputs


@pytest.mark.parametrize("model_name,M", [("llama", 128), ("llama", 512), ("qwen", 2048), ("llama", 1)])
def test_layer_production_paths_noise_free(spl, model_name, M):
    """The workloads' layers at their own sizes, eps = inf, through the path the bench times (fused
    noise + mask + split, bank of corrections in the online order, AUTO launch shapes), checked on
    sampled outputs of every projection."""
    model = wl.LLAMA_3_2_3B if model_name == "llama" else wl.QWEN3_4B
    draws = 2
    layer, inputs = _layer(model, M, draws, seed=17)
    eps, mech, seed = float("inf"), "laplace", 5
    layer.refill(eps, mech, seed, cycle=0)
    outs = layer.online(inputs, eps, mech, seed, 0, 1)
    torch.cuda.synchronize()
    rng = np.random.default_rng(M)
    rows = np.sort(rng.choice(M, size=min(16, M), replace=False))
    ri = torch.as_tensor(rows, device="cuda")
    for g in layer.groups:
        X = inputs[g.name][ri].cpu().numpy()
        Yg = outs[g.name][ri].cpu().numpy()
        cols = np.sort(rng.choice(g.N, size=min(512, g.N), replace=False))
        W = g.W[torch.as_tensor(cols, device="cuda")].cpu().numpy()
        check(Yg[:, cols], X, W, g.K, f"{model_name} M={M} {g.name}")
    assert spl.spl_get_device_status() == 0


@pytest.mark.parametrize("model_name,M", [("llama", 512), ("qwen", 8), ("llama", 1), ("qwen", 1)])
def test_stacked_production_paths_noise_free(spl, model_name, M):
    """The stacked schedule the bench times, eps = inf: every call multiplies the step's M rows and the
    next cycle's M noise rows (here zero) -- 1024-row tensor-core calls (Llama 512), the swapped kernel
    at 16 rows (Qwen 8), the one-launch decode kernel at 2 rows (M = 1) -- and the noise rows' outputs,
    the next cycle's corrections, are exactly zero; sampled outputs of every projection within 1e-5."""
    from paper_2609_15039_gb300.layer import MaskedLayer
    model = wl.LLAMA_3_2_3B if model_name == "llama" else wl.QWEN3_4B
    weights = {name: wl.weight(N, K, seed=wl.layer_seed(19, 0, pi), device="cuda")
               for pi, (name, K, N, g) in enumerate(model.projections())}
    layer = MaskedLayer.from_weights(model, weights)
    layer.deltas = {g: 825.3 for g, _k, _n in model.input_groups()}
    layer.allocate_stacked(M, 2)
    inputs = {g: wl.activations(M, K, seed=wl.layer_seed(19, 0, 50 + gi), device="cuda")
              for gi, (g, K, _n) in enumerate(model.input_groups())}
    eps, mech, seed = float("inf"), "gaussian", 7
    for cycle in range(2):
        for d in range(2):
            outs = layer.stacked_step(inputs, eps, mech, seed, d, cycle % 2, cycle=cycle)
    torch.cuda.synchronize()
    rng = np.random.default_rng(M + 3)
    rows = np.sort(rng.choice(M, size=min(16, M), replace=False))
    ri = torch.as_tensor(rows, device="cuda")
    for g in layer.groups:
        full = layer.stacked[g.name]["out"][0][1]  # the last step (cycle 1, draw 1) wrote parity 0's buffer
        assert not torch.any(full[M:]).item(), g.name  # zero noise: zero corrections
        X = inputs[g.name][ri].cpu().numpy()
        Yg = outs[g.name][ri].cpu().numpy()
        cols = np.sort(rng.choice(g.N, size=min(512, g.N), replace=False))
        W = g.W[torch.as_tensor(cols, device="cuda")].cpu().numpy()
        check(Yg[:, cols], X, W, g.K, f"stacked {model_name} M={M} {g.name} ({layer.stacked[g.name]['path']})")
    assert spl.spl_get_device_status() == 0


def test_fp16x3_range_limit_is_caught_by_the_path_choice(spl):
    """The FP16X3 split scales each row by one power of two, so entries far below the row's largest
    fall under fp16's normal range and keep an absolute error of about 2^-39 max|a_row| |w| instead
    of 2^-21 |a w|.  Rows whose entries lie 2^-36 below their maximum, with the few large entries
    meeting tiny weights (so that the small ones carry S = sum |a||w|), make that floor exceed the
    Thm.-4 bound by about an order of magnitude.  Every path stays within its stated error model, and
    the bound-based path choice (a8, spl_choose_path) turns FP16X3 down for such data; the path it
    takes stays inside the hard bound."""
    M, K, N = 128, 3072, 256
    rng = np.random.default_rng(7)
    X = (rng.standard_normal((M, K)) * 2.0 ** -36).astype(np.float32)
    big = rng.choice(K, size=16, replace=False)
    X[:, big] = rng.standard_normal((M, 16)).astype(np.float32)  # a few entries 2^36 larger
    W = (rng.standard_normal((N, K)) * 0.02).astype(np.float32)
    W[:, big] *= 2.0 ** -40  # the large entries meet tiny weights
    Wt = spl.Weight.prepare(dev(W))
    Xd, zero = dev(X), torch.zeros((M, K), device="cuda")
    ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N))
    ref = linear.reference_output(X, W)
    S = linear.abs_products(X, X, np.zeros_like(X), W)
    hard = bounds.hard_bound(*S, K)
    from _util import product_tolerance
    over = {}
    for path in ("fp16x3", "tf32x3", "fp32"):
        Y = torch.empty((M, N), device="cuda")
        spl.spl_masked_linear(Y, Xd, Wt, path=path, workspace=ws)
        err = np.abs(f32(Y).astype(np.float64) - ref)
        tol = product_tolerance(S[0], K, path, X, W)
        assert np.all(err <= tol), (path, float(np.max(err / tol)))  # each path within its error model
        over[path] = float(np.max(err / hard))
    assert over["tf32x3"] <= 1.0 and over["fp32"] <= 1.0, over
    chosen, stats = spl.spl_choose_path(Xd, zero, Wt)
    assert chosen != "fp16x3" or over["fp16x3"] <= 1.0, (chosen, over)
    assert over[chosen] <= 1.0, (chosen, over)
