"""Full-size parity: the five workloads at their own sizes, in the configuration the bench runs
(fused group weights, banks of corrections, AUTO path), checked on sampled outputs that the
oracle computes one by one against the hard bound (Thm. 4 + mask rounding).

Inputs are drawn on the device by the seeded generators; the oracle reads the sampled rows of
X and W and regenerates the sampled rows of eta from the Philox definition.  The noise scales
come from the oracle (||W||_2 from LAPACK singular values), so both sides get the same input.
"""

import numpy as np
import pytest
import torch

from oracle import bounds, linear, philox, sensitivity as osens
from paper_2609_15039_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def spl():
    from paper_2609_15039_gb300 import spl as binding
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    binding.lib()
    return binding


def make_layer(model, layer_idx, base_seed, draws, M):
    from paper_2609_15039_gb300.layer import MaskedLayer
    weights = {name: wl.weight(N, K, seed=wl.layer_seed(base_seed, layer_idx, pi), device="cuda")
               for pi, (name, K, N, g) in enumerate(model.projections())}
    layer = MaskedLayer.from_weights(model, weights)
    ones = np.ones(model.d_model)
    norms = {n: float(np.linalg.svd(weights[n].double().cpu().numpy(), compute_uv=False)[0])
             for n in ("v", "up", "gate")}
    layer.deltas = {
        "qkv": osens.delta_layernorm(ones),
        "gateup": osens.delta_layernorm(ones),
        "o": osens.delta_attention(ones, norms["v"]),
        "down": osens.delta_activation(ones, None, model.d_ff, norms["up"], norms["gate"]),
    }
    layer.allocate(M, draws)
    inputs = {g: wl.activations(M, K, seed=wl.layer_seed(base_seed, layer_idx, 50 + gi), device="cuda")
              for gi, (g, K, _n) in enumerate(model.input_groups())}
    return layer, inputs


def check_sampled(layer, inputs, outs, eps, mech, seed, cycle, d, n_rows=12, n_cols=48, rng_seed=0):
    """Oracle on sampled (row, column) outputs of every projection; returns worst err / hard bound."""
    rng = np.random.default_rng(rng_seed)
    M = layer.M
    rows = np.sort(rng.choice(M, size=min(n_rows, M), replace=False))
    worst = 0.0
    for gi, g in enumerate(layer.groups):
        X = inputs[g.name][torch.as_tensor(rows, device="cuda")].cpu().numpy()
        base = layer.block_offset(g, cycle, d)
        eta = np.stack([philox.noise((1, g.K), layer.deltas[g.name], eps, mech, seed, stream_id=gi,
                                     offset=base + int(m) * g.K // 4)[0] for m in rows])
        Xt = linear.mask(X, eta)
        Yg = outs[g.name][torch.as_tensor(rows, device="cuda")].double().cpu().numpy()
        for name in g.names:
            a, b = g.columns(name)
            cols = np.sort(rng.choice(b - a, size=min(n_cols, b - a), replace=False))
            W = layer.weight(name)[torch.as_tensor(cols, device="cuda")].cpu().numpy()
            S = linear.abs_products(X, Xt, eta, W)
            err = np.abs(Yg[:, a + cols] - linear.reference_output(X, W))
            hb = bounds.hard_bound(*S, g.K)
            assert np.all(err <= hb * (1 + 1e-5)), (name, float(np.max(err / hb)))
            worst = max(worst, float(np.max(err / hb)))
    return worst


@pytest.mark.parametrize("layer_idx", [0, 27])
def test_llama_stack_prefill_512(spl, layer_idx):
    cfg = wl.CONFIGS["llama_stack"]
    model, M, mech, eps = cfg["model"], cfg["M"], cfg["mech"], cfg["eps"][0]
    layer, inputs = make_layer(model, layer_idx, 7, cfg["draws"], M)
    seed = 1000 + layer_idx  # seeded per layer
    layer.refill(eps, mech, seed, cycle=0)
    for d in (0, cfg["draws"] - 1):
        outs = layer.online(inputs, eps, mech, seed, cycle=0, d=d)
        torch.cuda.synchronize()
        check_sampled(layer, inputs, outs, eps, mech, seed, 0, d, rng_seed=d)
    assert spl.spl_get_device_status() == 0


def test_llama_stack_decode_m1(spl):
    cfg = wl.CONFIGS["llama_stack"]
    model, mech, eps = cfg["model"], cfg["mech"], cfg["eps"][0]
    layer, inputs = make_layer(model, 3, 7, cfg["draws"], 1)
    seed = 77
    for step in range(10):  # crosses a bank refill
        cycle, d = divmod(step, cfg["draws"])
        if d == 0:
            layer.refill(eps, mech, seed, cycle=cycle)  # 8 draws at M = 1: the decode kernel at M = 8
        outs = layer.online(inputs, eps, mech, seed, cycle=cycle, d=d)
        torch.cuda.synchronize()
        check_sampled(layer, inputs, outs, eps, mech, seed, cycle, d, n_cols=256, rng_seed=step)


@pytest.mark.parametrize("eps", [0.1, 1.0, 10.0])
def test_qwen_stack_prefill_2048(spl, eps):
    cfg = wl.CONFIGS["qwen_stack"]
    model, M, mech = cfg["model"], cfg["M"], cfg["mech"]
    layer, inputs = make_layer(model, 0, 11, 2, M)
    seed = 4040
    layer.refill(eps, mech, seed, cycle=0)
    outs = layer.online(inputs, eps, mech, seed, cycle=0, d=1)
    torch.cuda.synchronize()
    worst = check_sampled(layer, inputs, outs, eps, mech, seed, 0, 1, n_rows=16)
    assert worst <= 1.0


@pytest.mark.parametrize("M", [1, 4, 16, 64, 256, 1024])
def test_qwen_sweep(spl, M):
    cfg = wl.CONFIGS["qwen_sweep"]
    model, mech, eps = cfg["model"], cfg["mech"], cfg["eps"][0]
    layer, inputs = make_layer(model, 1, 13, 2, M)
    seed = 5050 + M
    layer.refill(eps, mech, seed, cycle=0)
    for d in range(2):
        outs = layer.online(inputs, eps, mech, seed, cycle=0, d=d)
        torch.cuda.synchronize()
        check_sampled(layer, inputs, outs, eps, mech, seed, 0, d, rng_seed=M + d)


@pytest.mark.parametrize("mech", ["laplace", "gaussian"])
def test_mask_alone_1e9_sampled(spl, mech):
    n = 10 ** 9
    X = torch.empty(n, device="cuda")
    X.normal_(generator=torch.Generator(device="cuda").manual_seed(3))
    Xt = torch.empty_like(X)
    sens, eps, seed, sid, off = 719.8, 1.0, 99, 5, 12345
    spl.spl_noise_mask(Xt, None, X, sens, eps, mech, seed, stream_id=sid, offset=off)
    torch.cuda.synchronize()
    idx = np.sort(np.random.default_rng(1).choice(n, 100_000, replace=False))
    ti = torch.as_tensor(idx, device="cuda")
    x, xt = X[ti].cpu().numpy(), Xt[ti].double().cpu().numpy()
    b = np.float64(philox.scale_fp32(sens, eps))
    j = idx // 4 + off
    blocks = np.stack(philox.philox4x32_10(j & 0xFFFFFFFF, j >> 32, sid, 0, seed, 0), axis=1)
    lane = idx % 4
    if mech == "laplace":
        eta = philox.laplace_from_words(blocks[np.arange(idx.size), lane], b)
        tol = 4 * np.spacing(np.abs(eta.astype(np.float32))).astype(np.float64)
    else:
        g = philox.gaussian_from_blocks(blocks, b)
        eta = g[np.arange(idx.size), lane]
        u1 = ((blocks[np.arange(idx.size), 2 * (lane // 2)] >> np.uint32(8)).astype(np.float64) + 1) * 2.0 ** -24
        tol = 8 * 2.0 ** -24 * b * np.sqrt(-2 * np.log(u1)) + 2 * np.spacing(np.abs(eta.astype(np.float32)))
    exp = linear.mask(x, eta.astype(np.float32)).astype(np.float64)
    assert np.all(np.abs(xt - exp) <= tol + np.spacing(np.abs(exp.astype(np.float32))).astype(np.float64))


@pytest.mark.parametrize("M", [512, 1])
def test_llama_lm_head(spl, M):
    """The LM head (3072 -> 128256, Sec. 5.1, after the final RMSNorm: Delta from Thm. 1) at
    prefill and decode sizes, with a bank of 8 corrections summed in the online order."""
    model = wl.LLAMA_3_2_3B
    K, N, draws, eps, mech, seed = model.d_model, model.vocab, 8, 1.0, "gaussian", 606
    W = wl.weight(N, K, seed=9001, device="cuda")
    Wt = spl.Weight.prepare(W)
    X = wl.activations(M, K, seed=9002, device="cuda")
    delta = osens.delta_layernorm(np.ones(K))
    eta = torch.empty((draws * M, K), device="cuda")
    spl.spl_noise(eta, delta, eps, mech, seed)
    C = torch.empty((draws * M, N), device="cuda")
    ws = spl.workspace(max(spl.spl_precompute_matched_workspace_bytes(draws * M, K, N, M),
                           spl.spl_linear_workspace_bytes(M, K, N)))
    spl.spl_precompute_noise_product_matched(C, eta, Wt, M, workspace=ws)
    d = 3
    Xt = torch.empty_like(X)
    spl.spl_noise_mask(Xt, None, X, delta, eps, mech, seed, offset=d * M * K // 4)
    Y = torch.empty((M, N), device="cuda")
    spl.spl_masked_linear_unmask(Y, Xt, Wt, C[d * M:(d + 1) * M], workspace=ws)
    torch.cuda.synchronize()
    rng = np.random.default_rng(M)
    rows = np.sort(rng.choice(M, size=min(8, M), replace=False))
    cols = np.sort(rng.choice(N, size=256, replace=False))
    Xs = X[torch.as_tensor(rows, device="cuda")].cpu().numpy()
    eta_s = np.stack([philox.noise((1, K), delta, eps, mech, seed, offset=(d * M + int(m)) * K // 4)[0] for m in rows])
    Ws = W[torch.as_tensor(cols, device="cuda")].cpu().numpy()
    S = linear.abs_products(Xs, linear.mask(Xs, eta_s), eta_s, Ws)
    got = Y[torch.as_tensor(rows, device="cuda")][:, torch.as_tensor(cols, device="cuda")].double().cpu().numpy()
    err = np.abs(got - linear.reference_output(Xs, Ws))
    assert np.all(err <= bounds.hard_bound(*S, K) * (1 + 1e-5))


def test_llama_stacked_prefill_512(spl):
    """The bench's schedule at its own size: a Llama-3.2-3B-shaped layer at 512 tokens, each product of
    1024 rows carrying the next cycle's correction of its draw; the recovered outputs of the second
    cycle checked on sampled outputs against the hard bound (Laplace, eps = 1)."""
    from paper_2609_15039_gb300.layer import MaskedLayer
    model, M, draws, eps, mech = wl.LLAMA_3_2_3B, 512, 2, 1.0, "laplace"
    layer, inputs = make_layer(model, 3, 7, draws, M)
    stacked = MaskedLayer(model, layer.groups, deltas=layer.deltas)
    stacked.allocate_stacked(M, draws)
    seed = 1003
    for cycle in range(2):
        for d in range(draws):
            outs = stacked.stacked_step(inputs, eps, mech, seed, d, cycle % 2, cycle=cycle)
    torch.cuda.synchronize()
    worst = check_sampled(stacked, inputs, outs, eps, mech, seed, 1, draws - 1)
    assert worst < 0.05
    assert spl.spl_get_device_status() == 0
