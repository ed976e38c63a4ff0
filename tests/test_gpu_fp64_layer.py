"""A layer with its Down projection in binary64 (Sec. 5.5): the online step, replayed graphs and
the bank agree with the eager binary64 calls, and Down's recovered output is accurate."""

import numpy as np
import pytest
import torch

from oracle import linear, philox
from paper_2609_15039_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def spl():
    from paper_2609_15039_gb300 import spl as binding
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    binding.lib()
    return binding


def test_down_in_binary64_is_accurate_and_graph_safe(spl):
    from paper_2609_15039_gb300.layer import MaskedLayer
    model = wl.ModelShape("small", 1, 512, 2048, 512, 256, 1000)
    weights = {name: wl.weight(N, K, seed=500 + pi, device="cuda")
               for pi, (name, K, N, g) in enumerate(model.projections())}
    layer = MaskedLayer.from_weights(model, weights)
    layer.fp64 = {"down"}
    layer.deltas = {"qkv": 90.0, "gateup": 90.0, "o": 45.0, "down": 2.6e8}
    M, draws, eps, mech, seed = 16, 2, 1.0, "laplace", 9
    layer.allocate(M, draws)
    inputs = {g: wl.activations(M, K, seed=600 + gi, device="cuda")
              for gi, (g, K, _n) in enumerate(model.input_groups())}
    layer.refill(eps, mech, seed, 0)
    outs = {g: y.clone() for g, y in layer.online(inputs, eps, mech, seed, 0, 1).items()}
    torch.cuda.synchronize()
    assert layer.bank["down"]["C"].dtype == torch.float64
    X = inputs["down"].cpu().numpy()
    Wd = weights["down"].cpu().numpy()
    ref = linear.reference_output(X, Wd)
    err = np.abs(outs["down"].double().cpu().numpy() - ref)
    assert np.max(err) <= 4 * 2.0 ** -24 * np.max(np.abs(ref))
    # the same step replayed from captured graphs
    graphs, _ = layer.capture(inputs, eps, mech, seed)
    layer.set_cycle(0)
    graphs[0].replay()
    graphs[1].replay()
    torch.cuda.synchronize()
    for g in outs:
        assert torch.equal(layer.bank[g]["Y"], outs[g]), g
    # the binary64 mask regenerated for draw 1 is the oracle's mask
    eta = philox.noise((M, model.d_ff), 2.6e8, eps, mech, seed, stream_id=3, offset=layer.block_offset(layer.group("down"), 0, 1))
    xt = layer.bank["down"]["xt"].cpu().numpy()
    assert np.all(np.abs(xt - linear.mask_f64(X, eta)) <= 4 * 2.0 ** -24 * np.abs(eta) + 1e-300)
