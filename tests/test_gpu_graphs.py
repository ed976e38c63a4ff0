"""CUDA graphs of a bank cycle: replayed graphs compute, bit for bit, what the eager library
calls compute for the same steps, across bank refills (the Philox offsets then come from the
device and the last graph of a cycle moves them on)."""

import numpy as np
import pytest
import torch

from paper_2609_15039_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def spl():
    from paper_2609_15039_gb300 import spl as binding
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    binding.lib()
    return binding


def make_layer(model, M, draws):
    from paper_2609_15039_gb300.layer import MaskedLayer
    weights = {name: wl.weight(N, K, seed=300 + pi, device="cuda")
               for pi, (name, K, N, g) in enumerate(model.projections())}
    layer = MaskedLayer.from_weights(model, weights)
    layer.deltas = {"qkv": 90.0, "gateup": 90.0, "o": 45.0, "down": 700.0}
    layer.allocate(M, draws)
    inputs = {g: wl.activations(M, K, seed=400 + gi, device="cuda")
              for gi, (g, K, _n) in enumerate(model.input_groups())}
    return layer, inputs


@pytest.mark.parametrize("M", [128, 4])
def test_graph_replay_equals_eager_steps(spl, M):
    model = wl.ModelShape("small", 1, 512, 1024, 512, 256, 1000)
    draws, eps, mech, seed = 3, 1.0, "laplace", 77
    layer, inputs = make_layer(model, M, draws)

    def eager(s):
        cycle, d = divmod(s, draws)
        if d == 0:
            layer.refill(eps, mech, seed, cycle)
        return {g: y.clone() for g, y in layer.online(inputs, eps, mech, seed, cycle, d).items()}

    first, steps = 2 * draws, 2 * draws + 2  # from cycle 2 into cycle 4
    expected = [eager(s) for s in range(first, first + steps)]
    torch.cuda.synchronize()
    graphs, launches = layer.capture(inputs, eps, mech, seed)
    assert len(graphs) == draws and all(n > 0 for n in launches)
    layer.set_cycle(first // draws)
    for i, s in enumerate(range(first, first + steps)):
        graphs[s % draws].replay()
        torch.cuda.synchronize()
        for g in expected[i]:
            assert torch.equal(layer.bank[g]["Y"], expected[i][g]), (s, g)
    # the device bases moved on by one cycle per completed cycle
    exp_base = [layer.block_offset(g, (first + steps) // draws, 0) for g in layer.groups]
    assert layer.rng_base.cpu().tolist() == exp_base
    assert spl.spl_get_device_status() == 0


def test_device_offset_equals_host_offset(spl):
    n, seed, sid = 4096 + 3, 5, 2
    base = torch.tensor([12345], dtype=torch.int64, device="cuda")
    a = torch.empty(n, dtype=torch.int32, device="cuda")
    b = torch.empty_like(a)
    spl.spl_random_bits(a, seed, sid, offset=12345 + 7)
    spl.spl_random_bits(b, seed, sid, offset=7, offset_dev=base)
    assert torch.equal(a, b)
    X = torch.randn(33, 64, device="cuda")
    x1, x2 = torch.empty_like(X), torch.empty_like(X)
    spl.spl_noise_mask(x1, None, X, 3.0, 1.0, "gaussian", seed, sid, offset=12345 + 9)
    spl.spl_noise_mask(x2, None, X, 3.0, 1.0, "gaussian", seed, sid, offset=9, offset_dev=base)
    assert torch.equal(x1, x2)
    spl.spl_rng_advance(base, 2 ** 40)
    assert base.item() == 12345 + 2 ** 40
    # an offset word must be 8-byte aligned: refused before anything is launched
    assert spl.lib().spl_rng_advance(base.data_ptr() + 4, 1, None) == spl.SPL_EALIGN


@pytest.mark.parametrize("stored", [False, True])
def test_overlapped_cycle_graphs_equal_eager_steps(spl, stored):
    """Whole-cycle graphs that compute the next cycle's corrections during this cycle's steps (on
    streams of their own) give, step by step, the eager results -- across three cycles, so both
    correction buffers (and, with stored noise, both noise buffers) are filled by a graph and read
    by the other."""
    model = wl.ModelShape("small", 1, 512, 1024, 512, 256, 1000)
    draws, eps, mech, seed, M = 3, 1.0, "gaussian", 78, 128
    layer, inputs = make_layer(model, M, draws)
    layer.allocate(M, draws, stored_noise=stored)
    assert all(layer._fused_split(g, "auto", M) for g in layer.groups)

    def eager(s):
        cycle, d = divmod(s, draws)
        if d == 0:
            layer.refill(eps, mech, seed, cycle)
        return {g: y.clone() for g, y in layer.online(inputs, eps, mech, seed, cycle, d).items()}

    first, cycles = 2, 3
    expected = [eager(s) for s in range(first * draws, (first + cycles) * draws)]
    torch.cuda.synchronize()
    outs = []

    def after(d):  # each step's results, kept inside the graph
        outs.append({g.name: layer.bank[g.name]["Y"].clone() for g in layer.groups})

    graphs, launches = layer.capture_overlapped(inputs, eps, mech, seed, after=after)
    assert len(graphs) == 2 and all(n > 0 for n in launches)
    captured = list(outs)  # the tensors each graph writes its step results into
    layer.set_cycle(first)
    layer.refill(eps, mech, seed, 0, device_base=True, parallel=True, parity=first % 2)
    for i in range(cycles):
        c = first + i
        graphs[c % 2].replay()
        torch.cuda.synchronize()
        for d in range(draws):
            got = captured[(c % 2) * draws + d]
            for g in got:
                assert torch.equal(got[g], expected[i * draws + d][g]), (c, d, g)
    exp_base = [layer.block_offset(g, first + cycles, 0) for g in layer.groups]
    assert layer.rng_base.cpu().tolist() == exp_base
    assert spl.spl_get_device_status() == 0


def test_stack_overlapped_decode_graphs_equal_eager_steps(spl):
    """The stack's whole-cycle graphs -- every layer's next-cycle corrections on a stream of lower
    priority with a workspace of their own -- give the eager steps' results bit for bit on the FP32
    decode path (one row), where both the products and the corrections use a workspace: across
    three cycles, so each correction buffer is filled by one graph and read by the other."""
    from paper_2609_15039_gb300.layer import MaskedStack
    model = wl.ModelShape("small", 2, 512, 1024, 512, 256, 1000)
    draws, eps, mech, M = 3, 1.0, "laplace", 1
    stack = MaskedStack.build(model, 2, M, draws, base_seed=5, power_iters=50)
    inputs = stack.inputs(6)

    def eager(s):
        cycle, d = divmod(s, draws)
        res = []
        for layer, x, seed in zip(stack.layers, inputs, stack.seeds):
            if d == 0:
                layer.refill(eps, mech, seed, cycle)
            res.append({g: y.clone() for g, y in layer.online(x, eps, mech, seed, cycle, d).items()})
        return res

    first, cycles = 2, 3
    expected = [eager(s) for s in range(first * draws, (first + cycles) * draws)]
    torch.cuda.synchronize()
    outs = []

    def after(d):
        outs.append([{g.name: l.bank[g.name]["Y"].clone() for g in l.groups} for l in stack.layers])

    bank_ws = spl.workspace(max(l.workspace_bytes(M, draws) for l in stack.layers))
    graphs, launches = stack.capture_overlapped(inputs, eps, mech, bank_ws, after=after)
    assert len(graphs) == 2 and all(n > 0 for n in launches)
    captured = list(outs)
    stack.start_overlapped(first, eps, mech)
    for i in range(cycles):
        c = first + i
        graphs[c % 2].replay()
        torch.cuda.synchronize()
        for d in range(draws):
            got = captured[(c % 2) * draws + d]
            for li in range(len(stack.layers)):
                for g in got[li]:
                    assert torch.equal(got[li][g], expected[i * draws + d][li][g]), (c, d, li, g)
    for layer in stack.layers:
        assert layer.rng_base.cpu().tolist() == [layer.block_offset(g, first + cycles, 0) for g in layer.groups]
    assert spl.spl_get_device_status() == 0


@pytest.mark.parametrize("mech", ["laplace", "gaussian"])
def test_stored_noise_steps_equal_drawn_noise_steps(spl, mech):
    """Online steps that mask with the noise the refill kept give the results of steps that draw the
    noise again, bit for bit, across two bank cycles."""
    model = wl.ModelShape("small", 1, 512, 1024, 512, 256, 1000)
    draws, eps, seed, M = 3, 1.0, 81, 128
    res = []
    for stored in (True, False):
        layer, inputs = make_layer(model, M, draws)
        layer.allocate(M, draws, stored_noise=stored)
        outs = []
        for s in range(2 * draws):
            cycle, d = divmod(s, draws)
            if d == 0:
                layer.refill(eps, mech, seed, cycle)
            outs.append({g: y.clone() for g, y in layer.online(inputs, eps, mech, seed, cycle, d).items()})
        res.append(outs)
    for a, b in zip(*res):
        for g in a:
            assert torch.equal(a[g], b[g]), g
    assert spl.spl_get_device_status() == 0


# ------------------------------------------------ the stacked schedule (online rows beside a bank draw)
def make_stacked(model, M, draws, layers=1, zero_inputs=False):
    from paper_2609_15039_gb300.layer import MaskedLayer, MaskedStack
    stack_layers = []
    for li in range(layers):
        weights = {name: wl.weight(N, K, seed=500 + 10 * li + pi, device="cuda")
                   for pi, (name, K, N, g) in enumerate(model.projections())}
        layer = MaskedLayer.from_weights(model, weights)
        layer.deltas = {"qkv": 90.0, "gateup": 90.0, "o": 45.0, "down": 700.0}
        layer.allocate_stacked(M, draws)
        stack_layers.append(layer)
    stack = MaskedStack(stack_layers, [91 + li for li in range(layers)])
    inputs = [{g: (torch.zeros((M, K), device="cuda") if zero_inputs else
                   wl.activations(M, K, seed=600 + 10 * li + gi, device="cuda"))
               for gi, (g, K, _n) in enumerate(model.input_groups())} for li in range(layers)]
    return stack, inputs


@pytest.mark.parametrize("M,model", [(128, wl.ModelShape("small", 1, 512, 1024, 512, 256, 1000)),
                                     (512, wl.LLAMA_3_2_3B), (1, wl.LLAMA_3_2_3B),
                                     (2, wl.ModelShape("small", 1, 512, 1024, 512, 256, 1000)),
                                     (4, wl.ModelShape("small", 1, 512, 1024, 512, 256, 1000))])
def test_stacked_correction_cancels_exactly(spl, M, model):
    """With x = 0 the mask is the noise itself, so the recovered output is fl(eta W^T) - fl(eta W^T):
    exactly zero when the correction (computed in the previous cycle in the bank half of a product of
    2M rows) is summed in exactly the order of the online row that meets it (the masked half of a later
    product of the same shape) -- every element, at the bench's own sizes too.  Decode sizes (2M <= 4)
    take the one-launch form (noise, mask and product together); 2M = 8 the decode kernel after a
    separate mask."""
    draws, eps, mech = 2, 1.0, "laplace"
    stack, inputs = make_stacked(model, M, draws, zero_inputs=True)
    layer, seed = stack.layers[0], stack.seeds[0]
    for cycle in range(3):
        for d in range(draws):
            outs = layer.stacked_step(inputs[0], eps, mech, seed, d, cycle % 2, cycle=cycle)
            if cycle >= 1:  # cycle 0's corrections were never computed
                for g, y in outs.items():
                    assert not torch.any(y).item(), (cycle, d, g, float(y.abs().max()))
    assert spl.spl_get_device_status() == 0


@pytest.mark.parametrize("M", [128, 1])
def test_stacked_graphs_equal_eager_steps(spl, M):
    """Replayed stacked graphs (two layers, device-side Philox bases, the last graph of a cycle moving
    them on) give, bit for bit, the eager stacked steps of the same cycles; any number of steps.  One
    row: the decode form, one launch per group and step."""
    model = wl.ModelShape("small", 1, 512, 1024, 512, 256, 1000)
    draws, eps, mech = 3, 1.0, "gaussian"
    stack, inputs = make_stacked(model, M, draws, layers=2)
    expected = {}
    for cycle in range(4):
        for d in range(draws):
            for li, layer in enumerate(stack.layers):
                outs = layer.stacked_step(inputs[li], eps, mech, stack.seeds[li], d, cycle % 2, cycle=cycle)
                expected[(cycle * draws + d, li)] = {g: y.clone() for g, y in outs.items()}
    torch.cuda.synchronize()
    graphs, launches = stack.capture_stacked(inputs, eps, mech)
    assert all(n > 0 for p in launches for n in p)
    stack.start_stacked(2, graphs)  # runs cycle 1's graphs: cycle 2's corrections, bases at cycle 2
    for s in range(2 * draws, 4 * draws - 1):  # stop one short of a whole cycle: any step count works
        graphs[(s // draws) % 2][s % draws].replay()
        torch.cuda.synchronize()
        cycle, d = divmod(s, draws)
        for li, layer in enumerate(stack.layers):
            for g in layer.groups:
                y = layer.stacked[g.name]["out"][1 - cycle % 2][d][:M]
                assert torch.equal(y, expected[(s, li)][g.name]), (s, li, g.name)
    assert spl.spl_get_device_status() == 0


@pytest.mark.parametrize("M,draws,streams", [(128, 2, 2), (1, 2, 2), (128, 4, 2), (128, 4, 1)])
def test_stack_io_moves_every_step_exactly(spl, M, draws, streams):
    """StackIO: every layer's inputs copied in from page-locked host memory one step ahead and every
    layer's outputs copied back with one strided copy per group, on their own streams, with no host
    synchronisation between steps and the device output buffers rewritten while earlier copies may
    still be in flight: each step's host outputs equal, bit for bit, the device outputs of the same
    steps replayed one at a time with the inputs already in place."""
    from paper_2609_15039_gb300.layer import MaskedStack, StackIO
    model = wl.ModelShape("small", 1, 512, 1024, 512, 256, 1000)
    eps, mech = 1.0, "laplace"
    stack = MaskedStack.build(model, 3, M, draws, base_seed=5, power_iters=50, stacked=True)
    inputs = stack.inputs(17)
    host_in = {g: torch.stack([inp[g] for inp in inputs]).cpu().pin_memory() for g in inputs[0]}
    steps = list(range(2 * draws, 2 * draws + 4 * draws + 1))
    io = StackIO(stack, host_in, ring=len(steps), streams=streams)  # a host slot per step
    assert io.sets == draws  # inputs go in up to draws - 1 steps ahead
    assert io.bytes_per_step() == (sum(x.numel() * 4 for x in host_in.values()),
                                   sum(3 * M * g.N * 4 for g in stack.layers[0].groups))
    graphs, _ = stack.capture_stacked(io.layer_inputs(), eps, mech)
    stack.start_stacked(2, graphs)
    for s in steps:
        io.step(graphs, s, stop=steps[-1] + 1)
    assert not io._in  # nothing copied in for a step past the last
    io.finish()
    torch.cuda.synchronize()
    got = {s: {g: y.clone() for g, y in io.outputs(s)[0].items()} for s in steps}
    for dset in io.dev_in:  # the reference: both input sets in place beforehand, one step at a time
        for g, x in host_in.items():
            dset[g].copy_(x)
    stack.start_stacked(2, graphs)
    for s in steps:
        stack.replay_stacked(graphs, s)
        torch.cuda.synchronize()
        p, d = (s // draws) % 2, s % draws
        for g, pool in stack.out_pool.items():
            assert torch.equal(got[s][g], pool[1 - p, d, :, :M].cpu()), (s, g)
            for li, layer in enumerate(stack.layers):  # the pool is the layers' own output buffers
                assert layer.stacked[g]["out"][1 - p][d].data_ptr() == pool[1 - p, d, li].data_ptr()
    assert spl.spl_get_device_status() == 0
