"""Host-side checks of the layer orchestration that run before any device work: the stacked step
graphs' input sets and the host-transfer helper refuse arguments they cannot serve.  No GPU."""

import types

import pytest
import torch

from paper_2609_15039_gb300.layer import MaskedStack, StackIO


def fake_stack(draws=8, layers=2, M=4, pooled=True):
    group = types.SimpleNamespace(name="qkv", K=8, N=12, W=torch.zeros(12, 8))
    layer = types.SimpleNamespace(draws=draws, M=M, groups=[group])
    stack = MaskedStack([layer] * layers, list(range(layers)))
    if pooled:
        stack.out_pool = {"qkv": torch.zeros(2, draws, layers, 2 * M, 12)}
    return stack


def test_capture_stacked_wants_a_divisor_of_draws_as_input_sets():
    stack = fake_stack(draws=8)
    sets = [[{"qkv": torch.zeros(4, 8)}] * 2 for _ in range(3)]
    with pytest.raises(ValueError, match="divide draws"):
        stack.capture_stacked(sets, 1.0, "laplace")


def test_stack_io_refuses_what_it_cannot_serve():
    host = {"qkv": torch.zeros(2, 4, 8)}  # not page-locked (there is no GPU here)
    with pytest.raises(ValueError, match="stacked=True"):
        StackIO(fake_stack(pooled=False), host)
    with pytest.raises(ValueError, match="divisor of draws"):
        StackIO(fake_stack(draws=8), host, sets=3)
    with pytest.raises(ValueError, match="divisor of draws"):
        StackIO(fake_stack(draws=1), host)  # no two sets divide one draw
    with pytest.raises(ValueError, match="one per direction"):
        StackIO(fake_stack(), host, streams=3)
    with pytest.raises(ValueError, match="page-locked"):
        StackIO(fake_stack(), host)


def test_stack_io_default_sets_are_the_largest_divisor_up_to_eight():
    """The set count is chosen before the host buffers are checked, so an instance whose check
    refuses them (not page-locked here) still shows the choice."""
    for draws, sets in ((8, 8), (12, 6), (3, 3), (2, 2), (16, 8)):
        io = StackIO.__new__(StackIO)
        with pytest.raises(ValueError, match="page-locked"):
            io.__init__(fake_stack(draws=draws), {"qkv": torch.zeros(2, 4, 8)})
        assert io.sets == sets, (draws, io.sets)
