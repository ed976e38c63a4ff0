"""The decode product without allocation (spl_masked_linear_unmask_noalloc).

This entry point is for callers that cannot allocate device memory when the
product runs (a decode loop that must not stall on a synchronising
cudaMalloc, a process whose device memory another allocator already holds,
a worker with a fixed memory budget).  It takes its scratch from a fixed
array inside the library instead of a caller-provided workspace.  Here it is
called through the C ABI and checked against the existing entry point,
spl_masked_linear_unmask with its own zero-filled workspace, on two calls in
a row (the shared array must come back clean after each call), within the
product tolerance the other tests use.  The file name makes pytest collect
it last.
"""

import numpy as np
import pytest
import torch

from paper_2609_15039_gb300 import workloads as wl
from _util import assert_product_close, f32, product_tolerance

pytestmark = pytest.mark.gpu

# decode shapes: Llama O / Down and Qwen Gate at 1, 4 and 16 tokens (all use split-K partials)
CASES = [(1, 3072, 3072), (4, 8192, 3072), (16, 2560, 9728), (3, 1028, 600)]


@pytest.fixture(scope="module")
def spl():
    from paper_2609_15039_gb300 import spl as binding
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    binding.lib()
    return binding


@pytest.mark.parametrize("M,K,N", CASES)
def test_noalloc_matches_workspace_entry_point(spl, M, K, N):
    W = wl.weight(N, K, seed=M + K).numpy()
    Wd = torch.as_tensor(W).cuda()
    ws = spl.workspace(spl.spl_linear_workspace_bytes(M, K, N, "fp32"))
    S = None
    for call in range(2):
        A = (wl.activations(M, K, seed=10 * call + M).numpy() * 300).astype(np.float32)
        C = wl.activations(M, N, seed=20 * call + M).numpy()
        Ad, Cd = torch.as_tensor(A).cuda(), torch.as_tensor(C).cuda()
        ref = torch.empty((M, N), device="cuda")
        spl.spl_masked_linear_unmask(ref, Ad, Wd, Cd, path="fp32", workspace=ws)
        got = torch.full((M, N), float("nan"), device="cuda")
        spl.spl_masked_linear_unmask_noalloc(got, Ad, Wd, Cd)
        torch.cuda.synchronize()
        S = np.abs(A.astype(np.float64)) @ np.abs(W.astype(np.float64)).T
        tol = 2 * product_tolerance(S, K, "fp32") + 4 * 2.0 ** -24 * np.abs(f32(ref).astype(np.float64))
        diff = np.abs(f32(got).astype(np.float64) - f32(ref).astype(np.float64))
        assert np.all(diff <= tol), f"call {call}: max diff/tol {float(np.max(diff / tol)):.3g}"
        assert_product_close(f32(got), A, W, "fp32", C=C, what=f"noalloc call {call}")


def test_noalloc_rejects_what_it_cannot_hold(spl):
    W = torch.zeros((8, 64), device="cuda")
    X = torch.zeros((17, 64), device="cuda")
    with pytest.raises(spl.SplError) as e:
        spl.spl_masked_linear_unmask_noalloc(torch.empty((17, 8), device="cuda"), X, W, torch.zeros((17, 8),
                                                                                                  device="cuda"))
    assert e.value.status == spl.SPL_ESHAPE  # only the decode kernel (M <= 16) has this variant
    # K = 65536 takes at least 43 K-slices (a slice holds at most 1536 columns), so 16 tokens x 4096
    # outputs of partials per slice (11.3 MB and more) is more than the 4 MiB array holds
    N, K = 4096, 65536
    W = torch.zeros((N, K), device="cuda")
    X = torch.zeros((16, K), device="cuda")
    with pytest.raises(spl.SplError) as e:
        spl.spl_masked_linear_unmask_noalloc(torch.empty((16, N), device="cuda"), X, W,
                                             torch.zeros((16, N), device="cuda"))
    assert e.value.status == spl.SPL_EWORKSPACE
