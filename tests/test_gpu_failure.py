"""Failure detection on the GPU without faulting it.

The tensor-core kernel bounds every mbarrier wait (about 1 s of globaltimer).  The test hook
launches it with the copy of its first K stage never issued, so the waits of the converter and
MMA warps run out; the kernel must set the device status word, drain the copies it did issue,
free its tensor memory and return.  The host then reads SPL_ETIMEOUT, the flag clears, and the
same context computes a correct product afterwards.
"""

import time

import numpy as np
import pytest
import torch

from paper_2609_15039_gb300 import workloads as wl
from _util import assert_product_close, f32

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def spl():
    from paper_2609_15039_gb300 import spl as binding
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    binding.lib()
    return binding


def test_bounded_wait_times_out_and_context_survives(spl):
    M, K, N = 256, 256, 512
    W = wl.weight(N, K, seed=1).numpy()
    A = wl.activations(M, K, seed=2).numpy()
    Wd, Ad = torch.as_tensor(W).cuda(), torch.as_tensor(A).cuda()
    Wt = spl.Weight.prepare(Wd)
    assert spl.spl_get_device_status() == spl.SPL_OK
    out = torch.empty((M, N), device="cuda")
    t0 = time.time()
    spl.spl_test_tc_wait_timeout(out, Ad, Wt)
    st = spl.spl_get_device_status()  # synchronises
    elapsed = time.time() - t0
    assert st == spl.SPL_ETIMEOUT, spl.status_string(st)
    assert elapsed < 30.0
    assert spl.spl_get_device_status() == spl.SPL_OK  # reading the status clears it
    # the context is still usable: a normal product is correct
    Y = torch.empty((M, N), device="cuda")
    spl.spl_masked_linear(Y, Ad, Wt, path="tf32x3",
                          workspace=spl.workspace(spl.spl_linear_workspace_bytes(M, K, N, "tf32x3")))
    torch.cuda.synchronize()
    assert_product_close(f32(Y), A, W, "tf32x3", what="after timeout")
    assert spl.spl_get_device_status() == spl.SPL_OK
