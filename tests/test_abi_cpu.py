"""The C-ABI library on the CPU: it loads without a GPU, exports every entry
point include/spl.h declares, and its host-only logic agrees with the oracle.
No kernel is launched here."""

import ctypes
import math
import os
import re

import numpy as np
import pytest

from oracle import sensitivity as osens

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def spl():
    from paper_2609_15039_gb300 import build, spl as binding
    if not os.path.exists(binding.LIB_PATH):
        build.build()
    binding.lib()
    return binding


def declared_functions():
    names = []
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            text = open(os.path.join(ROOT, "include", fn)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names += re.findall(r"^\s*(?:const\s+)?\w+\*?\s+\*?(spl_\w+)\s*\(", text, flags=re.M)
    return sorted(set(names))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("spl_noise", "spl_mask", "spl_masked_linear", "spl_precompute_noise_product", "spl_unmask",
                     "spl_noise_mask", "spl_masked_linear_unmask", "spl_random_bits"):
        assert required in names


def test_library_exports_every_declared_symbol(spl):
    handle = ctypes.CDLL(spl.LIB_PATH)
    missing = [n for n in declared_functions() if not hasattr(handle, n)]
    assert not missing, missing
    # the binding declares a signature for every exported entry point
    assert set(declared_functions()) <= set(spl._SIGS)


def test_status_strings(spl):
    assert spl.status_string(0) == "SPL_OK"
    assert spl.status_string(7) == "SPL_EWORKSPACE"
    assert spl.status_string(99) == "SPL_UNKNOWN"


def test_argument_validation_without_launch(spl):
    L = spl.lib()
    rng = spl.spl_rng(0, 0, 0)
    # eps <= 0, NaN; negative sensitivity; bad mechanism -> EINVAL before any CUDA call
    for eps in (0.0, -1.0, float("nan")):
        assert L.spl_noise(None, 4, 4, 1.0, eps, 0, rng, None) == spl.SPL_EINVAL
    assert L.spl_noise(None, 4, 4, -1.0, 1.0, 0, rng, None) == spl.SPL_EINVAL
    assert L.spl_noise(None, 4, 4, float("inf"), 1.0, 0, rng, None) == spl.SPL_EINVAL
    assert L.spl_noise(None, 4, 4, 1.0, 1.0, 7, rng, None) == spl.SPL_EINVAL
    assert L.spl_noise(None, 4, 4, 1.0, 1.0, 0, rng, None) == spl.SPL_EINVAL  # NULL output
    # zero-sized problems are no-ops
    assert L.spl_noise(None, 0, 5, 1.0, 1.0, 0, rng, None) == spl.SPL_OK
    assert L.spl_mask(None, None, None, 3, 0, None) == spl.SPL_OK
    assert L.spl_unmask(None, None, None, 0, 0, None) == spl.SPL_OK
    assert L.spl_masked_linear(None, None, None, 0, 8, 8, 0, None, 0, None) == spl.SPL_OK
    # negative sizes, bad path, NULL operands, K % 4
    assert L.spl_masked_linear(None, None, None, -1, 8, 8, 0, None, 0, None) == spl.SPL_EINVAL
    assert L.spl_masked_linear(None, None, None, 4, 8, 8, 9, None, 0, None) == spl.SPL_EINVAL
    assert L.spl_masked_linear(None, None, None, 4, 8, 8, 0, None, 0, None) == spl.SPL_EINVAL
    buf = (ctypes.c_float * 64)()
    p = ctypes.cast(buf, ctypes.c_void_p).value
    base = p + (16 - p % 16) % 16
    w = spl.spl_weight(base, None, None, None, None, None)
    assert L.spl_masked_linear(base, base, None, 2, 8, 2, 2, None, 0, None) == spl.SPL_EINVAL  # no weight
    assert L.spl_masked_linear(base, base, ctypes.byref(w), 2, 6, 2, 2, None, 0, None) == spl.SPL_EALIGN
    assert L.spl_masked_linear(base + 4, base, ctypes.byref(w), 2, 8, 2, 2, None, 0, None) == spl.SPL_EALIGN
    w_bad = spl.spl_weight(base, None, None, base + 2, base, base)
    assert L.spl_masked_linear(base, base, ctypes.byref(w_bad), 2, 8, 2, 2, None, 0, None) == spl.SPL_EALIGN
    assert L.spl_masked_linear_unmask(base, base, ctypes.byref(w), None, 2, 8, 2, 2, None, 0, None) == spl.SPL_EINVAL
    assert L.spl_random_bits(None, -1, rng, None) == spl.SPL_EINVAL
    assert L.spl_split_tf32(base + 4, base, base, 4, None) == spl.SPL_EALIGN
    assert L.spl_split_fp16(base, base, base, base, 2, 12, None) == spl.SPL_EALIGN  # cols % 8
    assert L.spl_split_fp16(base, base, None, base, 2, 8, None) == spl.SPL_EINVAL
    assert L.spl_split_fp16(None, None, None, None, 0, 8, None) == spl.SPL_OK
    assert L.spl_noise_mask_f64(None, None, 4, 4, 1.0, 1.0, 0, rng, None) == spl.SPL_EINVAL
    assert L.spl_masked_linear_unmask_f64(base, base, base, base, 2, 6, 2, None, 0, None) == spl.SPL_EALIGN
    assert L.spl_precompute_noise_product_f64(None, base, base, 2, 8, 2, None, 0, None) == spl.SPL_EINVAL
    assert L.spl_precompute_noise_product_f64(None, None, None, 0, 8, 2, None, 0, None) == spl.SPL_OK
    assert L.spl_slalom_quantize(None, None, -1, None) == spl.SPL_EINVAL
    assert L.spl_slalom_mask(None, None, None, 0, 3, rng, None) == spl.SPL_OK
    assert L.spl_slalom_linear_unmask(base, base, base, base, 1, 1 << 22, 1, None, 0, None) == spl.SPL_ESHAPE
    # the mask fused with the fp16 split (drawn or stored noise)
    assert L.spl_mask_split(None, base, base, base, base, base, -1, 8, None) == spl.SPL_EINVAL
    assert L.spl_mask_split(None, None, None, None, None, None, 0, 8, None) == spl.SPL_OK
    assert L.spl_mask_split(None, None, base, base, base, base, 2, 8, None) == spl.SPL_EINVAL  # NULL hi
    assert L.spl_mask_split(None, base, base, base, base, None, 2, 8, None) == spl.SPL_EINVAL  # NULL noise
    assert L.spl_mask_split(None, base, base, base, base, base, 2, 12, None) == spl.SPL_EALIGN  # cols % 8
    assert L.spl_mask_split(None, base, base, base, base + 4, base, 2, 8, None) == spl.SPL_EALIGN
    assert L.spl_mask_split(None, base, base, base, base, base, 1, 16392, None) == spl.SPL_ESHAPE  # row too long
    assert L.spl_noise_mask_split(None, base, base, base, base, 2, 12, 1.0, 1.0, 0, rng, None) == spl.SPL_EALIGN
    assert L.spl_noise_mask_split(None, None, base, base, base, 2, 8, 1.0, 1.0, 0, rng, None) == spl.SPL_EINVAL
    # the stacked split: negative counts, a missing X for masked rows, cols % 8
    assert L.spl_noise_mask_split_stacked(base, base, base, base, 2, -1, 8, 1.0, 1.0, 0, rng, 0, None) == spl.SPL_EINVAL
    assert L.spl_noise_mask_split_stacked(base, base, base, None, 2, 2, 8, 1.0, 1.0, 0, rng, 0, None) == spl.SPL_EINVAL
    assert L.spl_noise_mask_split_stacked(base, base, base, base, 2, 2, 12, 1.0, 1.0, 0, rng, 0, None) == spl.SPL_EALIGN
    assert L.spl_noise_mask_split_stacked(None, None, None, None, 0, 0, 8, 1.0, 1.0, 0, rng, 0, None) == spl.SPL_OK
    # the tensor-core test hook refuses a persistent launch that breaks its conditions
    w16 = spl.spl_weight(base, None, None, base, base, base)
    for splits, seg, full in ((2, 0, 0), (1, 2, 0), (1, 0, 1)):
        assert L.spl_test_tc_product(base, base, ctypes.byref(w16), None, 2, 8, 8, spl.SPL_PATH_FP16X3, 256, 192,
                                     splits, full, seg, 1, None, 0, None) == spl.SPL_EINVAL
    assert L.spl_test_tc_product(base, base, ctypes.byref(w16), None, 2, 8, 8, spl.SPL_PATH_FP16X3, 128, 96,
                                 1, 0, 0, 1, None, 0, None) == spl.SPL_EINVAL  # two CTAs per SM: no persistent form
    stats = (ctypes.c_double * 27)()
    chosen = ctypes.c_int(5)
    assert L.spl_choose_path(ctypes.byref(chosen), stats, base, base, None, 4, 8, 8, None, 0, None) == spl.SPL_EINVAL
    assert chosen.value == spl.SPL_PATH_FP32


def test_listed_boundary_names(spl):
    """The names the boundary's call list uses for the weight split and the status calls are exported
    with their listed signatures and behave as the calls they stand for (no launch here)."""
    names = declared_functions()
    for listed in ("spl_prepare_weight_split", "spl_get_last_device_status", "spl_status_str"):
        assert listed in names
    L = spl.lib()
    for st in range(9):
        assert spl.spl_status_str(st) == spl.status_string(st)
    buf = (ctypes.c_float * 64)()
    p = ctypes.cast(buf, ctypes.c_void_p).value
    base = p + (16 - p % 16) % 16
    assert L.spl_prepare_weight_split(None, None, None, 0, 8, None) == spl.SPL_OK      # empty
    assert L.spl_prepare_weight_split(None, None, None, -1, 8, None) == spl.SPL_EINVAL
    assert L.spl_prepare_weight_split(None, base, base, 2, 8, None) == spl.SPL_EINVAL  # NULL W_hi
    assert L.spl_prepare_weight_split(base + 4, base, base, 2, 8, None) == spl.SPL_EALIGN
    assert L.spl_prepare_weight_split(base, base, base, 1 << 40, 1 << 40, None) == spl.SPL_ESHAPE


def test_precompute_and_swap_entries_validate_without_launch(spl):
    """The stacked product entry and the swapped-kernel hook refuse bad arguments before launching."""
    L = spl.lib()
    buf = (ctypes.c_float * 64)()
    p = ctypes.cast(buf, ctypes.c_void_p).value
    base = p + (16 - p % 16) % 16
    w = spl.spl_weight(base, None, None, None, None, None)
    a = spl.spl_weight(base, None, None, None, None, None)
    pre = L.spl_masked_linear_unmask_precompute
    assert pre(base, None, ctypes.byref(w), base, 2, 2, 8, 4, 0, None, 0, None) == spl.SPL_EINVAL   # no A
    assert pre(base, ctypes.byref(a), ctypes.byref(w), base, -1, 2, 8, 4, 0, None, 0, None) == spl.SPL_EINVAL
    assert pre(base, ctypes.byref(a), ctypes.byref(w), None, 2, 2, 8, 4, 0, None, 0, None) == spl.SPL_EINVAL  # C
    assert pre(base, ctypes.byref(a), ctypes.byref(w), None, 0, 0, 8, 4, 0, None, 0, None) == spl.SPL_OK      # empty
    # no tensor-core device here, so AUTO resolves to FP32: beyond 16 rows that is the SIMT kernel,
    # which has no row limit on C
    assert pre(base, ctypes.byref(a), ctypes.byref(w), base, 9, 8, 8, 4, 0, None, 0, None) == spl.SPL_EUNSUPPORTED
    fused = L.spl_noise_mask_linear_unmask_precompute
    rng = spl._rng(1, 0, 0, None)
    lap = spl._mech("laplace")

    def call(Xt, X, C, M, M_bank, eps=1.0, path=0, rng_=rng):
        return fused(base, Xt, X, ctypes.byref(w), C, M, M_bank, 8, 4, 1.0, eps, lap, rng_, 64, path, None, 0, None)

    assert call(base, base + 128, base, 1, 1, eps=-1.0) == spl.SPL_EINVAL         # eps
    assert call(base, base + 128, None, 1, 1) == spl.SPL_EINVAL                   # no C for the masked row
    assert call(base, base + 128, base, 0, 0) == spl.SPL_OK                       # empty
    assert call(base, base + 128, base, 2, 3) == spl.SPL_EUNSUPPORTED             # 5 rows: not one decode launch
    assert call(base, base + 128, base, 1, 1, path=spl._path("fp16x3")) == spl.SPL_EUNSUPPORTED
    assert call(base + 4, base + 128, base, 1, 1) == spl.SPL_EALIGN               # Xt
    assert call(base, base + 16, base, 1, 1) == spl.SPL_EINVAL                    # X overlaps Xt's two rows
    assert call(base, None, base, 1, 1) == spl.SPL_EINVAL                         # no X for the masked row
    assert call(base, base + 128, base, 1, 1, rng_=spl.spl_rng(1, 0, 0, base + 4)) == spl.SPL_EALIGN  # offset_dev
    swap = L.spl_test_tc_swap_product
    assert swap(base, base, ctypes.byref(w), None, 2, 8, 4, 24, 1, None, 0, None) == spl.SPL_EINVAL  # width
    assert swap(base, base, ctypes.byref(w), None, 2, 8, 4, 16, -1, None, 0, None) == spl.SPL_EINVAL  # ctas
    # valid arguments reach the device check: no tensor-core device here
    assert swap(base, base, ctypes.byref(w), None, 2, 8, 4, 16, 0, None, 0, None) == spl.SPL_EUNSUPPORTED
    assert L.spl_test_tc_swap_workspace_bytes(2, 8, 4, 24, 0) == 0  # width not listed
    assert L.spl_test_tc_swap_workspace_bytes(2, 64, 256, 16, 3) >= 64 * 1024 + 2 * 2 * 16 * 128 * 4
    assert swap(base, base, ctypes.byref(w), None, 2, 12, 4, 16, 1, None, 0, None) == spl.SPL_EALIGN  # K % 8
    assert swap(base, base, None, None, 2, 8, 4, 16, 1, None, 0, None) == spl.SPL_EINVAL


def test_split_operand_workspace(spl):
    """A product given its left operand split needs only the swapped kernel's counters and partial
    tiles (9-16 rows on FP16X3) and nothing for the kernels that reduce on chip; invalid arguments
    ask for nothing."""
    few = spl.spl_split_workspace_bytes(16, 3072, 5120, path="fp16x3")
    assert few >= 64 * 1024 + 2 * 16 * 128 * 4
    assert few < spl.spl_linear_workspace_bytes(16, 3072, 5120, "fp16x3")  # no room for the split itself
    assert spl.spl_split_workspace_bytes(128, 3072, 5120, path="fp16x3") == 0
    assert spl.spl_split_workspace_bytes(1024, 3072, 5120, 512, path="fp16x3") == 0
    # a bank of 8 draws in the order of 16-row products: the wider token tile's partial tiles
    assert spl.spl_split_workspace_bytes(128, 3072, 5120, 16, path="fp16x3") > few
    assert spl.spl_split_workspace_bytes(0, 3072, 5120, path="fp16x3") == 0
    assert spl.spl_split_workspace_bytes(16, 3072, 5120, path=9) == 0


def test_copy_2d_validates_without_a_copy(spl):
    """The host-link copy refuses null pointers and rows wider than a pitch before it queues anything;
    nothing to copy is a no-op."""
    L = spl.lib()
    buf = ctypes.create_string_buffer(64)
    p = ctypes.addressof(buf)
    assert L.spl_copy_2d(None, 16, p, 16, 8, 2, None) == spl.SPL_EINVAL
    assert L.spl_copy_2d(p, 16, None, 16, 8, 2, None) == spl.SPL_EINVAL
    assert L.spl_copy_2d(p, 8, p, 16, 16, 2, None) == spl.SPL_EINVAL  # wider than the destination pitch
    assert L.spl_copy_2d(p, 16, p, 8, 16, 2, None) == spl.SPL_EINVAL  # wider than the source pitch
    assert L.spl_copy_2d(None, 0, None, 0, 8, 0, None) == spl.SPL_OK
    assert L.spl_copy_2d(None, 0, None, 0, 0, 3, None) == spl.SPL_OK
    import torch
    with pytest.raises(ValueError):  # the binding checks the extent against the tensors
        spl.spl_copy_2d(torch.zeros(4), torch.zeros(8), 2, 16, 16, 16)


def test_workspace_sizes_are_consistent(spl):
    # decode shapes need split-K partials after the 64 KiB counter region; the tensor-core
    # kernels reduce split-K in a cluster and keep only the split of the left operand there
    # (TF32X3: hi and lo in fp32; FP16X3: row exponents, hi and lo in fp16)
    for M, K, N in [(1, 3072, 3072), (16, 8192, 3072), (128, 3072, 1024), (2048, 2560, 9728)]:
        auto = spl.spl_linear_workspace_bytes(M, K, N, "auto")
        assert auto >= spl.spl_linear_workspace_bytes(M, K, N, "fp32")
        assert auto >= spl.spl_linear_workspace_bytes(M, K, N, "tf32x3")
        assert auto >= spl.spl_linear_workspace_bytes(M, K, N, "fp16x3")
        assert spl.spl_linear_workspace_bytes(M, K, N, "tf32x3") >= 64 * 1024 + 8 * M * K
        assert spl.spl_linear_workspace_bytes(M, K, N, "fp16x3") >= 64 * 1024 + 4 * M + 4 * M * K
        assert spl.spl_precompute_matched_workspace_bytes(8 * M, K, N, M, "fp16x3") >= 64 * 1024 + 32 * M * (1 + K)
    assert spl.spl_linear_workspace_bytes(1, 3072, 3072, "fp32") > 64 * 1024
    assert spl.spl_linear_workspace_bytes(0, 8, 8) == 0


def test_sensitivities_match_oracle(spl):
    rng = np.random.default_rng(0)
    for d, d_ff in ((256, 512), (3072, 8192)):
        alpha = rng.standard_normal(d).astype(np.float32)
        beta = rng.standard_normal(d).astype(np.float32) * 0.1
        assert spl.spl_delta_layernorm(alpha) == pytest.approx(osens.delta_layernorm(alpha), rel=1e-12)
        assert spl.spl_delta_attention(alpha, 1.7) == pytest.approx(osens.delta_attention(alpha, 1.7), rel=1e-12)
        got = spl.spl_delta_activation(alpha, beta, d_ff, 2.9, 3.1)
        assert got == pytest.approx(osens.delta_activation(alpha, beta, d_ff, 2.9, 3.1), rel=1e-12)
        assert spl.spl_delta_activation(alpha, None, d_ff, 2.0, 2.0) == pytest.approx(
            osens.delta_activation(alpha, None, d_ff, 2.0, 2.0), rel=1e-12)
    ones = np.ones(3072, dtype=np.float32)
    assert spl.spl_delta_layernorm(ones) == pytest.approx(2 * 3072 ** 0.75, rel=1e-12)
    assert spl.lib().spl_delta_layernorm(None, 4) < 0
    assert math.isfinite(spl.spl_delta_layernorm(ones))
