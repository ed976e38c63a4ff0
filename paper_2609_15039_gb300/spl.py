"""Thin ctypes binding of libspl.so (include/spl.h), same function names.

Only argument marshalling happens here: shapes are read off the tensors,
pointers and the current CUDA stream are passed through, and a non-OK
status raises ``SplError``.  Every step of the path runs in the library's
CUDA kernels; there is no fallback.  The library is loaded on first use and
its absence is an error.
"""

import ctypes
import math
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libspl.so")

SPL_OK, SPL_EINVAL, SPL_ESHAPE, SPL_EALIGN, SPL_ECUDA, SPL_ETIMEOUT, SPL_EUNSUPPORTED, SPL_EWORKSPACE = range(8)
SPL_MECH_LAPLACE, SPL_MECH_GAUSSIAN = 0, 1
SPL_PATH_AUTO, SPL_PATH_TF32X3, SPL_PATH_FP32, SPL_PATH_FP16X3 = 0, 1, 2, 3
MECHS = {"laplace": SPL_MECH_LAPLACE, "gaussian": SPL_MECH_GAUSSIAN}
PATHS = {"auto": SPL_PATH_AUTO, "tf32x3": SPL_PATH_TF32X3, "fp32": SPL_PATH_FP32, "fp16x3": SPL_PATH_FP16X3}
PATH_NAMES = {v: k for k, v in PATHS.items()}


class SplError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        super().__init__(f"{where} failed: {status_string(status)} ({status})")


class spl_rng(ctypes.Structure):
    _fields_ = [("seed", ctypes.c_uint64), ("stream_id", ctypes.c_uint64), ("offset", ctypes.c_uint64),
                ("offset_dev", ctypes.c_void_p)]


class spl_weight(ctypes.Structure):
    _fields_ = [("w", ctypes.c_void_p), ("tf32_hi", ctypes.c_void_p), ("tf32_lo", ctypes.c_void_p),
                ("f16_hi", ctypes.c_void_p), ("f16_lo", ctypes.c_void_p), ("f16_exp", ctypes.c_void_p)]


_P = ctypes.c_void_p
_PW = ctypes.POINTER(spl_weight)
_I64 = ctypes.c_int64
_D = ctypes.c_double
_I = ctypes.c_int
_SZ = ctypes.c_size_t
_SIGS = {
    "spl_noise": (_I, [_P, _I64, _I64, _D, _D, _I, spl_rng, _P]),
    "spl_random_bits": (_I, [_P, _I64, spl_rng, _P]),
    "spl_rng_advance": (_I, [_P, ctypes.c_uint64, _P]),
    "spl_mask": (_I, [_P, _P, _P, _I64, _I64, _P]),
    "spl_noise_mask_f64": (_I, [_P, _P, _I64, _I64, _D, _D, _I, spl_rng, _P]),
    "spl_f64_workspace_bytes": (_SZ, [_I64, _I64, _I64]),
    "spl_slalom_quantize": (_I, [_P, _P, _I64, _P]),
    "spl_slalom_mask": (_I, [_P, _P, _P, _I64, _I64, spl_rng, _P]),
    "spl_slalom_linear_unmask": (_I, [_P, _P, _P, _P, _I64, _I64, _I64, _P, _SZ, _P]),
    "spl_precompute_noise_product_f64": (_I, [_P, _P, _P, _I64, _I64, _I64, _P, _SZ, _P]),
    "spl_masked_linear_unmask_f64": (_I, [_P, _P, _P, _P, _I64, _I64, _I64, _P, _SZ, _P]),
    "spl_noise_mask": (_I, [_P, _P, _P, _I64, _I64, _D, _D, _I, spl_rng, _P]),
    "spl_split_tf32": (_I, [_P, _P, _P, _I64, _P]),
    "spl_noise_mask_split": (_I, [_P, _P, _P, _P, _P, _I64, _I64, _D, _D, _I, spl_rng, _P]),
    "spl_mask_split": (_I, [_P, _P, _P, _P, _P, _P, _I64, _I64, _P]),
    "spl_noise_mask_split_stacked": (_I, [_P, _P, _P, _P, _I64, _I64, _I64, _D, _D, _I, spl_rng, ctypes.c_uint64,
                                          _P]),
    "spl_masked_linear_unmask_split": (_I, [_P, _PW, _PW, _P, _I64, _I64, _I64, _I, _P, _SZ, _P]),
    "spl_split_fp16": (_I, [_P, _P, _P, _P, _I64, _I64, _P]),
    "spl_resolve_path": (_I, [_I64, _I64, _I64, _I]),
    "spl_linear_workspace_bytes": (_SZ, [_I64, _I64, _I64, _I]),
    "spl_masked_linear": (_I, [_P, _P, _PW, _I64, _I64, _I64, _I, _P, _SZ, _P]),
    "spl_precompute_noise_product": (_I, [_P, _P, _PW, _I64, _I64, _I64, _I, _P, _SZ, _P]),
    "spl_precompute_matched_workspace_bytes": (_SZ, [_I64, _I64, _I64, _I64, _I]),
    "spl_split_workspace_bytes": (_SZ, [_I64, _I64, _I64, _I64, _I]),
    "spl_precompute_noise_product_matched": (_I, [_P, _P, _PW, _I64, _I64, _I64, _I64, _I, _P, _SZ, _P]),
    "spl_precompute_noise_product_matched_split": (_I, [_P, _PW, _PW, _I64, _I64, _I64, _I64, _I, _P, _SZ, _P]),
    "spl_unmask": (_I, [_P, _P, _P, _I64, _I64, _P]),
    "spl_masked_linear_unmask": (_I, [_P, _P, _PW, _P, _I64, _I64, _I64, _I, _P, _SZ, _P]),
    "spl_masked_linear_unmask_noalloc": (_I, [_P, _P, _P, _P, _I64, _I64, _I64, _P]),
    "spl_masked_linear_unmask_precompute": (_I, [_P, _PW, _PW, _P, _I64, _I64, _I64, _I64, _I, _P, _SZ, _P]),
    "spl_noise_mask_linear_unmask": (_I, [_P, _P, _P, _PW, _P, _I64, _I64, _I64, _D, _D, _I, spl_rng, _I, _P, _SZ,
                                          _P]),
    "spl_noise_mask_linear_unmask_precompute": (_I, [_P, _P, _P, _PW, _P, _I64, _I64, _I64, _I64, _D, _D, _I,
                                                     spl_rng, ctypes.c_uint64, _I, _P, _SZ, _P]),
    "spl_test_tc_swap_workspace_bytes": (_SZ, [_I64, _I64, _I64, _I, _I]),
    "spl_delta_layernorm": (_D, [_P, _I64]),
    "spl_delta_attention": (_D, [_P, _I64, _D]),
    "spl_delta_activation": (_D, [_P, _P, _I64, _I64, _D, _D]),
    "spl_spectral_norm": (_I, [ctypes.POINTER(ctypes.c_double), _P, _I64, _I64, _I, _P, _SZ, _P]),
    "spl_bound_check": (_I, [ctypes.POINTER(ctypes.c_double), _P, _P, _P, _P, _P, _I64, _I64, _I64, _P, _SZ, _P]),
    "spl_choose_path_workspace_bytes": (_SZ, [_I64, _I64, _I64]),
    "spl_choose_path": (_I, [ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_double), _P, _P, _PW, _I64,
                             _I64, _I64, _P, _SZ, _P]),
    "spl_test_tc_wait_timeout": (_I, [_P, _P, _PW, _I64, _I64, _I64, _P, _SZ, _P]),
    "spl_test_tc_capacity": (_I, [_I64, _I64, _I64, ctypes.POINTER(ctypes.c_int64)]),
    "spl_test_tc_shape": (_I, [_I64, _I64, _I64, _I64, ctypes.POINTER(ctypes.c_int64)]),
    "spl_test_tc_product": (_I, [_P, _P, _PW, _P, _I64, _I64, _I64, _I, _I, _I, _I, _I64, _I, _I, _P, _SZ, _P]),
    "spl_test_tc_swap_product": (_I, [_P, _P, _PW, _P, _I64, _I64, _I64, _I, _I, _P, _SZ, _P]),
    "spl_get_device_status": (_I, [_P]),
    "spl_launch_count": (ctypes.c_uint64, []),
    "spl_status_string": (ctypes.c_char_p, [_I]),
    "spl_prepare_weight_split": (_I, [_P, _P, _P, _I64, _I64, _P]),
    "spl_get_last_device_status": (_I, [_P]),
    "spl_status_str": (ctypes.c_char_p, [_I]),
    "spl_copy_2d": (_I, [_P, _SZ, _P, _SZ, _SZ, _SZ, _P]),
}

_lib = None


def lib():
    """Load libspl.so (once) and declare its signatures."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built; run `python -m paper_2609_15039_gb300.build`")
        handle = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            fn = getattr(handle, name)
            fn.restype = res
            fn.argtypes = args
        _lib = handle
    return _lib


def status_string(status):
    return lib().spl_status_string(int(status)).decode()


def _check(status, where):
    if status != SPL_OK:
        raise SplError(status, where)


def _stream(stream):
    if stream is None:
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, torch.cuda.Stream):
        return ctypes.c_void_p(stream.cuda_stream)
    return ctypes.c_void_p(int(stream))


def _dev(t, name, dtype=torch.float32):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype and name != "workspace":
        raise TypeError(f"{name} must be {dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _rows_cols(t):
    if t.dim() == 1:
        return 1, t.shape[0]
    return int(math.prod(t.shape[:-1])), int(t.shape[-1])


def _mech(mech):
    return MECHS[mech] if isinstance(mech, str) else int(mech)


def _path(path):
    return PATHS[path] if isinstance(path, str) else int(path)


def _eps(eps):
    return float("inf") if eps is None else float(eps)


def _rng(seed, stream_id, offset, offset_dev):
    """offset_dev: None or a one-element int64 CUDA tensor added on the device to offset."""
    if offset_dev is not None and (offset_dev.dtype != torch.int64 or not offset_dev.is_cuda):
        raise TypeError("offset_dev must be an int64 CUDA tensor")
    return spl_rng(seed % 2**64, stream_id % 2**64, offset % 2**64,
                   None if offset_dev is None else offset_dev.data_ptr())


def spl_noise(N, sensitivity, eps, mech, seed, stream_id=0, offset=0, stream=None, offset_dev=None):
    rows, cols = _rows_cols(N)
    _check(lib().spl_noise(_dev(N, "N"), rows, cols, float(sensitivity), _eps(eps), _mech(mech),
                           _rng(seed, stream_id, offset, offset_dev), _stream(stream)), "spl_noise")


def spl_random_bits(out, seed, stream_id=0, offset=0, stream=None, offset_dev=None):
    """Raw Philox words into a CUDA int32/uint32 tensor (bit pattern of the uint32 stream)."""
    if not out.is_cuda or out.element_size() != 4 or not out.is_contiguous():
        raise TypeError("out must be a contiguous 4-byte CUDA tensor")
    _check(lib().spl_random_bits(ctypes.c_void_p(out.data_ptr()), out.numel(), _rng(seed, stream_id, offset, offset_dev),
                                 _stream(stream)), "spl_random_bits")


def spl_rng_advance(offset_dev, delta, stream=None):
    if offset_dev.dtype != torch.int64 or not offset_dev.is_cuda:
        raise TypeError("offset_dev must be an int64 CUDA tensor")
    _check(lib().spl_rng_advance(ctypes.c_void_p(offset_dev.data_ptr()), int(delta) % 2**64, _stream(stream)),
           "spl_rng_advance")


def spl_mask(Xt, X, N, stream=None):
    rows, cols = _rows_cols(X)
    _check(lib().spl_mask(_dev(Xt, "Xt"), _dev(X, "X"), _dev(N, "N"), rows, cols, _stream(stream)), "spl_mask")


def spl_noise_mask(Xt, N_out, X, sensitivity, eps, mech, seed, stream_id=0, offset=0, stream=None, offset_dev=None):
    rows, cols = _rows_cols(X)
    _check(lib().spl_noise_mask(_dev(Xt, "Xt"), _dev(N_out, "N_out"), _dev(X, "X"), rows, cols, float(sensitivity),
                                _eps(eps), _mech(mech), _rng(seed, stream_id, offset, offset_dev), _stream(stream)),
           "spl_noise_mask")


def spl_noise_mask_f64(Xt, X, sensitivity, eps, mech, seed, stream_id=0, offset=0, stream=None, offset_dev=None):
    """Binary64 mask (Sec. 5.5): Xt float64 = X + eta, eta as spl_noise draws it."""
    rows, cols = _rows_cols(X)
    if Xt.numel() != rows * cols:
        raise ValueError("spl_noise_mask_f64: shape mismatch")
    _check(lib().spl_noise_mask_f64(_dev(Xt, "Xt", torch.float64), _dev(X, "X"), rows, cols, float(sensitivity),
                                    _eps(eps), _mech(mech), _rng(seed, stream_id, offset, offset_dev),
                                    _stream(stream)), "spl_noise_mask_f64")


def spl_f64_workspace_bytes(M, K, N):
    return int(lib().spl_f64_workspace_bytes(M, K, N))


def spl_precompute_noise_product_f64(C, Nz, W, workspace=None, stream=None):
    """C float64 [M, N] = Nz W^T in binary64 (Nz, W fp32)."""
    M, K = _rows_cols(Nz)
    N = W.shape[0]
    if W.shape[-1] != K or C.numel() != M * N:
        raise ValueError("spl_precompute_noise_product_f64: shape mismatch")
    if workspace is None:
        workspace = globals()["workspace"](spl_f64_workspace_bytes(M, K, N), Nz.device)
    wsp, wsb = _ws(workspace)
    _check(lib().spl_precompute_noise_product_f64(_dev(C, "C", torch.float64), _dev(Nz, "Nz"), _dev(W, "W"), M, K, N,
                                                  wsp, wsb, _stream(stream)), "spl_precompute_noise_product_f64")


def spl_masked_linear_unmask_f64(Y, Xt, W, C, workspace=None, stream=None):
    """Y fp32 = fl32(Xt W^T - C) with Xt and C float64 (binary64 sums)."""
    M, K = _rows_cols(Xt)
    N = W.shape[0]
    if W.shape[-1] != K or Y.numel() != M * N or C.numel() != M * N:
        raise ValueError("spl_masked_linear_unmask_f64: shape mismatch")
    if workspace is None:
        workspace = globals()["workspace"](spl_f64_workspace_bytes(M, K, N), Xt.device)
    wsp, wsb = _ws(workspace)
    _check(lib().spl_masked_linear_unmask_f64(_dev(Y, "Y"), _dev(Xt, "Xt", torch.float64), _dev(W, "W"),
                                              _dev(C, "C", torch.float64), M, K, N, wsp, wsb, _stream(stream)),
           "spl_masked_linear_unmask_f64")


def spl_noise_mask_split(Xt, hi, lo, row_exp, X, sensitivity, eps, mech, seed, stream_id=0, offset=0, stream=None,
                         offset_dev=None):
    """a2 + a3 + the fp16 split of X~ in one pass (Xt may be None; X None: the split of the noise
    itself, of hi's shape)."""
    rows, cols = _rows_cols(X if X is not None else hi)
    if hi.numel() != rows * cols or lo.numel() != rows * cols or row_exp.numel() != rows:
        raise ValueError("spl_noise_mask_split: shape mismatch")
    _check(lib().spl_noise_mask_split(_dev(Xt, "Xt"), _dev(hi, "hi", torch.int16), _dev(lo, "lo", torch.int16),
                                      _dev(row_exp, "row_exp", torch.int32), _dev(X, "X"), rows, cols,
                                      float(sensitivity), _eps(eps), _mech(mech),
                                      _rng(seed, stream_id, offset, offset_dev), _stream(stream)),
           "spl_noise_mask_split")


def spl_noise_mask_split_stacked(hi, lo, row_exp, X, sensitivity, eps, mech, seed, noise_rows, noise_block_delta,
                                 stream_id=0, offset=0, stream=None, offset_dev=None):
    """Split of [X + eta; eta'] in one pass: rows of X masked and split, then noise_rows rows of noise
    alone drawn noise_block_delta Philox blocks further on (see include/spl.h)."""
    x_rows, cols = _rows_cols(X)
    rows = x_rows + int(noise_rows)
    if hi.numel() != rows * cols or lo.numel() != rows * cols or row_exp.numel() != rows:
        raise ValueError("spl_noise_mask_split_stacked: shape mismatch")
    _check(lib().spl_noise_mask_split_stacked(_dev(hi, "hi", torch.int16), _dev(lo, "lo", torch.int16),
                                              _dev(row_exp, "row_exp", torch.int32), _dev(X, "X"), x_rows,
                                              int(noise_rows), cols, float(sensitivity), _eps(eps), _mech(mech),
                                              _rng(seed, stream_id, offset, offset_dev), int(noise_block_delta),
                                              _stream(stream)), "spl_noise_mask_split_stacked")


def spl_mask_split(Xt, hi, lo, row_exp, X, N, stream=None):
    """a3 with a stored noise N + the fp16 split of X~ in one pass (Xt may be None)."""
    rows, cols = _rows_cols(X)
    if (N.numel() != rows * cols or hi.numel() != rows * cols or lo.numel() != rows * cols
            or row_exp.numel() != rows):
        raise ValueError("spl_mask_split: shape mismatch")
    _check(lib().spl_mask_split(_dev(Xt, "Xt"), _dev(hi, "hi", torch.int16), _dev(lo, "lo", torch.int16),
                                _dev(row_exp, "row_exp", torch.int32), _dev(X, "X"), _dev(N, "N"), rows, cols,
                                _stream(stream)),
           "spl_mask_split")


def spl_masked_linear_unmask_split(Y, Xt, W, C, path="auto", workspace=None, stream=None):
    """Xt: a Weight holding X~ (w, may be None on FP16X3) and its fp16 split; W: a Weight."""
    W = _weight(W)
    M, K = Xt.shape
    N = W.shape[0]
    if W.shape[-1] != K or Y.numel() != M * N or C.numel() != M * N:
        raise ValueError("spl_masked_linear_unmask_split: shape mismatch")
    wsp, wsb = _ws(workspace)
    xs, ws_ = Xt.c_struct(), W.c_struct()
    _check(lib().spl_masked_linear_unmask_split(_dev(Y, "Y"), ctypes.byref(xs), ctypes.byref(ws_), _dev(C, "C"), M, K,
                                                N, _path(path), wsp, wsb, _stream(stream)),
           "spl_masked_linear_unmask_split")


def spl_masked_linear_unmask_precompute(YC, A, W, C, M, path="auto", workspace=None, stream=None):
    """The masked product of the first M rows of A with its unmask and the corrections of A's other rows
    in one launch: YC [M + M_bank, N], A a Weight over [M + M_bank, K] (fp32 and/or fp16 split),
    C [M, N]."""
    A, W = _weight(A), _weight(W)
    rows, K = A.shape
    N = W.shape[0]
    M_bank = rows - int(M)
    if W.shape[-1] != K or YC.numel() != rows * N or M_bank < 0 or (C is not None and C.numel() != int(M) * N):
        raise ValueError("spl_masked_linear_unmask_precompute: shape mismatch")
    wsp, wsb = _ws(workspace)
    xs, ws_ = A.c_struct(), W.c_struct()
    _check(lib().spl_masked_linear_unmask_precompute(_dev(YC, "YC"), ctypes.byref(xs), ctypes.byref(ws_),
                                                     _dev(C, "C"), int(M), M_bank, K, N, _path(path), wsp, wsb,
                                                     _stream(stream)), "spl_masked_linear_unmask_precompute")


def spl_slalom_quantize(out, v, stream=None):
    """Slalom fixed point (Sec. 6.2): out = rint(v 2^8) as fp32 integers."""
    _check(lib().spl_slalom_quantize(_dev(out, "out"), _dev(v, "v"), v.numel(), _stream(stream)), "spl_slalom_quantize")


def spl_slalom_mask(Xt_q, eta_out, X, seed, stream_id=0, offset=0, stream=None):
    """Slalom mask: Xt_q = (rint(X 2^8) mod q + eta) mod q, eta uniform in Z_q (fp32 integers)."""
    rows, cols = _rows_cols(X)
    _check(lib().spl_slalom_mask(_dev(Xt_q, "Xt_q"), _dev(eta_out, "eta_out"), _dev(X, "X"), rows, cols,
                                 _rng(seed, stream_id, offset, None), _stream(stream)), "spl_slalom_mask")


def spl_slalom_linear_unmask(Y, Xt_q, W_q, C, workspace=None, stream=None):
    """Y = de-quantized ((Xt_q W_q^T - C) mod q), the product exact in binary64."""
    M, K = _rows_cols(Xt_q)
    N = W_q.shape[0]
    if W_q.shape[-1] != K or Y.numel() != M * N or C.numel() != M * N:
        raise ValueError("spl_slalom_linear_unmask: shape mismatch")
    if workspace is None:
        workspace = globals()["workspace"](spl_f64_workspace_bytes(M, K, N), Xt_q.device)
    wsp, wsb = _ws(workspace)
    _check(lib().spl_slalom_linear_unmask(_dev(Y, "Y"), _dev(Xt_q, "Xt_q"), _dev(W_q, "W_q"),
                                          _dev(C, "C", torch.float64), M, K, N, wsp, wsb, _stream(stream)),
           "spl_slalom_linear_unmask")


def spl_split_tf32(hi, lo, src, stream=None):
    _check(lib().spl_split_tf32(_dev(hi, "hi"), _dev(lo, "lo"), _dev(src, "src"), src.numel(), _stream(stream)),
           "spl_split_tf32")


def spl_prepare_weight_split(W_hi, W_lo, W, stream=None):
    """The boundary's listed name for the TF32X3 weight split (spl_split_tf32 over W[N, K])."""
    N, K = W.shape
    if tuple(W_hi.shape) != (N, K) or tuple(W_lo.shape) != (N, K):
        raise ValueError("spl_prepare_weight_split: shape mismatch")
    _check(lib().spl_prepare_weight_split(_dev(W_hi, "W_hi"), _dev(W_lo, "W_lo"), _dev(W, "W"), N, K,
                                          _stream(stream)), "spl_prepare_weight_split")


def spl_split_fp16(hi, lo, row_exp, src, stream=None):
    """hi, lo: int16 [rows, cols] (binary16 bit patterns); row_exp: int32 [rows]."""
    rows, cols = _rows_cols(src)
    if hi.numel() != rows * cols or lo.numel() != rows * cols or row_exp.numel() != rows:
        raise ValueError("spl_split_fp16: shape mismatch")
    _check(lib().spl_split_fp16(_dev(hi, "hi", torch.int16), _dev(lo, "lo", torch.int16),
                                _dev(row_exp, "row_exp", torch.int32), _dev(src, "src"), rows, cols, _stream(stream)),
           "spl_split_fp16")


class Weight:
    """A device weight W [N, K] (fp32) with the splits the tensor-core paths read (spl_weight).

    ``Weight.prepare(W)`` runs the library's split kernels once; the splits live as long as
    this object.  A plain tensor passed where a weight is expected carries no split (FP32
    path only)."""

    def __init__(self, w, tf32_hi=None, tf32_lo=None, f16_hi=None, f16_lo=None, f16_exp=None):
        self.w, self.tf32_hi, self.tf32_lo = w, tf32_hi, tf32_lo
        self.f16_hi, self.f16_lo, self.f16_exp = f16_hi, f16_lo, f16_exp

    @classmethod
    def prepare(cls, w, tf32=True, fp16=True, stream=None):
        out = cls(w)
        if tf32:
            out.tf32_hi, out.tf32_lo = torch.empty_like(w), torch.empty_like(w)
            spl_split_tf32(out.tf32_hi, out.tf32_lo, w, stream=stream)
        if fp16 and w.shape[-1] % 8 == 0:
            out.f16_hi = torch.empty(w.shape, dtype=torch.int16, device=w.device)
            out.f16_lo = torch.empty_like(out.f16_hi)
            out.f16_exp = torch.empty(w.shape[0], dtype=torch.int32, device=w.device)
            spl_split_fp16(out.f16_hi, out.f16_lo, out.f16_exp, w, stream=stream)
        return out

    @property
    def shape(self):
        return self.w.shape if self.w is not None else self.f16_hi.shape

    def rows(self, a, b):
        """Rows a:b (output columns a:b of the product) as a Weight of views."""
        sl = lambda t: None if t is None else t[a:b]
        return Weight(self.w[a:b], sl(self.tf32_hi), sl(self.tf32_lo), sl(self.f16_hi), sl(self.f16_lo),
                      sl(self.f16_exp))

    def c_struct(self):
        return spl_weight(_dev(self.w, "W"), _dev(self.tf32_hi, "W.tf32_hi"), _dev(self.tf32_lo, "W.tf32_lo"),
                          _dev(self.f16_hi, "W.f16_hi", torch.int16), _dev(self.f16_lo, "W.f16_lo", torch.int16),
                          _dev(self.f16_exp, "W.f16_exp", torch.int32))


def _weight(W):
    return W if isinstance(W, Weight) else Weight(W)


def spl_resolve_path(M, K, N, path="auto"):
    return lib().spl_resolve_path(M, K, N, _path(path))


def spl_linear_workspace_bytes(M, K, N, path="auto"):
    return int(lib().spl_linear_workspace_bytes(M, K, N, _path(path)))


def workspace(nbytes, device=None):
    """A zero-filled device workspace of at least nbytes (uint8 tensor)."""
    return torch.zeros(max(int(nbytes), 256), dtype=torch.uint8, device=device or "cuda")


def _ws(ws):
    if ws is None:
        return None, 0
    return _dev(ws, "workspace"), ws.numel() * ws.element_size()


def _linear(fn, name, out, a, W, C, path, ws, stream):
    W = _weight(W)
    M, K = _rows_cols(a)
    N = W.shape[0]
    if W.shape[-1] != K or out.numel() != M * N or (C is not None and C.numel() != M * N):
        raise ValueError(f"{name}: shape mismatch")
    wsp, wsb = _ws(ws)
    ws_ = W.c_struct()
    args = [_dev(out, "out"), _dev(a, "input"), ctypes.byref(ws_)]
    if name == "spl_masked_linear_unmask":
        args.append(_dev(C, "C"))
    _check(fn(*args, M, K, N, _path(path), wsp, wsb, _stream(stream)), name)


def spl_masked_linear(Yt, Xt, W, path="auto", workspace=None, stream=None):
    """W: a Weight (or a plain fp32 tensor for the FP32 path)."""
    _linear(lib().spl_masked_linear, "spl_masked_linear", Yt, Xt, W, None, path, workspace, stream)


def spl_precompute_noise_product(C, Nz, W, path="auto", workspace=None, stream=None):
    _linear(lib().spl_precompute_noise_product, "spl_precompute_noise_product", C, Nz, W, None, path, workspace,
            stream)


def spl_split_workspace_bytes(M, K, N, order_rows=None, path="auto"):
    """Workspace bytes of a product (or a correction in the order of order_rows rows) whose left
    operand comes split; 0 when the kernel reduces on chip (see include/spl.h)."""
    return int(lib().spl_split_workspace_bytes(int(M), int(K), int(N), int(M if order_rows is None else order_rows),
                                               _path(path)))


def spl_precompute_matched_workspace_bytes(M, K, N, order_rows, path="auto"):
    return int(lib().spl_precompute_matched_workspace_bytes(M, K, N, order_rows, _path(path)))


def spl_precompute_noise_product_matched(C, Nz, W, order_rows, path="auto", workspace=None, stream=None):
    W = _weight(W)
    M, K = _rows_cols(Nz)
    N = W.shape[0]
    if W.shape[-1] != K or C.numel() != M * N:
        raise ValueError("spl_precompute_noise_product_matched: shape mismatch")
    wsp, wsb = _ws(workspace)
    ws_ = W.c_struct()
    _check(lib().spl_precompute_noise_product_matched(_dev(C, "C"), _dev(Nz, "Nz"), ctypes.byref(ws_), M, K, N,
                                                      int(order_rows), _path(path), wsp, wsb, _stream(stream)),
           "spl_precompute_noise_product_matched")


def spl_precompute_noise_product_matched_split(C, Nz, W, order_rows, path="auto", workspace=None, stream=None):
    """Nz: a Weight holding the noise (w, may be None on FP16X3) and its fp16 split."""
    W = _weight(W)
    M, K = Nz.shape
    N = W.shape[0]
    if W.shape[-1] != K or C.numel() != M * N:
        raise ValueError("spl_precompute_noise_product_matched_split: shape mismatch")
    wsp, wsb = _ws(workspace)
    ns, ws_ = Nz.c_struct(), W.c_struct()
    _check(lib().spl_precompute_noise_product_matched_split(_dev(C, "C"), ctypes.byref(ns), ctypes.byref(ws_), M, K, N,
                                                            int(order_rows), _path(path), wsp, wsb, _stream(stream)),
           "spl_precompute_noise_product_matched_split")


def spl_unmask(Y, Yt, C, stream=None):
    rows, cols = _rows_cols(Yt)
    _check(lib().spl_unmask(_dev(Y, "Y"), _dev(Yt, "Yt"), _dev(C, "C"), rows, cols, _stream(stream)), "spl_unmask")


def spl_masked_linear_unmask(Y, Xt, W, C, path="auto", workspace=None, stream=None):
    _linear(lib().spl_masked_linear_unmask, "spl_masked_linear_unmask", Y, Xt, W, C, path, workspace, stream)


def spl_noise_mask_linear_unmask(Y, Xt, X, W, C, sensitivity, eps, mech, seed, stream_id=0, offset=0, path="auto",
                                 workspace=None, stream=None, offset_dev=None):
    """a2 + a3 + a5 + a6: Xt = X + eta (written), Y = Xt W^T - C; one launch for M <= 4 on FP32."""
    W = _weight(W)
    M, K = _rows_cols(X)
    N = W.shape[0]
    if W.shape[-1] != K or Xt.numel() != M * K or Y.numel() != M * N or C.numel() != M * N:
        raise ValueError("spl_noise_mask_linear_unmask: shape mismatch")
    wsp, wsb = _ws(workspace)
    ws_ = W.c_struct()
    _check(lib().spl_noise_mask_linear_unmask(_dev(Y, "Y"), _dev(Xt, "Xt"), _dev(X, "X"), ctypes.byref(ws_),
                                              _dev(C, "C"), M, K, N, float(sensitivity), _eps(eps), _mech(mech),
                                              _rng(seed, stream_id, offset, offset_dev), _path(path), wsp, wsb,
                                              _stream(stream)),
           "spl_noise_mask_linear_unmask")


def spl_noise_mask_linear_unmask_precompute(YC, Xt, X, W, C, sensitivity, eps, mech, seed, noise_rows,
                                            noise_block_delta, stream_id=0, offset=0, path="auto", workspace=None,
                                            stream=None, offset_dev=None):
    """a2-a6 in one decode launch: rows of X masked and multiplied (unmasked with C), then noise_rows rows
    of noise alone drawn noise_block_delta Philox blocks further on, multiplied (see include/spl.h)."""
    W = _weight(W)
    K = W.shape[-1]
    if X is None:
        M = 0
    else:
        M, K = _rows_cols(X)
    rows = M + int(noise_rows)
    N = W.shape[0]
    if W.shape[-1] != K or Xt.numel() != rows * K or YC.numel() != rows * N or (
            M > 0 and (C is None or C.numel() != M * N)):
        raise ValueError("spl_noise_mask_linear_unmask_precompute: shape mismatch")
    wsp, wsb = _ws(workspace)
    ws_ = W.c_struct()
    _check(lib().spl_noise_mask_linear_unmask_precompute(
        _dev(YC, "YC"), _dev(Xt, "Xt"), _dev(X, "X"), ctypes.byref(ws_), _dev(C, "C") if M > 0 else None, M,
        int(noise_rows), K, N, float(sensitivity), _eps(eps), _mech(mech), _rng(seed, stream_id, offset, offset_dev),
        int(noise_block_delta), _path(path), wsp, wsb, _stream(stream)), "spl_noise_mask_linear_unmask_precompute")


def spl_masked_linear_unmask_noalloc(Y, Xt, W, C, stream=None):
    """Decode product + unmask (M <= 16) using the library's built-in scratch array."""
    M, K = _rows_cols(Xt)
    N = W.shape[0]
    if W.shape[-1] != K or Y.numel() != M * N or C.numel() != M * N:
        raise ValueError("spl_masked_linear_unmask_noalloc: shape mismatch")
    _check(lib().spl_masked_linear_unmask_noalloc(_dev(Y, "Y"), _dev(Xt, "Xt"), _dev(W, "W"), _dev(C, "C"), M, K,
                                                  N, _stream(stream)), "spl_masked_linear_unmask_noalloc")


def _host_f32(t):
    t = torch.as_tensor(t, dtype=torch.float32).contiguous().cpu()
    return t, ctypes.c_void_p(t.data_ptr())


def spl_delta_layernorm(alpha):
    a, p = _host_f32(alpha)
    return lib().spl_delta_layernorm(p, a.numel())


def spl_delta_attention(alpha, wval_spectral_norm):
    a, p = _host_f32(alpha)
    return lib().spl_delta_attention(p, a.numel(), float(wval_spectral_norm))


def spl_delta_activation(alpha, beta, d_ff, wup_spectral_norm, wgate_spectral_norm):
    a, pa = _host_f32(alpha)
    if beta is None:
        pb = None
    else:
        b, pb = _host_f32(beta)
    return lib().spl_delta_activation(pa, pb, a.numel(), int(d_ff), float(wup_spectral_norm),
                                      float(wgate_spectral_norm))


def spl_spectral_norm(W, iters=100, workspace=None, stream=None):
    N, K = W.shape
    ws = workspace if workspace is not None else globals()["workspace"](4 * (N + 2 * K) + 256, W.device)
    wsp, wsb = _ws(ws)
    out = ctypes.c_double(0.0)
    _check(lib().spl_spectral_norm(ctypes.byref(out), _dev(W, "W"), N, K, int(iters), wsp, wsb, _stream(stream)),
           "spl_spectral_norm")
    return out.value


BOUND_STATS = ("max_err_over_hard", "max_err_over_log", "log_violations", "sum_err", "sum_log_bound",
               "sum_hard_bound", "elements", "max_abs_ref", "max_err")


def _stats_dict(arr):
    d = {k: float(v) for k, v in zip(BOUND_STATS, arr)}
    n = max(d["elements"], 1.0)
    d["violation_pct"] = 100.0 * d["log_violations"] / n
    d["mean_err"] = d["sum_err"] / n
    d["mean_log_bound"] = d["sum_log_bound"] / n
    d["log_bound_over_err"] = d["sum_log_bound"] / d["sum_err"] if d["sum_err"] > 0 else float("inf")
    return d


def spl_bound_check(Y, X, Xt, Nz, W, stream=None):
    """The paper's bound on the GPU for every row of Y; returns a dict of statistics."""
    rows, K = _rows_cols(X)
    N = W.shape[0]
    stats = (ctypes.c_double * 9)()
    ws = workspace(256, X.device)
    _check(lib().spl_bound_check(stats, _dev(Y, "Y"), _dev(X, "X"), _dev(Xt, "Xt"), _dev(Nz, "Nz"), _dev(W, "W"),
                                 rows, K, N, _dev(ws, "workspace"), 256, _stream(stream)), "spl_bound_check")
    return _stats_dict(stats)


def spl_choose_path(X, Nz, W, stream=None):
    """a8: returns (chosen path name, {path name: stats}) for the sample X + Nz (W: a Weight)."""
    W = _weight(W)
    rows, K = _rows_cols(X)
    N = W.shape[0]
    nbytes = int(lib().spl_choose_path_workspace_bytes(rows, K, N))
    ws = workspace(nbytes, X.device)
    chosen = ctypes.c_int(0)
    st = (ctypes.c_double * 27)()
    ws_ = W.c_struct()
    _check(lib().spl_choose_path(ctypes.byref(chosen), st, _dev(X, "X"), _dev(Nz, "Nz"), ctypes.byref(ws_), rows, K,
                                 N, _dev(ws, "workspace"), nbytes, _stream(stream)), "spl_choose_path")
    stats = {name: _stats_dict(st[9 * i:9 * (i + 1)]) for i, name in enumerate(("fp32", "tf32x3", "fp16x3"))}
    return PATH_NAMES.get(chosen.value, str(chosen.value)), stats


def spl_test_tc_wait_timeout(out, A, W, workspace=None, stream=None):
    W = _weight(W)
    M, K = _rows_cols(A)
    N = W.shape[0]
    ws_ = W.c_struct()
    if workspace is None:
        workspace = globals()["workspace"](spl_linear_workspace_bytes(M, K, N, "tf32x3"), A.device)
    wsp, wsb = _ws(workspace)
    _check(lib().spl_test_tc_wait_timeout(_dev(out, "out"), _dev(A, "A"), ctypes.byref(ws_), M, K, N, wsp, wsb,
                                          _stream(stream)), "spl_test_tc_wait_timeout")


def spl_test_tc_shape(M, K, N, seg_splits=0):
    """Launch shape of the tensor-core product (or of a correction in a seg_splits-way order):
    (tile width, ring KB, unsplit tiles, split tiles, K-split, persistent)."""
    out = (ctypes.c_int64 * 6)()
    _check(lib().spl_test_tc_shape(int(M), int(K), int(N), int(seg_splits), out), "spl_test_tc_shape")
    return tuple(int(v) for v in out)


def spl_test_tc_capacity(tile_n, ring_kb, cluster):
    """Co-resident clusters of `cluster` CTAs of the launch variant (tile_n, ring_kb)."""
    out = ctypes.c_int64(0)
    _check(lib().spl_test_tc_capacity(int(tile_n), int(ring_kb), int(cluster), ctypes.byref(out)),
           "spl_test_tc_capacity")
    return int(out.value)


def spl_test_tc_product(Y, Xt, W, C=None, path="fp16x3", tile_n=256, ring_kb=192, splits=1, workspace=None,
                        stream=None, full_tiles=0, seg_splits=0, persistent=False):
    """The tensor-core product with a fixed launch variant and K-split, the unsplit tiles optionally in
    segmented mode (a test hook)."""
    W = _weight(W)
    M, K = _rows_cols(Xt)
    N = W.shape[0]
    if W.shape[-1] != K or Y.numel() != M * N or (C is not None and C.numel() != M * N):
        raise ValueError("spl_test_tc_product: shape mismatch")
    if workspace is None:
        workspace = globals()["workspace"](spl_linear_workspace_bytes(M, K, N, path), Xt.device)
    wsp, wsb = _ws(workspace)
    ws_ = W.c_struct()
    _check(lib().spl_test_tc_product(_dev(Y, "Y"), _dev(Xt, "Xt"), ctypes.byref(ws_), _dev(C, "C"), M, K, N,
                                     _path(path), int(tile_n), int(ring_kb), int(splits), int(full_tiles),
                                     int(seg_splits), int(bool(persistent)), wsp, wsb, _stream(stream)),
           "spl_test_tc_product")


def spl_test_tc_swap_workspace_bytes(M, K, N, tile_tokens=16, ctas=0):
    return int(lib().spl_test_tc_swap_workspace_bytes(int(M), int(K), int(N), int(tile_tokens), int(ctas)))


def spl_test_tc_swap_product(Y, Xt, W, C=None, tile_tokens=16, ctas=0, workspace=None, stream=None):
    """The FP16X3 product on the swapped kernel with a fixed token-tile width and CTA count per token
    tile (0: the library's), a test hook."""
    W = _weight(W)
    M, K = _rows_cols(Xt)
    N = W.shape[0]
    if W.shape[-1] != K or Y.numel() != M * N or (C is not None and C.numel() != M * N):
        raise ValueError("spl_test_tc_swap_product: shape mismatch")
    if workspace is None:
        workspace = globals()["workspace"](spl_test_tc_swap_workspace_bytes(M, K, N, tile_tokens, ctas), Xt.device)
    wsp, wsb = _ws(workspace)
    ws_ = W.c_struct()
    _check(lib().spl_test_tc_swap_product(_dev(Y, "Y"), _dev(Xt, "Xt"), ctypes.byref(ws_), _dev(C, "C"), M, K, N,
                                          int(tile_tokens), int(ctas), wsp, wsb, _stream(stream)),
           "spl_test_tc_swap_product")


def spl_copy_2d(dst, src, rows, width_bytes, dst_pitch, src_pitch, stream=None):
    """``rows`` rows of ``width_bytes`` bytes from src to dst, rows ``src_pitch`` / ``dst_pitch`` bytes
    apart (host-link plumbing, not a step of the method).  Each tensor is contiguous and on the GPU
    or in page-locked host memory; the copied extent lies inside both."""
    for t, name, pitch in ((dst, "dst", dst_pitch), (src, "src", src_pitch)):
        if not t.is_contiguous() or not (t.is_cuda or t.is_pinned()):
            raise ValueError(f"spl_copy_2d: {name} must be contiguous, on the GPU or page-locked")
        if rows and width_bytes and (rows - 1) * pitch + width_bytes > t.numel() * t.element_size():
            raise ValueError(f"spl_copy_2d: the copied extent does not fit {name}")
    _check(lib().spl_copy_2d(dst.data_ptr(), int(dst_pitch), src.data_ptr(), int(src_pitch), int(width_bytes),
                             int(rows), _stream(stream)), "spl_copy_2d")


def spl_launch_count():
    return int(lib().spl_launch_count())


def spl_get_device_status(stream=None):
    return lib().spl_get_device_status(_stream(stream))


def spl_get_last_device_status(stream=None):
    """The boundary's listed name for spl_get_device_status."""
    return lib().spl_get_last_device_status(_stream(stream))


def spl_status_str(status):
    """The boundary's listed name for spl_status_string."""
    return lib().spl_status_str(int(status)).decode()
