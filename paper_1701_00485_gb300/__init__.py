"""Two-Bit Networks (arXiv:1701.00485) on GB300: Python binding of libtbn.

Thin ctypes layer over the C ABI declared in ``include/tbn.h``.  Each
function here has the C entry point's name, checks tensor shapes/devices,
passes raw device pointers and the current CUDA stream, and raises
``TBNError`` on a non-OK status.  All arithmetic runs in the CUDA kernels of
``libtbn.so``; there is no CPU path.  PyTorch supplies device memory and
streams only.

The library must have been built (``python -m paper_1701_00485_gb300.build``
or ``__graft_entry__.build()``); importing a function that needs it raises
``RuntimeError`` when ``libtbn.so`` is missing.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

__all__ = [
    "TBNError", "lib", "lib_path", "packed_words",
    "tbn_quantize_pack", "tbn_quantize_pack_group", "tbn_unpack", "tbn_conv2d_fwd",
    "tbn_linear_fwd", "tbn_linear_fwd_ws", "tbn_linear_workspace_bytes",
    "tbn_linear_fwd_noalloc", "tbn_maxpool2d_nhwc", "tbn_nchw_to_nhwc", "tbn_device_error",
    "tbn_conv2d_select_algo", "conv_out_hw", "tbn_conv2d_bwd_data", "tbn_conv2d_bwd_filter",
    "TBN_F32", "TBN_BF16", "TBN_NCHW", "TBN_NHWC", "TBN_NCHW_NHWC", "TBN_UNPACK_I8", "TBN_UNPACK_F32",
    "TBN_UNPACK_BF16", "TBN_CONV_AUTO", "TBN_CONV_DIRECT", "TBN_CONV_IMPLICIT_GEMM",
    "TBN_CONV_SMALL_TAPS", "TBN_DEVERR_TIMEOUT", "TBN_DEVERR_BAD_LAUNCH",
    "tbn_selftest_wait_timeout", "tbn_repack", "TBN_REPACK_CANONICAL_TO_PLANAR",
    "TBN_REPACK_PLANAR_TO_CANONICAL", "tbn_dense_conv2d_fwd", "tbn_avgpool2d_global_nhwc",
    "tbn_dense_linear_fwd", "tbn_space_to_depth", "space_to_depth_shape", "TBN_S2D_NHWC",
    "tbn_linear_prepare_f8", "tbn_linear_f8_workspace_bytes", "tbn_linear_fwd_f8",
    "tbn_linear_f8_prepared_words", "tbn_conv2d_fwd_quant",
]

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "libtbn.so")

TBN_OK, TBN_ERR_INVALID_ARG, TBN_ERR_UNSUPPORTED, TBN_ERR_MISALIGNED, TBN_ERR_CUDA, \
    TBN_ERR_TIMEOUT = range(6)
TBN_F32, TBN_BF16 = 0, 1
TBN_NCHW, TBN_NHWC, TBN_NCHW_NHWC, TBN_S2D_NHWC = 0, 1, 2, 3
TBN_UNPACK_I8, TBN_UNPACK_F32, TBN_UNPACK_BF16 = 0, 1, 2
TBN_CONV_AUTO, TBN_CONV_DIRECT, TBN_CONV_IMPLICIT_GEMM, TBN_CONV_SMALL_TAPS = 0, 1, 2, 3
TBN_MAX_QUANT_JOBS = 16
TBN_DEVERR_TIMEOUT, TBN_DEVERR_BAD_LAUNCH = 1, 2   # bits of the device error word
TBN_REPACK_CANONICAL_TO_PLANAR, TBN_REPACK_PLANAR_TO_CANONICAL = 0, 1

# every symbol include/tbn.h declares
EXPORTED = [
    "tbn_abi_version", "tbn_packed_words", "tbn_status_string", "tbn_last_error",
    "tbn_device_error", "tbn_quantize_pack", "tbn_quantize_pack_group", "tbn_unpack",
    "tbn_conv2d_fwd", "tbn_conv2d_fwd_algo", "tbn_conv2d_select_algo", "tbn_linear_fwd",
    "tbn_linear_workspace_bytes", "tbn_linear_fwd_ws", "tbn_linear_fwd_noalloc",
    "tbn_maxpool2d_nhwc", "tbn_nchw_to_nhwc", "tbn_conv2d_bwd_data_workspace_bytes",
    "tbn_conv2d_bwd_data", "tbn_conv2d_bwd_filter_workspace_bytes", "tbn_conv2d_bwd_filter",
    "tbn_selftest_wait_timeout", "tbn_repack", "tbn_dense_conv2d_fwd",
    "tbn_avgpool2d_global_nhwc", "tbn_dense_linear_fwd", "tbn_space_to_depth_elems",
    "tbn_space_to_depth", "tbn_linear_prepare_f8", "tbn_linear_f8_workspace_bytes",
    "tbn_linear_fwd_f8", "tbn_linear_f8_prepared_words", "tbn_conv2d_fwd_quant",
]


class TBNError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str):
        self.status = status
        super().__init__("%s failed: status %d (%s): %s" % (
            where, status, _status_name(status), detail))


class QuantJob(ctypes.Structure):
    _fields_ = [("W", ctypes.c_void_p), ("K", ctypes.c_int64), ("n", ctypes.c_int64),
                ("codes", ctypes.c_void_p), ("alpha", ctypes.c_void_p)]


class Epilogue(ctypes.Structure):
    _fields_ = [("relu", ctypes.c_int), ("residual", ctypes.c_void_p), ("pool", ctypes.c_int)]


_lock = threading.Lock()
_lib = None


ABI_VERSION = 9  # must match TBN_ABI_VERSION in include/tbn.h


def lib_path() -> str:
    return _LIB_PATH


def lib():
    """The loaded libtbn.so (ctypes.CDLL).  Raises if it was not built."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError("libtbn.so not found at %s: build it with "
                               "`python -m paper_1701_00485_gb300.build`" % _LIB_PATH)
        L = ctypes.CDLL(_LIB_PATH)
        P, I64, I32, U32P = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_void_p
        sig = {
            "tbn_abi_version": ([], I32),
            "tbn_packed_words": ([I64], I64),
            "tbn_status_string": ([I32], ctypes.c_char_p),
            "tbn_last_error": ([], ctypes.c_char_p),
            "tbn_device_error": ([ctypes.POINTER(ctypes.c_uint32)], I32),
            "tbn_selftest_wait_timeout": ([ctypes.c_uint32, P], I32),
            "tbn_quantize_pack": ([P, I64, I64, U32P, P, P], I32),
            "tbn_quantize_pack_group": ([ctypes.POINTER(QuantJob), I32, P], I32),
            "tbn_unpack": ([U32P, P, I64, I64, P, I32, P], I32),
            "tbn_conv2d_fwd": ([P, I32, I32, I64, I64, I64, I64, U32P, P, I64, I64, I64,
                                I64, I64, I64, I64, P, I32, ctypes.POINTER(Epilogue), P], I32),
            "tbn_conv2d_fwd_algo": ([P, I32, I32, I64, I64, I64, I64, U32P, P, I64, I64, I64,
                                     I64, I64, I64, I64, P, I32, ctypes.POINTER(Epilogue), I32,
                                     P], I32),
            "tbn_conv2d_select_algo": ([I32, I32, I64, I64, I64, I64, I64, I64, I64, I64, I64,
                                        I64, I64], I32),
            "tbn_linear_fwd": ([P, I32, I64, I64, U32P, P, I64, P, I32,
                                ctypes.POINTER(Epilogue), P], I32),
            "tbn_linear_workspace_bytes": ([I32, I64, I64, I64], ctypes.c_size_t),
            "tbn_linear_fwd_ws": ([P, I32, I64, I64, U32P, P, I64, P, I32,
                                   ctypes.POINTER(Epilogue), P, ctypes.c_size_t, P], I32),
            "tbn_linear_fwd_noalloc": ([P, I32, I64, I64, U32P, P, I64, P, I32,
                                        ctypes.POINTER(Epilogue), P], I32),
            "tbn_maxpool2d_nhwc": ([P, I32] + [I64] * 10 + [P, P], I32),
            "tbn_repack": ([U32P, I64, I64, U32P, I32, P], I32),
            "tbn_dense_conv2d_fwd": ([P, I32, I32, I64, I64, I64, I64, P] + [I64] * 7 +
                                     [P, I32, I32, P], I32),
            "tbn_avgpool2d_global_nhwc": ([P, I32, I64, I64, I64, I64, P, I32, P], I32),
            "tbn_dense_linear_fwd": ([P, I64, I64, P, I64, P, I32, I32, P], I32),
            "tbn_conv2d_bwd_data_workspace_bytes": ([I64] * 11, ctypes.c_size_t),
            "tbn_conv2d_bwd_data": ([P, I64, I64, I64, I64, U32P, P] + [I64] * 7 +
                                    [P, I32, P, ctypes.c_size_t, P], I32),
            "tbn_conv2d_bwd_filter_workspace_bytes": ([I64] * 11, ctypes.c_size_t),
            "tbn_conv2d_bwd_filter": ([P, P] + [I64] * 11 + [P, P, ctypes.c_size_t, P], I32),
            "tbn_nchw_to_nhwc": ([P, I32, I64, I64, I64, I64, I64, P, P], I32),
            "tbn_space_to_depth_elems": ([I64] * 10, I64),
            "tbn_space_to_depth": ([P, I32, I32] + [I64] * 10 + [P, P], I32),
            "tbn_linear_prepare_f8": ([U32P, I64, I64, U32P, P], I32),
            "tbn_linear_f8_workspace_bytes": ([I64, I64, I64], ctypes.c_size_t),
            "tbn_linear_f8_prepared_words": ([I64, I64], I64),
            "tbn_conv2d_fwd_quant": ([P, I32, I32, I64, I64, I64, I64, P] + [I64] * 7 +
                                     [U32P, P, P, I32, ctypes.POINTER(Epilogue), P,
                                      ctypes.c_size_t, P], I32),
            "tbn_linear_fwd_f8": ([P, I32, I64, I64, U32P, P, I64, P, I32,
                                   ctypes.POINTER(Epilogue), P, ctypes.c_size_t, P], I32),
        }
        for name, (args, res) in sig.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = res
        if L.tbn_abi_version() != ABI_VERSION:
            raise RuntimeError("libtbn ABI version mismatch")
        _lib = L
        return L


def _status_name(s: int) -> str:
    try:
        return lib().tbn_status_string(int(s)).decode()
    except Exception:  # pragma: no cover - only while reporting another failure
        return "?"


def _check(status: int, where: str):
    if status != TBN_OK:
        detail = lib().tbn_last_error().decode(errors="replace")
        raise TBNError(status, where, detail)


def _dt(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return TBN_F32
    if t.dtype == torch.bfloat16:
        return TBN_BF16
    raise TypeError("tensor dtype must be float32 or bfloat16, got %s" % t.dtype)


def _torch_dt(code: int):
    return torch.float32 if code == TBN_F32 else torch.bfloat16


def _cuda(t: torch.Tensor, name: str) -> torch.Tensor:
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise ValueError("%s must be a CUDA tensor" % name)
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)
    return t


def _stream(stream) -> ctypes.c_void_p:
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _epi(relu: bool, residual, pool: int = 0) -> Epilogue | None:
    if not relu and residual is None and not pool:
        return None
    return Epilogue(1 if relu else 0, residual.data_ptr() if residual is not None else None,
                    int(pool))


def packed_words(n: int) -> int:
    """ceil(n / 16): uint32 words per filter of n two-bit codes."""
    return int(lib().tbn_packed_words(int(n)))


def conv_out_hw(H, W, R, S, stride=(1, 1), pad=(0, 0)):
    return (H + 2 * pad[0] - R) // stride[0] + 1, (W + 2 * pad[1] - S) // stride[1] + 1


def tbn_quantize_pack(W: torch.Tensor, codes: torch.Tensor | None = None,
                      alpha: torch.Tensor | None = None, stream=None):
    """Eq. 3 + Eq. 5 + packing for each row of W [K, n] (fp32, CUDA).

    Returns (codes int32 [K, ceil(n/16)] holding the uint32 words, alpha fp32 [K])."""
    _cuda(W, "W")
    if W.dtype != torch.float32 or W.dim() != 2:
        raise ValueError("W must be a 2-D float32 tensor [K, n]")
    K, n = W.shape
    if codes is None:
        codes = torch.empty((K, packed_words(n)), dtype=torch.int32, device=W.device)
    if alpha is None:
        alpha = torch.empty((K,), dtype=torch.float32, device=W.device)
    _cuda(codes, "codes"), _cuda(alpha, "alpha")
    _check(lib().tbn_quantize_pack(W.data_ptr(), K, n, codes.data_ptr(), alpha.data_ptr(),
                                   _stream(stream)), "tbn_quantize_pack")
    return codes, alpha


def tbn_quantize_pack_group(jobs, stream=None):
    """One launch for up to 16 layers; jobs = [(W [K,n], codes, alpha), ...]."""
    if not 1 <= len(jobs) <= TBN_MAX_QUANT_JOBS:
        raise ValueError("need 1..16 jobs")
    arr = (QuantJob * len(jobs))()
    for i, (W, codes, alpha) in enumerate(jobs):
        _cuda(W, "W"), _cuda(codes, "codes"), _cuda(alpha, "alpha")
        K, n = W.shape
        arr[i] = QuantJob(W.data_ptr(), K, n, codes.data_ptr(), alpha.data_ptr())
    _check(lib().tbn_quantize_pack_group(arr, len(jobs), _stream(stream)),
           "tbn_quantize_pack_group")


def tbn_unpack(codes: torch.Tensor, alpha: torch.Tensor | None, n: int,
               fmt: int = TBN_UNPACK_I8, stream=None) -> torch.Tensor:
    """codes [K, ceil(n/16)] -> int8 W~ or fp32/bf16 alpha*W~ [K, n]."""
    _cuda(codes, "codes")
    K = codes.shape[0]
    dt = {TBN_UNPACK_I8: torch.int8, TBN_UNPACK_F32: torch.float32,
          TBN_UNPACK_BF16: torch.bfloat16}[fmt]
    out = torch.empty((K, n), dtype=dt, device=codes.device)
    _check(lib().tbn_unpack(codes.data_ptr(), alpha.data_ptr() if alpha is not None else None,
                            K, n, out.data_ptr(), fmt, _stream(stream)), "tbn_unpack")
    return out


def tbn_conv2d_fwd(x: torch.Tensor, codes: torch.Tensor, alpha: torch.Tensor, K: int, R: int,
                   S: int, stride=(1, 1), pad=(0, 0), layout: int = TBN_NHWC,
                   out_dtype=None, relu: bool = False, residual: torch.Tensor | None = None,
                   algo: int = TBN_CONV_AUTO, out: torch.Tensor | None = None, stream=None,
                   pool: int = 0, in_chw=None):
    """Two-bit convolution, Eq. 1.  x is [N,C,H,W] (NCHW, NCHW_NHWC) or
    [N,H,W,C] (NHWC); y is NCHW for NCHW, else NHWC.
    pool=2 fuses a 2x2 / stride-2 max pool (after ReLU) into the epilogue.
    With layout TBN_S2D_NHWC, x is the output of tbn_space_to_depth for this
    convolution and in_chw = (C, H, W) gives the original input's size."""
    _cuda(x, "x"), _cuda(codes, "codes"), _cuda(alpha, "alpha")
    if layout == TBN_S2D_NHWC:
        if in_chw is None:
            raise ValueError("layout TBN_S2D_NHWC needs in_chw = (C, H, W)")
        N = x.shape[0]
        C, H, W = in_chw
        if tuple(x.shape) != space_to_depth_shape(N, C, H, W, R, S, stride, pad):
            raise ValueError("x is not the space-to-depth form of this convolution's input")
    elif layout == TBN_NHWC:
        N, H, W, C = x.shape
    else:
        N, C, H, W = x.shape
    P, Q = conv_out_hw(H, W, R, S, stride, pad)
    if pool:
        P, Q = P // 2, Q // 2
    ydt = _dt(x) if out_dtype is None else (TBN_F32 if out_dtype == torch.float32 else TBN_BF16)
    shape = (N, K, P, Q) if layout == TBN_NCHW else (N, P, Q, K)
    if out is None:
        out = torch.empty(shape, dtype=_torch_dt(ydt), device=x.device)
    elif tuple(out.shape) != shape or _dt(out) != ydt:
        raise ValueError("out has the wrong shape or dtype")
    if residual is not None:
        _cuda(residual, "residual")
        if tuple(residual.shape) != shape or _dt(residual) != ydt:
            raise ValueError("residual must match y's shape and dtype")
    e = _epi(relu, residual, pool)
    _check(lib().tbn_conv2d_fwd_algo(
        x.data_ptr(), _dt(x), layout, N, C, H, W, codes.data_ptr(), alpha.data_ptr(), K, R, S,
        stride[0], stride[1], pad[0], pad[1], out.data_ptr(), ydt,
        ctypes.byref(e) if e is not None else None, algo, _stream(stream)), "tbn_conv2d_fwd")
    return out


def tbn_conv2d_fwd_quant(x: torch.Tensor, W: torch.Tensor, K: int, R: int, S: int,
                         stride=(1, 1), pad=(0, 0), out_dtype=None, relu: bool = False,
                         residual: torch.Tensor | None = None, pool: int = 0,
                         codes: torch.Tensor | None = None, alpha: torch.Tensor | None = None,
                         workspace: torch.Tensor | None = None, out: torch.Tensor | None = None,
                         stream=None):
    """Quantization (Eq. 3, Eq. 5) of the fp32 filters W [K, R*S*C] ((r, s, c)
    order) and the two-bit convolution of NHWC bf16 x [N, H, W, C] with them,
    in one launch.  Returns (y, codes, alpha); codes and alpha equal what
    tbn_quantize_pack writes for W."""
    _cuda(x, "x"), _cuda(W, "W")
    N, H, Wd, C = x.shape
    n = W.shape[1]
    if W.dtype != torch.float32 or tuple(W.shape) != (K, R * S * C) or not W.is_contiguous():
        raise ValueError("W must be a contiguous float32 tensor [K, R*S*C]")
    if codes is None:
        codes = torch.empty((K, packed_words(n)), dtype=torch.int32, device=x.device)
    if alpha is None:
        alpha = torch.empty((K,), dtype=torch.float32, device=x.device)
    if workspace is None:
        workspace = torch.empty((64,), dtype=torch.uint8, device=x.device)
    P, Q = conv_out_hw(H, Wd, R, S, stride, pad)
    if pool:
        P, Q = P // 2, Q // 2
    ydt = _dt(x) if out_dtype is None else (TBN_F32 if out_dtype == torch.float32 else TBN_BF16)
    if out is None:
        out = torch.empty((N, P, Q, K), dtype=_torch_dt(ydt), device=x.device)
    e = _epi(relu, residual, pool)
    _check(lib().tbn_conv2d_fwd_quant(
        x.data_ptr(), _dt(x), TBN_NHWC, N, C, H, Wd, W.data_ptr(), K, R, S, stride[0], stride[1],
        pad[0], pad[1], codes.data_ptr(), alpha.data_ptr(), out.data_ptr(), ydt,
        ctypes.byref(e) if e is not None else None, workspace.data_ptr(),
        workspace.numel() * workspace.element_size(), _stream(stream)), "tbn_conv2d_fwd_quant")
    return out, codes, alpha


def space_to_depth_shape(N: int, C: int, H: int, W: int, R: int, S: int, stride=(4, 4),
                         pad=(0, 0)):
    """Shape [N, Hs, Ws, 64] of tbn_space_to_depth's output for this
    convolution (Hs = P + ceil(R / s) - 1, Ws = Q + ceil(S / s) - 1)."""
    n = lib().tbn_space_to_depth_elems(N, C, H, W, R, S, stride[0], stride[1], pad[0], pad[1])
    if n < 0:
        raise ValueError("no space-to-depth form for this convolution (needs equal strides "
                         ">= 2 and stride^2 * C <= 64)")
    P, Q = conv_out_hw(H, W, R, S, stride, pad)
    s = stride[0]
    return (N, P + (R + s - 1) // s - 1, Q + (S + s - 1) // s - 1, 64)


def tbn_space_to_depth(x: torch.Tensor, R: int, S: int, stride=(4, 4), pad=(0, 0),
                       layout: int = TBN_NCHW, out: torch.Tensor | None = None,
                       stream=None) -> torch.Tensor:
    """Space-to-depth form [N, Hs, Ws, 64] bf16 of the bf16 input x (NCHW or
    NHWC) of an R x S convolution with this stride and padding, for
    tbn_conv2d_fwd(..., layout=TBN_S2D_NHWC, in_chw=(C, H, W))."""
    _cuda(x, "x")
    if layout == TBN_NHWC:
        N, H, W, C = x.shape
    else:
        N, C, H, W = x.shape
    shape = space_to_depth_shape(N, C, H, W, R, S, stride, pad)
    if out is None:
        out = torch.empty(shape, dtype=torch.bfloat16, device=x.device)
    elif tuple(out.shape) != shape or out.dtype != torch.bfloat16:
        raise ValueError("out has the wrong shape or dtype")
    _check(lib().tbn_space_to_depth(x.data_ptr(), _dt(x), layout, N, C, H, W, R, S, stride[0],
                                    stride[1], pad[0], pad[1], out.data_ptr(), _stream(stream)),
           "tbn_space_to_depth")
    return out


def _bwd_shape(N, C, H, W, K, R, S, stride, pad):
    return (N, C, H, W, K, R, S, stride[0], stride[1], pad[0], pad[1])


def tbn_conv2d_bwd_data(dy: torch.Tensor, codes: torch.Tensor, alpha: torch.Tensor, C: int,
                        in_hw, R: int, S: int, stride=(1, 1), pad=(0, 0), out_dtype=None,
                        workspace: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Algorithm 1 TwoBitBackward, input gradient: dy [N,P,Q,K] bf16 (NHWC) ->
    dx [N,H,W,C] through the convolution with alpha*W~ (codes in (r,s,c) order)."""
    _cuda(dy, "dy"), _cuda(codes, "codes"), _cuda(alpha, "alpha")
    N, P, Q, K = dy.shape
    H, W = in_hw
    shape = _bwd_shape(N, C, H, W, K, R, S, stride, pad)
    n = int(lib().tbn_conv2d_bwd_data_workspace_bytes(*shape))
    if workspace is None:
        workspace = torch.empty(max(n, 256), dtype=torch.uint8, device=dy.device)
    ydt = TBN_BF16 if out_dtype in (None, torch.bfloat16) else TBN_F32
    dx = torch.empty((N, H, W, C), dtype=_torch_dt(ydt), device=dy.device)
    _check(lib().tbn_conv2d_bwd_data(dy.data_ptr(), N, C, H, W, codes.data_ptr(),
                                     alpha.data_ptr(), K, R, S, stride[0], stride[1], pad[0],
                                     pad[1], dx.data_ptr(), ydt, workspace.data_ptr(),
                                     workspace.numel() * workspace.element_size(),
                                     _stream(stream)), "tbn_conv2d_bwd_data")
    return dx


def tbn_conv2d_bwd_filter(x: torch.Tensor, dy: torch.Tensor, R: int, S: int, stride=(1, 1),
                          pad=(0, 0), workspace: torch.Tensor | None = None,
                          stream=None) -> torch.Tensor:
    """Algorithm 1 TwoBitBackward, gradient w.r.t. alpha*W~: x [N,H,W,C] and
    dy [N,P,Q,K] bf16 (NHWC) -> dW^ [K, R*S*C] fp32 in (r,s,c) order."""
    _cuda(x, "x"), _cuda(dy, "dy")
    N, H, W, C = x.shape
    K = dy.shape[3]
    shape = _bwd_shape(N, C, H, W, K, R, S, stride, pad)
    n = int(lib().tbn_conv2d_bwd_filter_workspace_bytes(*shape))
    if workspace is None:
        workspace = torch.empty(max(n, 256), dtype=torch.uint8, device=x.device)
    dw = torch.empty((K, R * S * C), dtype=torch.float32, device=x.device)
    _check(lib().tbn_conv2d_bwd_filter(x.data_ptr(), dy.data_ptr(), *shape, dw.data_ptr(),
                                       workspace.data_ptr(),
                                       workspace.numel() * workspace.element_size(),
                                       _stream(stream)), "tbn_conv2d_bwd_filter")
    return dw


def tbn_conv2d_select_algo(x_dtype, layout, N, C, H, W, K, R, S, stride=(1, 1), pad=(0, 0)):
    xdt = TBN_F32 if x_dtype == torch.float32 else TBN_BF16
    return int(lib().tbn_conv2d_select_algo(xdt, layout, N, C, H, W, K, R, S, stride[0],
                                            stride[1], pad[0], pad[1]))


def tbn_linear_fwd(x: torch.Tensor, codes: torch.Tensor, alpha: torch.Tensor, K_out: int,
                   out_dtype=None, relu: bool = False, residual: torch.Tensor | None = None,
                   out: torch.Tensor | None = None, stream=None):
    """Fully-connected layer (Section 3): x [B, K_in] -> y [B, K_out]."""
    _cuda(x, "x"), _cuda(codes, "codes"), _cuda(alpha, "alpha")
    B, K_in = x.shape
    ydt = _dt(x) if out_dtype is None else (TBN_F32 if out_dtype == torch.float32 else TBN_BF16)
    if out is None:
        out = torch.empty((B, K_out), dtype=_torch_dt(ydt), device=x.device)
    e = _epi(relu, residual)
    _check(lib().tbn_linear_fwd(x.data_ptr(), _dt(x), B, K_in, codes.data_ptr(), alpha.data_ptr(),
                                K_out, out.data_ptr(), ydt,
                                ctypes.byref(e) if e is not None else None, _stream(stream)),
           "tbn_linear_fwd")
    return out


def tbn_linear_workspace_bytes(B: int, K_in: int, K_out: int, x_dtype=torch.bfloat16) -> int:
    """Scratch bytes tbn_linear_fwd_ws needs for the table-lookup GEMV (0: none)."""
    xdt = TBN_F32 if x_dtype == torch.float32 else TBN_BF16
    return int(lib().tbn_linear_workspace_bytes(xdt, B, K_in, K_out))


def tbn_linear_fwd_ws(x: torch.Tensor, codes: torch.Tensor, alpha: torch.Tensor, K_out: int,
                      workspace: torch.Tensor | None, out_dtype=None, relu: bool = False,
                      residual: torch.Tensor | None = None, out: torch.Tensor | None = None,
                      stream=None):
    """tbn_linear_fwd with caller-owned device scratch: a CUDA tensor of at least
    tbn_linear_workspace_bytes(...) bytes (its contents on entry do not
    matter), or None."""
    _cuda(x, "x"), _cuda(codes, "codes"), _cuda(alpha, "alpha")
    B, K_in = x.shape
    ydt = _dt(x) if out_dtype is None else (TBN_F32 if out_dtype == torch.float32 else TBN_BF16)
    if out is None:
        out = torch.empty((B, K_out), dtype=_torch_dt(ydt), device=x.device)
    ws_ptr, ws_bytes = None, 0
    if workspace is not None:
        _cuda(workspace, "workspace")
        ws_ptr, ws_bytes = workspace.data_ptr(), workspace.numel() * workspace.element_size()
    e = _epi(relu, residual)
    _check(lib().tbn_linear_fwd_ws(x.data_ptr(), _dt(x), B, K_in, codes.data_ptr(),
                                   alpha.data_ptr(), K_out, out.data_ptr(), ydt,
                                   ctypes.byref(e) if e is not None else None, ws_ptr, ws_bytes,
                                   _stream(stream)),
           "tbn_linear_fwd_ws")
    return out


def tbn_linear_f8_prepared_words(K_out: int, K_in: int) -> int:
    return int(lib().tbn_linear_f8_prepared_words(K_out, K_in))


def tbn_linear_prepare_f8(codes: torch.Tensor, K_in: int, out: torch.Tensor | None = None,
                          stream=None) -> torch.Tensor:
    """The codes [K_out, packed_words(K_in)] rewritten in the fp8 GEMV's
    prepared layout (once per weight matrix): a flat int32 tensor of
    tbn_linear_f8_prepared_words(K_out, K_in) words."""
    _cuda(codes, "codes")
    K_out = codes.shape[0]
    n = tbn_linear_f8_prepared_words(K_out, K_in)
    if n < 0:
        raise ValueError("no fp8 GEMV layout for K_in = %d (a multiple of 512 is needed)" % K_in)
    if out is None:
        out = torch.empty((n,), dtype=torch.int32, device=codes.device)
    elif out.numel() != n:
        raise ValueError("out must hold tbn_linear_f8_prepared_words(K_out, K_in) words")
    _check(lib().tbn_linear_prepare_f8(codes.data_ptr(), K_out, K_in, out.data_ptr(),
                                       _stream(stream)), "tbn_linear_prepare_f8")
    return out


def tbn_linear_f8_workspace_bytes(B: int, K_in: int, K_out: int) -> int:
    return int(lib().tbn_linear_f8_workspace_bytes(B, K_in, K_out))


def tbn_linear_fwd_f8(x: torch.Tensor, prepared: torch.Tensor, alpha: torch.Tensor, K_out: int,
                      workspace: torch.Tensor, out_dtype=None, relu: bool = False,
                      residual: torch.Tensor | None = None, out: torch.Tensor | None = None,
                      stream=None):
    """Batch-1 fp8 tensor-core linear layer on codes from tbn_linear_prepare_f8
    (x bf16 [1, K_in]; workspace of at least tbn_linear_f8_workspace_bytes)."""
    _cuda(x, "x"), _cuda(prepared, "prepared"), _cuda(alpha, "alpha"), _cuda(workspace, "workspace")
    B, K_in = x.shape
    ydt = _dt(x) if out_dtype is None else (TBN_F32 if out_dtype == torch.float32 else TBN_BF16)
    if out is None:
        out = torch.empty((B, K_out), dtype=_torch_dt(ydt), device=x.device)
    e = _epi(relu, residual)
    _check(lib().tbn_linear_fwd_f8(x.data_ptr(), _dt(x), B, K_in, prepared.data_ptr(),
                                   alpha.data_ptr(), K_out, out.data_ptr(), ydt,
                                   ctypes.byref(e) if e is not None else None,
                                   workspace.data_ptr(),
                                   workspace.numel() * workspace.element_size(), _stream(stream)),
           "tbn_linear_fwd_f8")
    return out


def tbn_linear_fwd_noalloc(x: torch.Tensor, codes: torch.Tensor, alpha: torch.Tensor,
                           K_out: int, out_dtype=None, relu: bool = False,
                           residual: torch.Tensor | None = None, out: torch.Tensor | None = None,
                           stream=None):
    """The batch-1 fp32 table GEMV with its scratch inside the library (the C
    call allocates nothing; `out` is allocated here only when not given)."""
    _cuda(x, "x"), _cuda(codes, "codes"), _cuda(alpha, "alpha")
    B, K_in = x.shape
    ydt = _dt(x) if out_dtype is None else (TBN_F32 if out_dtype == torch.float32 else TBN_BF16)
    if out is None:
        out = torch.empty((B, K_out), dtype=_torch_dt(ydt), device=x.device)
    e = _epi(relu, residual)
    _check(lib().tbn_linear_fwd_noalloc(x.data_ptr(), _dt(x), B, K_in, codes.data_ptr(),
                                        alpha.data_ptr(), K_out, out.data_ptr(), ydt,
                                        ctypes.byref(e) if e is not None else None,
                                        _stream(stream)),
           "tbn_linear_fwd_noalloc")
    return out


def tbn_maxpool2d_nhwc(x, k=(2, 2), stride=(2, 2), out=None, stream=None, pad=(0, 0)):
    """Max pooling over NHWC; taps in the padding are skipped (-inf padding)."""
    _cuda(x, "x")
    N, H, W, C = x.shape
    Ho, Wo = conv_out_hw(H, W, k[0], k[1], stride, pad)
    if out is None:
        out = torch.empty((N, Ho, Wo, C), dtype=x.dtype, device=x.device)
    _check(lib().tbn_maxpool2d_nhwc(x.data_ptr(), _dt(x), N, H, W, C, k[0], k[1], stride[0],
                                    stride[1], pad[0], pad[1], out.data_ptr(), _stream(stream)),
           "tbn_maxpool2d_nhwc")
    return out


def tbn_repack(codes: torch.Tensor, n: int, direction: int, out=None, stream=None):
    """Codes [K, ceil(n/16)] between the byte-planar layout and the canonical
    interchange layout (TBN_REPACK_CANONICAL_TO_PLANAR / _PLANAR_TO_CANONICAL)."""
    _cuda(codes, "codes")
    K = codes.shape[0]
    if out is None:
        out = torch.empty_like(codes)
    _cuda(out, "out")
    _check(lib().tbn_repack(codes.data_ptr(), K, n, out.data_ptr(), direction, _stream(stream)),
           "tbn_repack")
    return out


def tbn_dense_conv2d_fwd(x: torch.Tensor, w: torch.Tensor, stride=(1, 1), pad=(0, 0),
                         layout: int = TBN_NCHW_NHWC, out_dtype=None, relu: bool = False,
                         out: torch.Tensor | None = None, stream=None):
    """Full-precision convolution with fp32 weights w [K, C, R, S] (the first
    layer a two-bit network keeps in fp32).  x is [N,C,H,W] for NCHW and
    NCHW_NHWC, [N,H,W,C] for NHWC; y is NCHW for NCHW, else NHWC."""
    _cuda(x, "x"), _cuda(w, "w")
    if w.dtype != torch.float32 or w.dim() != 4:
        raise ValueError("w must be a float32 [K, C, R, S] tensor")
    K, C, R, S = w.shape
    if layout == TBN_NHWC:
        N, H, W, C2 = x.shape
    else:
        N, C2, H, W = x.shape
    if C2 != C:
        raise ValueError("x has %d channels, w expects %d" % (C2, C))
    P, Q = conv_out_hw(H, W, R, S, stride, pad)
    ydt = _dt(x) if out_dtype is None else (TBN_F32 if out_dtype == torch.float32 else TBN_BF16)
    shape = (N, K, P, Q) if layout == TBN_NCHW else (N, P, Q, K)
    if out is None:
        out = torch.empty(shape, dtype=_torch_dt(ydt), device=x.device)
    elif tuple(out.shape) != shape or _dt(out) != ydt:
        raise ValueError("out has the wrong shape or dtype")
    _check(lib().tbn_dense_conv2d_fwd(x.data_ptr(), _dt(x), layout, N, C, H, W, w.data_ptr(), K, R,
                                      S, stride[0], stride[1], pad[0], pad[1], out.data_ptr(), ydt,
                                      1 if relu else 0, _stream(stream)), "tbn_dense_conv2d_fwd")
    return out


def tbn_avgpool2d_global_nhwc(x: torch.Tensor, out_dtype=torch.float32, out=None, stream=None):
    """Mean over H and W of x [N, H, W, C] -> [N, C]."""
    _cuda(x, "x")
    N, H, W, C = x.shape
    ydt = TBN_F32 if out_dtype == torch.float32 else TBN_BF16
    if out is None:
        out = torch.empty((N, C), dtype=_torch_dt(ydt), device=x.device)
    _check(lib().tbn_avgpool2d_global_nhwc(x.data_ptr(), _dt(x), N, H, W, C, out.data_ptr(), ydt,
                                           _stream(stream)), "tbn_avgpool2d_global_nhwc")
    return out


def tbn_dense_linear_fwd(x: torch.Tensor, w: torch.Tensor, out_dtype=torch.float32,
                         relu: bool = False, out=None, stream=None):
    """Full-precision fully-connected layer: x [B, K_in] fp32, w [K_out, K_in] fp32."""
    _cuda(x, "x"), _cuda(w, "w")
    if x.dtype != torch.float32 or w.dtype != torch.float32:
        raise ValueError("x and w must be float32")
    B, K_in = x.shape
    K_out = w.shape[0]
    if w.shape[1] != K_in:
        raise ValueError("w must be [K_out, K_in]")
    ydt = TBN_F32 if out_dtype == torch.float32 else TBN_BF16
    if out is None:
        out = torch.empty((B, K_out), dtype=_torch_dt(ydt), device=x.device)
    _check(lib().tbn_dense_linear_fwd(x.data_ptr(), B, K_in, w.data_ptr(), K_out, out.data_ptr(),
                                      ydt, 1 if relu else 0, _stream(stream)),
           "tbn_dense_linear_fwd")
    return out


def tbn_nchw_to_nhwc(x: torch.Tensor, C_pad: int | None = None, out=None, stream=None):
    _cuda(x, "x")
    N, C, H, W = x.shape
    C_pad = C if C_pad is None else C_pad
    if out is None:
        out = torch.empty((N, H, W, C_pad), dtype=x.dtype, device=x.device)
    _check(lib().tbn_nchw_to_nhwc(x.data_ptr(), _dt(x), N, C, H, W, C_pad, out.data_ptr(),
                                  _stream(stream)), "tbn_nchw_to_nhwc")
    return out


def tbn_device_error() -> int:
    """Read and clear the current device's error word (synchronizes)."""
    v = ctypes.c_uint32(0)
    _check(lib().tbn_device_error(ctypes.byref(v)), "tbn_device_error")
    return int(v.value)


def tbn_selftest_wait_timeout(limit_us: int, stream=None) -> None:
    """Launch the bounded-wait self-check: a wait that nothing ends runs out
    after limit_us and sets TBN_DEVERR_TIMEOUT in the device error word."""
    _check(lib().tbn_selftest_wait_timeout(limit_us, _stream(stream)),
           "tbn_selftest_wait_timeout")
