"""CPU oracle for Two-Bit Networks (arXiv:1701.00485) -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product (``paper_1701_00485_gb300``
and its CUDA library) never does, and the two share no code.

The arithmetic lives in ``tbn_oracle.c`` (plain C, IEEE double, loops in the
order the paper states them).  This module compiles it with gcc on first use
and wraps each function for numpy arrays.  Functions and the passage each one
follows:

  discretize      Eq. 3 (Section 2)
  alpha           Eq. 5 (Section 2)
  quantize        Algorithm 1, quantization loop (Eq. 3 + Eq. 5 per filter)
  pack / unpack   two-bit storage; the paper fixes only "two bits per weight",
                  the field layout is documented in tbn_oracle.h
  pack_canonical / unpack_canonical   the canonical (sequential) two-bit
                  layout, the interchange format (same fields, code i at bits
                  2i, 2i+1 of its word)
  quant_error     Eq. 2 objective, evaluated directly
  conv2d_nchw     Eq. 1, seven nested loops, zero padding, cross-correlation
  conv2d_sites    Eq. 1 at selected output sites
  conv2d_bwd_data, conv2d_bwd_filter   Algorithm 1 TwoBitBackward through
                  Eq. 1: the input gradient (the adjoint of the convolution
                  with alpha*W~) and the gradient w.r.t. alpha*W~
  linear          Section 3: fully-connected layer treated as a convolution
  epilogue, maxpool2d_nchw   network glue of the benchmark workloads
  dense_conv2d_nchw, avgpool_global_nchw, dense_linear   the full-precision
                  first convolution, global average pool and last
                  fully-connected layer of the ResNet-18 workload (not part
                  of the paper's method)
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "tbn_oracle.c")
_HDR = os.path.join(_HERE, "tbn_oracle.h")
LIB_PATH = os.path.join(_HERE, "liborcl_tbn.so")

_lock = threading.Lock()
_default = None


def _compile(src: str, out: str) -> None:
    tmp = out + ".tmp.%d" % os.getpid()
    cmd = ["gcc", "-std=c11", "-O2", "-fno-fast-math", "-ffp-contract=off",
           "-fopenmp", "-fPIC", "-shared", "-I", _HERE, "-o", tmp, src, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)


def build(force: bool = False) -> str:
    """Compile the oracle shared library with gcc (OpenMP, no fast-math)."""
    stale = (not os.path.exists(LIB_PATH)) or any(
        os.path.getmtime(p) > os.path.getmtime(LIB_PATH) for p in (_SRC, _HDR))
    if force or stale:
        _compile(_SRC, LIB_PATH)
    return LIB_PATH


def build_variant(c_source_text: str, out_path: str) -> str:
    """Compile a modified copy of tbn_oracle.c (used by the tests that plant
    a mistake in the oracle to show that the pins catch it)."""
    src = out_path + ".c"
    with open(src, "w") as f:
        f.write(c_source_text)
    _compile(src, out_path)
    return out_path


def source_text() -> str:
    with open(_SRC) as f:
        return f.read()


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _f32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float32))


def out_hw(H, W, R, S, stride, pad):
    sh, sw = stride
    ph, pw = pad
    return (H + 2 * ph - R) // sh + 1, (W + 2 * pw - S) // sw + 1


class Oracle:
    """numpy wrappers around one build of the C oracle."""

    def __init__(self, lib_path: str):
        lib = ctypes.CDLL(lib_path)
        P = ctypes.c_void_p
        I = ctypes.c_int64
        sig = {
            "orc_discretize_one": ([ctypes.c_double], ctypes.c_int),
            "orc_discretize": ([P, I, P], None),
            "orc_alpha": ([P, I], ctypes.c_double),
            "orc_quantize": ([P, I, I, P, P], None),
            "orc_words_per_filter": ([I], I),
            "orc_pack": ([P, I, I, P], ctypes.c_int),
            "orc_unpack": ([P, I, I, P], ctypes.c_int),
            "orc_quant_error": ([P, P, I, ctypes.c_double], ctypes.c_double),
            "orc_conv2d_nchw": ([P, I, I, I, I, P, P, I, I, I, I, I, I, I, P, P], None),
            "orc_conv2d_nchw_sites": ([P, I, I, I, I, P, P, I, I, I, I, I, I, I, P, I, P, P],
                                      None),
            "orc_linear": ([P, I, I, P, P, I, P, P], None),
            "orc_conv2d_bwd_data_nchw": ([P, I, I, I, I, P, P, I, I, I, I, I, I, I, I, I, P, P],
                                         None),
            "orc_conv2d_bwd_filter_nchw": ([P, I, I, I, I, P, I, I, I, I, I, I, I, I, I, P, P],
                                           None),
            "orc_epilogue": ([P, P, I, ctypes.c_int], None),
            "orc_maxpool2d_nchw": ([P, I, I, I, I, I, I, I, I, I, I, P], None),
            "orc_pack_canonical": ([P, I, I, P], ctypes.c_int),
            "orc_unpack_canonical": ([P, I, I, P], ctypes.c_int),
            "orc_dense_conv2d_nchw": ([P, I, I, I, I, P, I, I, I, I, I, I, I, P, P], None),
            "orc_avgpool_global_nchw": ([P, I, I, I, I, P], None),
            "orc_dense_linear": ([P, I, I, P, I, P, P], None),
            "orc_num_threads": ([], ctypes.c_int),
            "orc_set_num_threads": ([ctypes.c_int], None),
        }
        for name, (args, res) in sig.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = res
        self.lib = lib

    def num_threads(self) -> int:
        return int(self.lib.orc_num_threads())

    def set_num_threads(self, n: int) -> None:
        """Threads of the parallel loops (timing the oracle on one core)."""
        self.lib.orc_set_num_threads(int(n))

    def discretize_one(self, w: float) -> int:
        """Eq. 3 for a single weight (evaluated on the value widened to double)."""
        return int(self.lib.orc_discretize_one(float(w)))

    def discretize(self, W) -> np.ndarray:
        """Eq. 3 elementwise; returns int8 codes with W's shape."""
        W = _f32(W)
        out = np.empty(W.shape, dtype=np.int8)
        self.lib.orc_discretize(_ptr(W), W.size, _ptr(out))
        return out

    def alpha(self, W) -> float:
        """Eq. 5 for one filter (all of W's elements)."""
        W = _f32(W)
        if W.size == 0:
            raise ValueError("Eq. 5 needs n >= 1")
        return float(self.lib.orc_alpha(_ptr(W), W.size))

    def quantize(self, W2d):
        """Quantization loop of Algorithm 1 over the rows of a [K, n] matrix.

        Returns (codes int8 [K, n], alpha float64 [K])."""
        W = _f32(W2d)
        if W.ndim != 2 or W.shape[1] == 0:
            raise ValueError("expected a [K, n] matrix with n >= 1")
        K, n = W.shape
        wt = np.empty((K, n), dtype=np.int8)
        al = np.empty((K,), dtype=np.float64)
        self.lib.orc_quantize(_ptr(W), K, n, _ptr(wt), _ptr(al))
        return wt, al

    def words_per_filter(self, n: int) -> int:
        return int(self.lib.orc_words_per_filter(int(n)))

    def pack(self, wt2d) -> np.ndarray:
        """Pack int8 codes [K, n] into uint32 words [K, ceil(n/16)]."""
        wt = np.ascontiguousarray(np.asarray(wt2d, dtype=np.int8))
        K, n = wt.shape
        out = np.empty((K, self.words_per_filter(n)), dtype=np.uint32)
        if self.lib.orc_pack(_ptr(wt), K, n, _ptr(out)) != 0:
            raise ValueError("codes must be in {-2,-1,1,2}")
        return out

    def unpack(self, words2d, n: int) -> np.ndarray:
        """Inverse of pack; raises if a padding field is non-zero."""
        w = np.ascontiguousarray(np.asarray(words2d, dtype=np.uint32))
        K = w.shape[0]
        if w.shape[1] != self.words_per_filter(n):
            raise ValueError("word count does not match n")
        out = np.empty((K, n), dtype=np.int8)
        if self.lib.orc_unpack(_ptr(w), K, n, _ptr(out)) != 0:
            raise ValueError("non-zero padding field")
        return out

    def quant_error(self, W, wt, a: float) -> float:
        """Eq. 2 objective ||W - a W~||^2 evaluated directly."""
        W = _f32(W).ravel()
        wt = np.ascontiguousarray(np.asarray(wt, dtype=np.int8)).ravel()
        return float(self.lib.orc_quant_error(_ptr(W), _ptr(wt), W.size, float(a)))

    def conv2d_nchw(self, x, wt, al, stride=(1, 1), pad=(0, 0)):
        """Eq. 1 with the dequantized filter alpha*W~ (seven loops, NCHW).

        x float32 [N, C, H, W]; wt int8 [K, C, R, S]; al float64 [K].
        Returns (y, bound) float64 [N, K, P, Q]."""
        x = _f32(x)
        wt = np.ascontiguousarray(np.asarray(wt, dtype=np.int8))
        al = np.ascontiguousarray(np.asarray(al, dtype=np.float64))
        N, C, H, W = x.shape
        K, C2, R, S = wt.shape
        assert C2 == C and al.shape == (K,)
        P, Q = out_hw(H, W, R, S, stride, pad)
        y = np.empty((N, K, P, Q), dtype=np.float64)
        bound = np.empty_like(y)
        self.lib.orc_conv2d_nchw(_ptr(x), N, C, H, W, _ptr(wt), _ptr(al), K, R, S,
                                 stride[0], stride[1], pad[0], pad[1], _ptr(y), _ptr(bound))
        return y, bound

    def conv2d_bwd_data(self, dy, wt, al, in_hw, stride=(1, 1), pad=(0, 0)):
        """Algorithm 1 TwoBitBackward: dx through Eq. 1 with alpha*W~ (NCHW).

        dy float32 [N, K, P, Q]; wt int8 [K, C, R, S]; al float64 [K];
        in_hw = (H, W) of x.  Returns (dx, bound) float64 [N, C, H, W]."""
        dy = _f32(dy)
        wt = np.ascontiguousarray(np.asarray(wt, dtype=np.int8))
        al = np.ascontiguousarray(np.asarray(al, dtype=np.float64))
        N, K, P, Q = dy.shape
        K2, C, R, S = wt.shape
        H, W = in_hw
        assert K2 == K and al.shape == (K,) and out_hw(H, W, R, S, stride, pad) == (P, Q)
        dx = np.empty((N, C, H, W), dtype=np.float64)
        bound = np.empty_like(dx)
        self.lib.orc_conv2d_bwd_data_nchw(_ptr(dy), N, K, P, Q, _ptr(wt), _ptr(al), C, H, W, R,
                                          S, stride[0], stride[1], pad[0], pad[1], _ptr(dx),
                                          _ptr(bound))
        return dx, bound

    def conv2d_bwd_filter(self, x, dy, RS, stride=(1, 1), pad=(0, 0)):
        """Algorithm 1 TwoBitBackward: gradient w.r.t. the approximate filters
        W^ = alpha*W~ of Eq. 1 (NCHW).  x float32 [N, C, H, W]; dy float32
        [N, K, P, Q]; RS = (R, S).  Returns (dw, bound) float64 [K, C, R, S]."""
        x, dy = _f32(x), _f32(dy)
        N, C, H, W = x.shape
        N2, K, P, Q = dy.shape
        R, S = RS
        assert N2 == N and out_hw(H, W, R, S, stride, pad) == (P, Q)
        dw = np.empty((K, C, R, S), dtype=np.float64)
        bound = np.empty_like(dw)
        self.lib.orc_conv2d_bwd_filter_nchw(_ptr(x), N, C, H, W, _ptr(dy), K, P, Q, R, S,
                                            stride[0], stride[1], pad[0], pad[1], _ptr(dw),
                                            _ptr(bound))
        return dw, bound

    def conv2d_sites(self, x, wt, al, sites, stride=(1, 1), pad=(0, 0)):
        """Eq. 1 at output sites [(b, k, p, q), ...]; returns (y, bound) [npts]."""
        x = _f32(x)
        wt = np.ascontiguousarray(np.asarray(wt, dtype=np.int8))
        al = np.ascontiguousarray(np.asarray(al, dtype=np.float64))
        sites = np.ascontiguousarray(np.asarray(sites, dtype=np.int64).reshape(-1, 4))
        N, C, H, W = x.shape
        K, C2, R, S = wt.shape
        assert C2 == C
        n = sites.shape[0]
        y = np.empty((n,), dtype=np.float64)
        bound = np.empty_like(y)
        self.lib.orc_conv2d_nchw_sites(_ptr(x), N, C, H, W, _ptr(wt), _ptr(al), K, R, S,
                                       stride[0], stride[1], pad[0], pad[1], _ptr(sites), n,
                                       _ptr(y), _ptr(bound))
        return y, bound

    def linear(self, x, wt, al):
        """Fully-connected layer (Section 3); x [B, Kin], wt [Kout, Kin]."""
        x = _f32(x)
        wt = np.ascontiguousarray(np.asarray(wt, dtype=np.int8))
        al = np.ascontiguousarray(np.asarray(al, dtype=np.float64))
        B, Kin = x.shape
        Kout = wt.shape[0]
        assert wt.shape[1] == Kin
        y = np.empty((B, Kout), dtype=np.float64)
        bound = np.empty_like(y)
        self.lib.orc_linear(_ptr(x), B, Kin, _ptr(wt), _ptr(al), Kout, _ptr(y), _ptr(bound))
        return y, bound

    def epilogue(self, y, residual=None, relu=False):
        """y (+ residual), then ReLU if requested; returns a new float64 array."""
        out = np.array(y, dtype=np.float64, copy=True, order="C")
        res = None
        if residual is not None:
            res = np.ascontiguousarray(np.asarray(residual, dtype=np.float64))
            assert res.shape == out.shape
        self.lib.orc_epilogue(_ptr(out), _ptr(res) if res is not None else None,
                              out.size, int(bool(relu)))
        return out

    def maxpool2d_nchw(self, x, k=(2, 2), stride=(2, 2), pad=(0, 0)):
        """Max pooling, NCHW; taps in the padding are skipped (-inf padding)."""
        x = np.ascontiguousarray(np.asarray(x, dtype=np.float64))
        N, C, H, W = x.shape
        Ho, Wo = out_hw(H, W, k[0], k[1], stride, pad)
        y = np.empty((N, C, Ho, Wo), dtype=np.float64)
        self.lib.orc_maxpool2d_nchw(_ptr(x), N, C, H, W, k[0], k[1], stride[0], stride[1],
                                    pad[0], pad[1], _ptr(y))
        return y

    def pack_canonical(self, wt2d) -> np.ndarray:
        """Pack int8 codes [K, n] in the canonical layout (code i at bits 2i, 2i+1)."""
        wt = np.ascontiguousarray(np.asarray(wt2d, dtype=np.int8))
        K, n = wt.shape
        out = np.empty((K, self.words_per_filter(n)), dtype=np.uint32)
        if self.lib.orc_pack_canonical(_ptr(wt), K, n, _ptr(out)) != 0:
            raise ValueError("codes must be in {-2,-1,1,2}")
        return out

    def unpack_canonical(self, words2d, n: int) -> np.ndarray:
        """Inverse of pack_canonical; raises if a padding field is non-zero."""
        w = np.ascontiguousarray(np.asarray(words2d, dtype=np.uint32))
        K = w.shape[0]
        if w.shape[1] != self.words_per_filter(n):
            raise ValueError("word count does not match n")
        out = np.empty((K, n), dtype=np.int8)
        if self.lib.orc_unpack_canonical(_ptr(w), K, n, _ptr(out)) != 0:
            raise ValueError("non-zero padding field")
        return out

    def dense_conv2d_nchw(self, x, w, stride=(1, 1), pad=(0, 0)):
        """Full-precision convolution (fp32 weights), NCHW; returns (y, bound)
        float64 [N, K, P, Q], bound = sum of |x * w| over the taps."""
        x, w = _f32(x), _f32(w)
        N, C, H, W = x.shape
        K, C2, R, S = w.shape
        assert C2 == C
        P, Q = out_hw(H, W, R, S, stride, pad)
        y = np.empty((N, K, P, Q), dtype=np.float64)
        bound = np.empty_like(y)
        self.lib.orc_dense_conv2d_nchw(_ptr(x), N, C, H, W, _ptr(w), K, R, S, stride[0],
                                       stride[1], pad[0], pad[1], _ptr(y), _ptr(bound))
        return y, bound

    def avgpool_global_nchw(self, x):
        """Mean over H and W of x [N, C, H, W]; returns float64 [N, C]."""
        x = np.ascontiguousarray(np.asarray(x, dtype=np.float64))
        N, C, H, W = x.shape
        y = np.empty((N, C), dtype=np.float64)
        self.lib.orc_avgpool_global_nchw(_ptr(x), N, C, H, W, _ptr(y))
        return y

    def dense_linear(self, x, w):
        """Full-precision fully-connected layer: x [B, Kin], w [Kout, Kin] fp32;
        returns (y, bound) float64 [B, Kout]."""
        x, w = _f32(x), _f32(w)
        B, Kin = x.shape
        Kout = w.shape[0]
        assert w.shape[1] == Kin
        y = np.empty((B, Kout), dtype=np.float64)
        bound = np.empty_like(y)
        self.lib.orc_dense_linear(_ptr(x), B, Kin, _ptr(w), Kout, _ptr(y), _ptr(bound))
        return y, bound


def default() -> Oracle:
    """The oracle built from tbn_oracle.c (compiled on first use)."""
    global _default
    with _lock:
        if _default is None:
            _default = Oracle(build())
        return _default


def __getattr__(name):
    # module-level convenience: oracle.quantize(...), oracle.conv2d_nchw(...)
    if name.startswith("_"):
        raise AttributeError(name)
    return getattr(default(), name)
