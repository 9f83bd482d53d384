"""Host-side checks of the C ABI (no GPU needed): the library builds and
loads, exports every function include/tbn.h declares, and rejects invalid
arguments on the host before launching anything."""
import ctypes
import os
import re

import pytest

import paper_1701_00485_gb300 as tbn
from paper_1701_00485_gb300 import build as tbn_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "tbn.h")


@pytest.fixture(scope="module")
def L():
    tbn_build.build()
    return tbn.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = re.findall(r"\b(tbn_[a-z0-9_]+)\s*\(", text)
    return sorted(set(names))


def test_header_declares_the_python_export_list():
    assert declared_functions() == sorted(tbn.EXPORTED)


def test_every_declared_symbol_is_exported(L):
    for name in declared_functions():
        assert hasattr(L, name), name


def test_abi_version_and_sizes(L):
    assert L.tbn_abi_version() == 9
    assert [tbn.packed_words(n) for n in (1, 15, 16, 17, 27, 1152, 16384)] == \
        [1, 1, 1, 2, 2, 72, 1024]
    assert L.tbn_packed_words(0) == -1
    assert L.tbn_status_string(0) == b"ok"
    assert L.tbn_status_string(2) == b"unsupported"


def test_quantize_rejects_bad_arguments(L):
    dummy = ctypes.c_void_p(256)
    assert L.tbn_quantize_pack(None, 4, 16, dummy, dummy, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_quantize_pack(dummy, 0, 16, dummy, dummy, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_quantize_pack(dummy, 4, 0, dummy, dummy, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_quantize_pack(ctypes.c_void_p(258), 4, 16, dummy, dummy, None) == \
        tbn.TBN_ERR_MISALIGNED
    assert L.tbn_quantize_pack(dummy, 4, 1 << 31, dummy, dummy, None) == tbn.TBN_ERR_UNSUPPORTED
    assert b"quantize" in L.tbn_last_error()
    jobs = (tbn.QuantJob * 17)()
    assert L.tbn_quantize_pack_group(jobs, 17, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_quantize_pack_group(jobs, 0, None) == tbn.TBN_ERR_INVALID_ARG


def test_unpack_rejects_bad_arguments(L):
    d = ctypes.c_void_p(256)
    assert L.tbn_unpack(None, d, 1, 1, d, 0, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_unpack(d, None, 1, 1, d, tbn.TBN_UNPACK_F32, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_unpack(d, d, 1, 1, d, 7, None) == tbn.TBN_ERR_INVALID_ARG


def _conv(L, **kw):
    d = ctypes.c_void_p(256)
    a = dict(x=d, xdt=1, layout=1, N=1, C=64, H=8, W=8, codes=d, alpha=d, K=64, R=3, S=3,
             sh=1, sw=1, ph=1, pw=1, y=d, ydt=1, epi=None, algo=0)
    a.update(kw)
    return L.tbn_conv2d_fwd_algo(a["x"], a["xdt"], a["layout"], a["N"], a["C"], a["H"], a["W"],
                                 a["codes"], a["alpha"], a["K"], a["R"], a["S"], a["sh"], a["sw"],
                                 a["ph"], a["pw"], a["y"], a["ydt"], a["epi"], a["algo"], None)


def test_conv_rejects_bad_arguments(L):
    assert _conv(L, x=None) == tbn.TBN_ERR_INVALID_ARG
    assert _conv(L, N=0) == tbn.TBN_ERR_INVALID_ARG
    assert _conv(L, xdt=5) == tbn.TBN_ERR_INVALID_ARG
    assert _conv(L, layout=9) == tbn.TBN_ERR_INVALID_ARG
    assert _conv(L, layout=4) == tbn.TBN_ERR_INVALID_ARG
    assert _conv(L, sh=0) == tbn.TBN_ERR_INVALID_ARG
    assert _conv(L, ph=-1) == tbn.TBN_ERR_INVALID_ARG
    assert _conv(L, H=2, W=2, ph=0, pw=0) == tbn.TBN_ERR_INVALID_ARG   # kernel > input
    assert _conv(L, x=ctypes.c_void_p(257)) == tbn.TBN_ERR_MISALIGNED
    assert _conv(L, C=1 << 20, H=1 << 12, W=1) == tbn.TBN_ERR_UNSUPPORTED
    assert _conv(L, algo=11) == tbn.TBN_ERR_INVALID_ARG
    # huge sizes are refused before any sum or product of them is formed
    assert _conv(L, ph=1 << 62) == tbn.TBN_ERR_UNSUPPORTED
    assert _conv(L, N=1 << 62) == tbn.TBN_ERR_UNSUPPORTED
    assert _conv(L, C=1 << 40, R=1 << 30) == tbn.TBN_ERR_UNSUPPORTED
    assert _conv(L, N=1 << 20, H=8, W=8, C=1, ph=0xFFFF, pw=0xFFFF) == \
        tbn.TBN_ERR_UNSUPPORTED                                      # N P Q above 2^46


def test_space_to_depth_host_rules(L):
    # out [N][Hs][Ws][64], Hs = P + ceil(R/s) - 1, Ws = Q + ceil(S/s) - 1
    assert L.tbn_space_to_depth_elems(256, 3, 227, 227, 11, 11, 4, 4, 0, 0) == 256 * 57 * 57 * 64
    assert L.tbn_space_to_depth_elems(2, 16, 17, 19, 5, 5, 2, 2, 2, 2) == 2 * 11 * 12 * 64
    assert L.tbn_space_to_depth_elems(1, 3, 227, 227, 11, 11, 1, 1, 0, 0) == -1   # stride 1
    assert L.tbn_space_to_depth_elems(1, 5, 227, 227, 11, 11, 4, 4, 0, 0) == -1   # 80 channels
    assert L.tbn_space_to_depth_elems(1, 3, 227, 227, 11, 11, 4, 2, 0, 0) == -1   # unequal
    assert L.tbn_space_to_depth_elems(1, 3, 5, 5, 11, 11, 4, 4, 0, 0) == -1       # kernel > input
    assert L.tbn_space_to_depth_elems(0, 3, 227, 227, 11, 11, 4, 4, 0, 0) == -1
    d, o = ctypes.c_void_p(256), ctypes.c_void_p(1 << 40)
    args = [1, 3, 227, 227, 11, 11, 4, 4, 0, 0]
    assert L.tbn_space_to_depth(None, 1, 0, *args, o, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_space_to_depth(d, 0, 0, *args, o, None) == tbn.TBN_ERR_UNSUPPORTED     # fp32
    assert L.tbn_space_to_depth(d, 1, 2, *args, o, None) == tbn.TBN_ERR_INVALID_ARG     # layout
    assert L.tbn_space_to_depth(d, 1, 0, *args, ctypes.c_void_p((1 << 40) + 8), None) == \
        tbn.TBN_ERR_MISALIGNED
    assert L.tbn_space_to_depth(d, 1, 0, *args, ctypes.c_void_p(512), None) == \
        tbn.TBN_ERR_INVALID_ARG                                                    # overlap
    # the convolution over it: the implicit GEMM only, bf16, equal strides
    s2d = dict(layout=3, C=3, H=227, W=227, K=96, R=11, S=11, sh=4, sw=4, ph=0, pw=0)
    assert _conv(L, algo=1, **s2d) == tbn.TBN_ERR_UNSUPPORTED
    assert _conv(L, algo=3, **s2d) == tbn.TBN_ERR_UNSUPPORTED
    assert _conv(L, xdt=0, **s2d) == tbn.TBN_ERR_UNSUPPORTED
    assert _conv(L, **dict(s2d, K=129)) == tbn.TBN_ERR_UNSUPPORTED
    assert _conv(L, **dict(s2d, sw=2)) == tbn.TBN_ERR_UNSUPPORTED
    assert b"space-to-depth" in L.tbn_last_error()


def test_f8_linear_host_rules(L):
    # prepared layout: ceil(K_out / 128) * 128 rows x K_in / 16 words; K_in % 512 == 0
    assert L.tbn_linear_f8_prepared_words(1000, 16384) == 1024 * 1024
    assert L.tbn_linear_f8_prepared_words(128, 512) == 128 * 32
    assert L.tbn_linear_f8_prepared_words(128, 500) == -1
    assert L.tbn_linear_f8_prepared_words(0, 512) == -1
    assert L.tbn_linear_f8_workspace_bytes(1, 4096, 4096) >= 256
    assert L.tbn_linear_f8_workspace_bytes(2, 4096, 4096) == 0      # batch 1 only
    assert L.tbn_linear_f8_workspace_bytes(1, 32768, 64) == 0       # K_in <= 16384
    assert L.tbn_linear_f8_workspace_bytes(1, 1000, 64) == 0        # K_in % 512
    d = ctypes.c_void_p(256)
    assert L.tbn_linear_prepare_f8(None, 4, 512, d, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_linear_prepare_f8(d, 4, 500, ctypes.c_void_p(1 << 40), None) == tbn.TBN_ERR_UNSUPPORTED
    assert L.tbn_linear_prepare_f8(d, 4, 512, ctypes.c_void_p((1 << 40) + 4), None) == \
        tbn.TBN_ERR_MISALIGNED
    assert L.tbn_linear_prepare_f8(d, 4, 512, ctypes.c_void_p(512), None) == \
        tbn.TBN_ERR_INVALID_ARG                                                  # overlap
    ws = ctypes.c_void_p(1 << 20)
    args = [d, 1, 1, 4096, d, d, 64, d, 1, None]
    assert L.tbn_linear_fwd_f8(*args[:1], 0, *args[2:], ws, 1 << 20, None) == \
        tbn.TBN_ERR_UNSUPPORTED                                                  # fp32 x
    assert L.tbn_linear_fwd_f8(d, 1, 2, 4096, d, d, 64, d, 1, None, ws, 1 << 20, None) == \
        tbn.TBN_ERR_UNSUPPORTED                                                  # B = 2
    assert L.tbn_linear_fwd_f8(d, 1, 1, 4096, d, d, 64, d, 1, None, None, 0, None) == \
        tbn.TBN_ERR_INVALID_ARG                                                  # no workspace


def test_conv_quant_host_rules(L):
    # tbn_conv2d_fwd_quant: filters, a barrier word, no overlap of the filters
    # with the codes and alpha it writes; checked before anything is launched
    v = [ctypes.c_void_p(i << 30) for i in range(1, 7)]
    x, Wf, codes, alpha, y, ws = v

    def call(layout=tbn.TBN_NHWC, C=64, W=Wf, c=codes, a=alpha, w=ws, wb=64):
        return L.tbn_conv2d_fwd_quant(x, 1, layout, 2, C, 8, 8, W, 128, 3, 3, 1, 1, 1, 1, c, a,
                                      y, 1, None, w, wb, None)
    assert call(W=None) == tbn.TBN_ERR_INVALID_ARG
    assert call(w=None, wb=0) == tbn.TBN_ERR_INVALID_ARG
    assert call(wb=2) == tbn.TBN_ERR_INVALID_ARG
    assert call(W=ctypes.c_void_p((2 << 30) + 2)) == tbn.TBN_ERR_MISALIGNED
    assert call(w=ctypes.c_void_p((6 << 30) + 2)) == tbn.TBN_ERR_MISALIGNED
    assert call(c=ctypes.c_void_p((2 << 30) + 4096)) == tbn.TBN_ERR_INVALID_ARG    # overlap
    assert call(a=ctypes.c_void_p((2 << 30) + 4096)) == tbn.TBN_ERR_INVALID_ARG    # overlap
    assert call(C=4096) == tbn.TBN_ERR_UNSUPPORTED                                 # C R S > 32768


def test_select_algo_host_rules(L):
    # without a GPU (or for shapes it cannot take) AUTO falls back to DIRECT;
    # shapes the implicit GEMM never takes are DIRECT everywhere
    assert tbn.tbn_conv2d_select_algo(__import__("torch").float32, tbn.TBN_NHWC,
                                      1, 64, 8, 8, 64, 3, 3) == tbn.TBN_CONV_DIRECT
    assert tbn.tbn_conv2d_select_algo(__import__("torch").bfloat16, tbn.TBN_NCHW,
                                      1, 64, 8, 8, 64, 3, 3) == tbn.TBN_CONV_DIRECT
    # short bf16 filters (C*R*S <= 64) go to the small-tap kernel in either layout
    assert tbn.tbn_conv2d_select_algo(__import__("torch").bfloat16, tbn.TBN_NHWC,
                                      1, 3, 8, 8, 64, 3, 3) == tbn.TBN_CONV_SMALL_TAPS
    assert tbn.tbn_conv2d_select_algo(__import__("torch").bfloat16, tbn.TBN_NCHW,
                                      1, 7, 8, 8, 64, 3, 3) == tbn.TBN_CONV_SMALL_TAPS
    assert tbn.tbn_conv2d_select_algo(__import__("torch").bfloat16, tbn.TBN_NCHW,
                                      1, 8, 8, 8, 64, 3, 3) == tbn.TBN_CONV_DIRECT
    # NCHW in, NHWC out: small-tap for short bf16 filters, else the direct kernel
    assert tbn.tbn_conv2d_select_algo(__import__("torch").bfloat16, tbn.TBN_NCHW_NHWC,
                                      128, 3, 32, 32, 128, 3, 3, (1, 1), (1, 1)) == \
        tbn.TBN_CONV_SMALL_TAPS
    assert tbn.tbn_conv2d_select_algo(__import__("torch").bfloat16, tbn.TBN_NCHW_NHWC,
                                      1, 64, 8, 8, 64, 3, 3) == tbn.TBN_CONV_DIRECT
    assert tbn.tbn_conv2d_select_algo(__import__("torch").float32, tbn.TBN_NCHW_NHWC,
                                      1, 3, 8, 8, 64, 3, 3) == tbn.TBN_CONV_DIRECT


def test_linear_and_glue_reject_bad_arguments(L):
    d = ctypes.c_void_p(256)
    assert L.tbn_linear_fwd(None, 1, 1, 64, d, d, 8, d, 1, None, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_linear_fwd(d, 1, 0, 64, d, d, 8, d, 1, None, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_linear_fwd(d, 1, 1 << 40, 64, d, d, 8, d, 1, None, None) == \
        tbn.TBN_ERR_UNSUPPORTED
    assert L.tbn_linear_fwd_ws(None, 1, 1, 64, d, d, 8, d, 1, None, d, 4096, None) == \
        tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_linear_fwd_ws(d, 1, 1, 64, d, d, 8, ctypes.c_void_p(257), 1, None, d, 4096,
                               None) == tbn.TBN_ERR_MISALIGNED
    assert L.tbn_maxpool2d_nhwc(d, 1, 1, 4, 4, 8, 5, 5, 1, 1, 0, 0, d, None) == \
        tbn.TBN_ERR_INVALID_ARG
    # padding must stay below the window
    assert L.tbn_maxpool2d_nhwc(d, 1, 1, 8, 8, 8, 3, 3, 2, 2, 3, 1, d, None) == \
        tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_maxpool2d_nhwc(d, 1, 1, 8, 8, 8, 3, 3, 2, 2, -1, 1, d, None) == \
        tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_nchw_to_nhwc(d, 1, 1, 4, 4, 4, 3, d, None) == tbn.TBN_ERR_INVALID_ARG


def test_repack_and_dense_layers_reject_bad_arguments(L):
    d = ctypes.c_void_p(256)
    assert L.tbn_repack(None, 4, 16, d, 0, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_repack(d, 4, 16, d, 2, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_repack(d, 0, 16, d, 0, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_repack(d, 4, 16, ctypes.c_void_p(258), 0, None) == tbn.TBN_ERR_MISALIGNED
    # partial overlap is refused (in == out is allowed)
    assert L.tbn_repack(d, 4, 16, ctypes.c_void_p(260), 0, None) == tbn.TBN_ERR_INVALID_ARG
    args = [d, 1, tbn.TBN_NCHW_NHWC, 2, 3, 16, 16, d, 64, 7, 7, 2, 2, 3, 3, d, 1, 1, None]
    bad = list(args); bad[7] = None
    assert L.tbn_dense_conv2d_fwd(*bad) == tbn.TBN_ERR_INVALID_ARG
    bad = list(args); bad[9] = 30                     # kernel larger than the padded input
    assert L.tbn_dense_conv2d_fwd(*bad) == tbn.TBN_ERR_INVALID_ARG
    bad = list(args); bad[7] = ctypes.c_void_p(258)   # weights not 4-byte aligned
    assert L.tbn_dense_conv2d_fwd(*bad) == tbn.TBN_ERR_MISALIGNED
    assert L.tbn_avgpool2d_global_nhwc(d, 1, 2, 0, 7, 512, d, 0, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_avgpool2d_global_nhwc(d, 3, 2, 7, 7, 512, d, 0, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_dense_linear_fwd(d, 2, 512, None, 1000, d, 0, 0, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_dense_linear_fwd(d, 2, 512, d, 1000, ctypes.c_void_p(258), 0, 0, None) == \
        tbn.TBN_ERR_MISALIGNED
    assert L.tbn_dense_linear_fwd(d, 2, 1 << 40, d, 1000, d, 0, 0, None) == \
        tbn.TBN_ERR_UNSUPPORTED


def test_linear_workspace_query(L):
    """Scratch of the batch-1 fp32 table GEMV: the fp32 partial sum of every
    512-input chunk for each row (rows rounded up to blocks of 128), rounded
    to 256 bytes; none for one chunk or where the kernel does not apply."""
    f32 = __import__("torch").float32
    ws = lambda B, K_in, K_out: tbn.tbn_linear_workspace_bytes(B, K_in, K_out, f32)
    assert ws(1, 16384, 16384) == 32 * 16384 * 4
    assert ws(1, 4096, 1000) == 8 * 1024 * 4
    assert ws(1, 576, 33) == 2 * 128 * 4
    assert ws(1, 512, 4096) == 0            # one chunk: results written directly
    assert ws(2, 4096, 4096) == 0           # batch > 1
    assert ws(1, 4000, 4096) == 0           # K_in % 64 != 0: no TMA rows
    assert tbn.tbn_linear_workspace_bytes(1, 4096, 4096) == 0   # bf16 x: tensor-core GEMV


def test_python_binding_requires_cuda_tensors():
    import torch
    with pytest.raises(ValueError):
        tbn.tbn_quantize_pack(torch.zeros(2, 16))


def _bwd_data(L, **kw):
    d = ctypes.c_void_p(256)
    a = dict(dy=d, N=2, C=64, H=8, W=8, codes=d, alpha=d, K=64, R=3, S=3, sh=1, sw=1, ph=1,
             pw=1, dx=d, dxdt=1, ws=d, wsb=1 << 30)
    a.update(kw)
    return L.tbn_conv2d_bwd_data(a["dy"], a["N"], a["C"], a["H"], a["W"], a["codes"],
                                 a["alpha"], a["K"], a["R"], a["S"], a["sh"], a["sw"], a["ph"],
                                 a["pw"], a["dx"], a["dxdt"], a["ws"], a["wsb"], None)


def _bwd_filter(L, **kw):
    d = ctypes.c_void_p(256)
    a = dict(x=d, dy=d, N=2, C=64, H=8, W=8, K=64, R=3, S=3, sh=1, sw=1, ph=1, pw=1, dw=d,
             ws=d, wsb=1 << 30)
    a.update(kw)
    return L.tbn_conv2d_bwd_filter(a["x"], a["dy"], a["N"], a["C"], a["H"], a["W"], a["K"],
                                   a["R"], a["S"], a["sh"], a["sw"], a["ph"], a["pw"], a["dw"],
                                   a["ws"], a["wsb"], None)


@pytest.mark.parametrize("call", [_bwd_data, _bwd_filter])
def test_bwd_rejects_bad_arguments(L, call):
    """Every check of the TwoBitBackward entry points returns before a launch."""
    first = "dy" if call is _bwd_data else "x"
    assert call(L, **{first: None}) == tbn.TBN_ERR_INVALID_ARG
    assert call(L, ws=None) == tbn.TBN_ERR_INVALID_ARG
    assert call(L, N=0) == tbn.TBN_ERR_INVALID_ARG
    assert call(L, K=-1) == tbn.TBN_ERR_INVALID_ARG
    assert call(L, sh=0) == tbn.TBN_ERR_INVALID_ARG
    assert call(L, pw=-1) == tbn.TBN_ERR_INVALID_ARG
    assert call(L, H=1, W=1, ph=0, pw=0) == tbn.TBN_ERR_INVALID_ARG   # kernel > input
    assert call(L, ph=3) == tbn.TBN_ERR_UNSUPPORTED                    # pad > R - 1
    assert call(L, ph=1 << 62) == tbn.TBN_ERR_UNSUPPORTED              # no overflow first
    assert call(L, N=1 << 31) == tbn.TBN_ERR_UNSUPPORTED
    assert call(L, N=1 << 20, H=1 << 10, W=1 << 10) == tbn.TBN_ERR_UNSUPPORTED
    assert call(L, C=1 << 28) == tbn.TBN_ERR_UNSUPPORTED               # R S C >= 2^30
    assert call(L, wsb=0) == tbn.TBN_ERR_INVALID_ARG                   # workspace too small
    assert call(L, ws=ctypes.c_void_p(128)) == tbn.TBN_ERR_MISALIGNED  # workspace 256-aligned
    assert call(L, dy=ctypes.c_void_p(257)) == tbn.TBN_ERR_MISALIGNED
    if call is _bwd_data:
        assert call(L, dxdt=7) == tbn.TBN_ERR_INVALID_ARG
        assert call(L, codes=None) == tbn.TBN_ERR_INVALID_ARG
    else:
        assert call(L, dw=ctypes.c_void_p(258)) == tbn.TBN_ERR_MISALIGNED


def test_bwd_workspace_queries(L):
    """Zero for shapes the entry points refuse; for valid shapes the input
    gradient's scratch covers the transposed codes, the unit scales and the
    dilated alpha-scaled dy, and the filter gradient's holds at least one
    fp32 partial of dW."""
    qd, qf = L.tbn_conv2d_bwd_data_workspace_bytes, L.tbn_conv2d_bwd_filter_workspace_bytes
    assert qd(0, 64, 8, 8, 64, 3, 3, 1, 1, 1, 1) == 0
    assert qf(2, 64, 8, 8, 64, 3, 3, 1, 1, 3, 1) == 0
    assert qf(2, 64, 8, 8, 64, 3, 3, 1, 1, 1 << 62, 1) == 0
    N, C, H, W, K, R, S = 2, 64, 8, 8, 96, 3, 3
    wd = qd(N, C, H, W, K, R, S, 2, 2, 1, 1)
    words_t = C * ((R * S * K + 15) // 16) * 4
    Hd, Wd = H + 2 - R + 1, W + 2 - S + 1                      # dilated dy extent
    assert wd >= words_t + C * 4 + N * Hd * Wd * K * 2 and wd % 256 == 0
    wf = qf(N, C, H, W, K, R, S, 1, 1, 1, 1)
    assert wf >= K * R * S * C * 4 and wf % 256 == 0
    assert wf <= (64 << 20) + 256                              # partial tiles capped at 64 MB


def test_selftest_wait_timeout_rejects_bad_limits(L):
    assert L.tbn_selftest_wait_timeout(0, None) == tbn.TBN_ERR_INVALID_ARG
    assert L.tbn_selftest_wait_timeout(1000001, None) == tbn.TBN_ERR_INVALID_ARG
