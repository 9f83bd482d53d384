"""Guard bands around every caller-owned buffer a kernel writes (outputs and
workspaces): the buffer sits 256 bytes into an allocation whose every byte
holds a sentinel.  After the call the bytes before and after it must still
hold the sentinel (no kernel wrote outside its buffer), and the result must
equal, bit for bit, the same call into a fresh tensor.  This stands in for
a memory checker on the shapes with ragged edges of each kernel path."""
import pytest
import torch

import paper_1701_00485_gb300 as tbn
from paper_1701_00485_gb300 import inputs

pytestmark = pytest.mark.gpu

GUARD = 256          # bytes on each side (keeps 16-byte alignment for TMA)
SENTINEL = 0xA7


def guarded(shape, dtype):
    """(allocation, view of `shape` 256 bytes into it), all bytes = sentinel."""
    es = torch.empty((), dtype=dtype).element_size()
    g = GUARD // es
    n = 1
    for d in shape:
        n *= d
    buf = torch.empty(n + 2 * g, dtype=dtype, device="cuda")
    buf.view(torch.uint8).fill_(SENTINEL)
    return buf, buf[g:g + n].view(shape)


def assert_guards(buf, what):
    raw = buf.view(torch.uint8)
    assert bool(torch.all(raw[:GUARD] == SENTINEL)), "%s: write before the buffer" % what
    assert bool(torch.all(raw[-GUARD:] == SENTINEL)), "%s: write after the buffer" % what


def _layer(K, n, seed):
    W = inputs.normal((K, n), 1.2, inputs.generator(seed)).cuda()
    return W, *tbn.tbn_quantize_pack(W)


@pytest.mark.parametrize("K,n", [(37, 300), (1, 1), (130, 1152)])
def test_quantize_stays_inside_codes_and_alpha(K, n):
    W, codes_ref, alpha_ref = _layer(K, n, K + n)
    cb, codes = guarded((K, tbn.packed_words(n)), torch.int32)
    ab, alpha = guarded((K,), torch.float32)
    tbn.tbn_quantize_pack(W, codes=codes, alpha=alpha)
    torch.cuda.synchronize()
    assert_guards(cb, "codes")
    assert_guards(ab, "alpha")
    assert torch.equal(codes, codes_ref) and torch.equal(alpha, alpha_ref)


CONV = [
    # N, C, H, W, K, R, S, stride, pad, layout, out dtype, algo, pool
    (3, 64, 13, 13, 96, 3, 3, (1, 1), (1, 1), tbn.TBN_NHWC, torch.bfloat16,
     tbn.TBN_CONV_IMPLICIT_GEMM, 0),                          # TMA store, K < 128
    (5, 64, 7, 7, 200, 3, 3, (1, 1), (1, 1), tbn.TBN_NHWC, torch.float32,
     tbn.TBN_CONV_IMPLICIT_GEMM, 0),                          # fp32 out, ragged K
    (3, 128, 16, 16, 200, 3, 3, (1, 1), (1, 1), tbn.TBN_NHWC, torch.bfloat16,
     tbn.TBN_CONV_IMPLICIT_GEMM, 2),                          # fused 2x2 pool, ragged K
    (2, 5, 9, 7, 70, 3, 3, (1, 1), (1, 1), tbn.TBN_NHWC, torch.float32,
     tbn.TBN_CONV_IMPLICIT_GEMM, 0),                          # gathered activations
    (2, 3, 32, 32, 128, 3, 3, (1, 1), (1, 1), tbn.TBN_NHWC, torch.bfloat16,
     tbn.TBN_CONV_SMALL_TAPS, 0),                             # tcgen05 small-tap
    (3, 4, 15, 13, 37, 3, 3, (2, 2), (1, 1), tbn.TBN_NCHW, torch.float32,
     tbn.TBN_CONV_SMALL_TAPS, 0),                             # mma.sync small-tap
    (2, 70, 5, 5, 65, 3, 3, (1, 1), (1, 1), tbn.TBN_NCHW, torch.float32,
     tbn.TBN_CONV_DIRECT, 0),                                 # direct
]


@pytest.mark.parametrize("case", CONV)
def test_conv_stays_inside_its_output(case):
    N, C, H, W, K, R, S, st, pd, layout, ydt, algo, pool = case
    g = inputs.generator(sum(case[:7]))
    x = torch.randn(N, C, H, W, generator=g).to(torch.bfloat16)
    if layout == tbn.TBN_NHWC:
        x = x.permute(0, 2, 3, 1).contiguous()
    x = x.cuda()
    _, codes, alpha = _layer(K, C * R * S, 7 + K)
    ref = tbn.tbn_conv2d_fwd(x, codes, alpha, K, R, S, st, pd, layout=layout, out_dtype=ydt,
                             relu=True, algo=algo, pool=pool)
    yb, y = guarded(tuple(ref.shape), ydt)
    tbn.tbn_conv2d_fwd(x, codes, alpha, K, R, S, st, pd, layout=layout, out_dtype=ydt,
                       relu=True, algo=algo, pool=pool, out=y)
    torch.cuda.synchronize()
    assert_guards(yb, "conv %s" % (case[:9],))
    assert torch.equal(y, ref)
    assert tbn.tbn_device_error() == 0


LINEAR = [
    # B, K_in, K_out, x dtype, out dtype
    (3, 1024, 1000, torch.bfloat16, torch.bfloat16),   # tensor-core GEMV, ragged rows
    (1, 4096, 520, torch.bfloat16, torch.float32),
    (1, 512, 700, torch.float32, torch.float32),       # table-lookup GEMV
    (20, 192, 33, torch.bfloat16, torch.bfloat16),     # 1x1 convolution path
]


@pytest.mark.parametrize("case", LINEAR)
def test_linear_stays_inside_its_output(case):
    B, K_in, K_out, xdt, ydt = case
    x = torch.randn(B, K_in, generator=inputs.generator(K_in + K_out)).to(xdt).cuda()
    _, codes, alpha = _layer(K_out, K_in, 3 * K_out)
    ref = tbn.tbn_linear_fwd(x, codes, alpha, K_out, out_dtype=ydt)
    yb, y = guarded((B, K_out), ydt)
    tbn.tbn_linear_fwd(x, codes, alpha, K_out, out_dtype=ydt, out=y)
    torch.cuda.synchronize()
    assert_guards(yb, "linear %s" % (case,))
    assert torch.equal(y, ref)


BWD = [
    # N, C, H, W, K, R, S, stride, pad
    (2, 64, 8, 8, 96, 3, 3, (1, 1), (1, 1)),          # tcgen05 filter gradient, ragged K
    (2, 16, 10, 9, 24, 3, 3, (2, 2), (1, 1)),         # stride 2 (dilated dy)
    (2, 3, 9, 7, 5, 3, 3, (1, 1), (1, 1)),            # register path, C = 3
]


@pytest.mark.parametrize("case", BWD)
def test_bwd_stays_inside_its_workspace(case):
    N, C, H, W, K, R, S, st, pd = case
    g = inputs.generator(sum(case[:7]) + 5)
    P, Q = tbn.conv_out_hw(H, W, R, S, st, pd)
    x = torch.randn(N, H, W, C, generator=g).to(torch.bfloat16).cuda()
    dy = torch.randn(N, P, Q, K, generator=g).to(torch.bfloat16).cuda()
    _, codes, alpha = _layer(K, C * R * S, 11 + K)
    shape = (N, C, H, W, K, R, S, st[0], st[1], pd[0], pd[1])
    nd = int(tbn.lib().tbn_conv2d_bwd_data_workspace_bytes(*shape))
    nf = int(tbn.lib().tbn_conv2d_bwd_filter_workspace_bytes(*shape))
    dx_ref = tbn.tbn_conv2d_bwd_data(dy, codes, alpha, C, (H, W), R, S, st, pd)
    dw_ref = tbn.tbn_conv2d_bwd_filter(x, dy, R, S, st, pd)
    wb, ws = guarded((nd,), torch.uint8)
    dx = tbn.tbn_conv2d_bwd_data(dy, codes, alpha, C, (H, W), R, S, st, pd, workspace=ws)
    torch.cuda.synchronize()
    assert_guards(wb, "bwd data workspace %s" % (case,))
    wb, ws = guarded((nf,), torch.uint8)
    dw = tbn.tbn_conv2d_bwd_filter(x, dy, R, S, st, pd, workspace=ws)
    torch.cuda.synchronize()
    assert_guards(wb, "bwd filter workspace %s" % (case,))
    assert torch.equal(dx, dx_ref) and torch.equal(dw, dw_ref)
    assert tbn.tbn_device_error() == 0


DENSE = [
    # N, C, H, W, K, R, S, stride, pad, layout, out dtype
    (2, 3, 37, 45, 64, 7, 7, (2, 2), (3, 3), tbn.TBN_NCHW_NHWC, torch.bfloat16),   # stem, staged
    (1, 5, 13, 70, 72, 3, 3, (1, 1), (1, 1), tbn.TBN_NCHW_NHWC, torch.bfloat16),   # two filter blocks
    (2, 3, 19, 21, 20, 5, 5, (2, 2), (2, 2), tbn.TBN_NCHW_NHWC, torch.float32),    # direct stores
    (1, 4, 9, 11, 12, 3, 3, (1, 1), (0, 0), tbn.TBN_NHWC, torch.bfloat16),         # K % 8 != 0
]


@pytest.mark.parametrize("case", DENSE)
def test_dense_conv_stays_inside_its_output(case):
    N, C, H, W, K, R, S, st, pd, layout, ydt = case
    g = inputs.generator(sum(case[:7]) + 3)
    x = torch.randn(N, C, H, W, generator=g).to(torch.bfloat16)
    if layout == tbn.TBN_NHWC:
        x = x.permute(0, 2, 3, 1).contiguous()
    x = x.cuda()
    w = inputs.normal((K, C, R, S), 0.2, g).cuda()
    ref = tbn.tbn_dense_conv2d_fwd(x, w, st, pd, layout=layout, out_dtype=ydt, relu=True)
    yb, y = guarded(tuple(ref.shape), ydt)
    tbn.tbn_dense_conv2d_fwd(x, w, st, pd, layout=layout, out_dtype=ydt, relu=True, out=y)
    torch.cuda.synchronize()
    assert_guards(yb, "dense conv %s" % (case[:9],))
    assert torch.equal(y, ref)


def test_fused_quant_conv_stays_inside_its_outputs():
    # codes, alpha and y of the fused quantize-and-convolve launch
    N, C, H, W, K = 2, 96, 9, 11, 200
    g = inputs.generator(91)
    x = torch.randn(N, H, W, C, generator=g).to(torch.bfloat16).cuda()
    Wl = inputs.normal((K, 9 * C), 1.2, g).cuda()
    y_ref, c_ref, a_ref = tbn.tbn_conv2d_fwd_quant(x, Wl, K, 3, 3, (1, 1), (1, 1), relu=True)
    cb, codes = guarded(tuple(c_ref.shape), torch.int32)
    ab, alpha = guarded((K,), torch.float32)
    yb, y = guarded(tuple(y_ref.shape), torch.bfloat16)
    tbn.tbn_conv2d_fwd_quant(x, Wl, K, 3, 3, (1, 1), (1, 1), relu=True, codes=codes, alpha=alpha,
                             out=y)
    torch.cuda.synchronize()
    for buf, what in ((cb, "codes"), (ab, "alpha"), (yb, "y")):
        assert_guards(buf, "fused quant conv " + what)
    assert torch.equal(codes, c_ref) and torch.equal(alpha, a_ref) and torch.equal(y, y_ref)
    assert tbn.tbn_device_error() == 0


def test_space_to_depth_stays_inside_its_output():
    N, C, H, W = 2, 3, 45, 51
    x = torch.randn(N, C, H, W, generator=inputs.generator(92)).to(torch.bfloat16).cuda()
    ref = tbn.tbn_space_to_depth(x, 11, 11, (4, 4), (0, 0), layout=tbn.TBN_NCHW)
    ob, out = guarded(tuple(ref.shape), torch.bfloat16)
    tbn.tbn_space_to_depth(x, 11, 11, (4, 4), (0, 0), layout=tbn.TBN_NCHW, out=out)
    torch.cuda.synchronize()
    assert_guards(ob, "space to depth")
    assert torch.equal(out, ref)
