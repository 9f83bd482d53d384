"""GPU parity of the space-to-depth path of a strided first layer:
tbn_space_to_depth (a layout change: bit-exact against its definition
written out in NumPy below) and tbn_conv2d_fwd with layout TBN_S2D_NHWC (the
implicit GEMM with the filter decoded once into tensor memory), compared
per output with the oracle's seven-loop convolution of the original input:
|y_gpu - y_orc| <= 2e-3 * |alpha| * sum|x| (+ the bf16 output rounding)."""
import numpy as np
import pytest
import torch

import paper_1701_00485_gb300 as tbn
from paper_1701_00485_gb300 import inputs
from parity_util import ConvCase, assert_within, random_sites

pytestmark = pytest.mark.gpu


def s2d_reference(x_nchw: np.ndarray, R, S, s, pad):
    """out[n, Y, X, (dy s + dx) C + c] = x[n, c, s Y + dy - ph, s X + dx - pw]."""
    N, C, H, W = x_nchw.shape
    ph, pw = pad
    P = (H + 2 * ph - R) // s + 1
    Q = (W + 2 * pw - S) // s + 1
    Hs = P + (R + s - 1) // s - 1
    Ws = Q + (S + s - 1) // s - 1
    out = np.zeros((N, Hs, Ws, 64), dtype=x_nchw.dtype)
    for dy in range(s):
        for dx in range(s):
            for c in range(C):
                j = (dy * s + dx) * C + c
                for Y in range(Hs):
                    h = s * Y + dy - ph
                    if not 0 <= h < H:
                        continue
                    w = s * np.arange(Ws) + dx - pw
                    ok = (w >= 0) & (w < W)
                    out[:, Y, ok, j] = x_nchw[:, c, h, w[ok]]
    return out


S2D_LAYOUT = [
    # N, C, H, W, R, S, stride, pad
    (2, 3, 31, 29, 11, 11, 4, (0, 0)),
    (1, 3, 227, 227, 11, 11, 4, (0, 0)),   # AlexNet's first layer
    (2, 16, 17, 19, 5, 5, 2, (2, 2)),      # 64 channels used
    (3, 5, 20, 14, 7, 5, 3, (1, 2)),       # 45 channels, padding
    (1, 3, 300, 9, 3, 3, 2, (1, 1)),       # tall image
    (1, 1, 9, 300, 3, 3, 2, (0, 1)),       # a row wider than one 64-pixel chunk
]


@pytest.mark.parametrize("case", S2D_LAYOUT)
@pytest.mark.parametrize("layout", [tbn.TBN_NCHW, tbn.TBN_NHWC])
def test_space_to_depth_is_bit_exact(case, layout):
    N, C, H, W, R, S, s, pad = case
    g = inputs.generator(N * 1000 + C * 100 + H + W + R)
    x = torch.randn(N, C, H, W, generator=g).to(torch.bfloat16)
    xin = x if layout == tbn.TBN_NCHW else x.permute(0, 2, 3, 1).contiguous()
    out = tbn.tbn_space_to_depth(xin.cuda(), R, S, (s, s), pad, layout=layout)
    torch.cuda.synchronize()
    got = out.cpu().view(torch.int16).numpy()
    want = s2d_reference(x.view(torch.int16).numpy(), R, S, s, pad)
    assert got.shape == want.shape
    bad = np.argwhere(got != want)
    assert bad.size == 0, "first difference at %s" % (bad[0].tolist(),)


S2D_CONV = [
    # N, C, H, W, K, R, S, stride, pad
    (2, 3, 227, 227, 96, 11, 11, 4, (0, 0)),   # AlexNet conv1: 9 resident K blocks
    (3, 3, 31, 29, 96, 11, 11, 4, (0, 0)),     # ragged tiles
    (2, 3, 39, 41, 128, 11, 11, 4, (2, 1)),    # padding, K = 128
    (2, 16, 17, 19, 40, 5, 5, 2, (2, 2)),      # 64 s2d channels, ragged K
    (2, 5, 20, 14, 8, 7, 5, 3, (1, 2)),        # 45 channels, R != S
    (4, 4, 16, 16, 64, 3, 3, 2, (1, 1)),       # 2x2 resident K blocks
    (1, 5, 60, 44, 8, 7, 5, 3, (1, 2)),        # R' != S', ragged last tile
    (2, 3, 63, 63, 96, 11, 11, 4, (0, 0)),     # one tile per image
    (1, 12, 64, 64, 32, 3, 3, 2, (1, 1)),      # 3x3 / 2 over 12 channels
]


def _run_s2d(c: ConvCase, out_dtype, relu=False):
    N, C, H, W = c.x.shape
    Wl, codes, alpha = c.quantize_gpu(tbn.TBN_NHWC)          # (r, s, c) order
    xs = tbn.tbn_space_to_depth(c.x.to(torch.bfloat16).cuda(), c.R, c.S, c.stride, c.pad,
                                layout=tbn.TBN_NCHW)
    y = tbn.tbn_conv2d_fwd(xs, codes, alpha, c.K, c.R, c.S, c.stride, c.pad,
                           layout=tbn.TBN_S2D_NHWC, in_chw=(C, H, W), out_dtype=out_dtype,
                           relu=relu)
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    return y.float().cpu().permute(0, 3, 1, 2).contiguous().numpy()


@pytest.mark.parametrize("case", S2D_CONV)
@pytest.mark.parametrize("ydt", [torch.bfloat16, torch.float32])
def test_space_to_depth_conv_matches_oracle(case, ydt):
    N, C, H, W, K, R, S, s, pad = case
    g = inputs.generator(sum(case[:7]) + 17)
    x = torch.randn(N, C, H, W, generator=g)
    Wt = inputs.normal((K, C, R, S), 1.3, g)   # wide weights: all four codes occur
    c = ConvCase(x, Wt, (s, s), pad)
    y = _run_s2d(c, ydt)
    if N * K * y.shape[2] * y.shape[3] <= 400_000:
        y_orc, bound = c.oracle_full(torch.bfloat16)
        assert_within(y, y_orc, bound, out_bf16=(ydt == torch.bfloat16), what="s2d %s" % (case,))
    else:
        sites = random_sites(y.shape, 3000, seed=sum(case[:7]))
        y_orc, bound = c.oracle_sites(torch.bfloat16, sites)
        got = y[tuple(sites.T)]
        assert_within(got, y_orc, bound, out_bf16=(ydt == torch.bfloat16),
                      what="s2d sites %s" % (case,))


def test_space_to_depth_conv_with_relu():
    # He-normal weights (the networks' draw), fp32 output, fused ReLU
    N, C, H, W, K = 2, 3, 63, 63, 96
    g = inputs.generator(4242)
    x = torch.randn(N, C, H, W, generator=g)
    c = ConvCase(x, inputs.he_normal(K, C, 11, 11, g), (4, 4), (0, 0))
    y = _run_s2d(c, torch.float32, relu=True)
    y_orc, bound = c.oracle_full(torch.bfloat16)
    assert_within(y, np.maximum(y_orc, 0.0), bound, out_bf16=False, epilogue=True,
                  what="s2d relu")


@pytest.mark.parametrize("bad", [
    dict(K=129),                       # two filter blocks: not resident
    dict(stride=(4, 2)),               # unequal strides
])
def test_space_to_depth_conv_refuses_unsupported(bad):
    N, C, H, W, K, R, S = 1, 3, 31, 31, bad.get("K", 96), 11, 11
    stride = bad.get("stride", (4, 4))
    g = inputs.generator(5)
    Wt = inputs.he_normal(K, C, R, S, g).permute(0, 2, 3, 1).reshape(K, -1).contiguous().cuda()
    codes, alpha = tbn.tbn_quantize_pack(Wt)
    xs = torch.zeros(tbn.space_to_depth_shape(N, C, H, W, R, S, (4, 4), (0, 0)),
                     dtype=torch.bfloat16, device="cuda")
    with pytest.raises((tbn.TBNError, ValueError)):
        tbn.tbn_conv2d_fwd(xs, codes, alpha, K, R, S, stride, (0, 0), layout=tbn.TBN_S2D_NHWC,
                           in_chw=(C, H, W))
