"""GPU parity of the fused quantize-and-convolve call (tbn_conv2d_fwd_quant,
Algorithm 1's quantization loop and TwoBitForward in one launch): its codes
and alpha are bitwise those of tbn_quantize_pack, its output bitwise that of
tbn_conv2d_fwd with them, and both match the oracle."""
import numpy as np
import pytest
import torch

import paper_1701_00485_gb300 as tbn
from paper_1701_00485_gb300 import inputs
from parity_util import ConvCase, assert_within, check_quantize, u32

pytestmark = pytest.mark.gpu

CASES = [
    # N, C, H, W, K, R, S, stride, pad, wscale
    (2, 64, 16, 16, 128, 3, 3, 1, 1, 1.3),     # 64-channel TMA, one filter block
    (4, 128, 16, 16, 256, 3, 3, 1, 1, None),   # two filter blocks (VGG c4-like), He weights
    (2, 96, 13, 13, 256, 5, 5, 1, 2, 1.3),     # 32-channel TMA (AlexNet conv2 geometry)
    (3, 64, 9, 11, 200, 3, 3, 2, 1, 1.5),      # stride 2, ragged K
    (2, 32, 12, 12, 64, 1, 1, 1, 0, 1.3),      # short filters (<= 16 words: one thread per filter)
    (2, 160, 7, 7, 96, 1, 1, 2, 0, 1.3),       # 1x1 stride 2 (a projection shortcut), 32-channel TMA
    (1, 1024, 4, 4, 64, 3, 3, 1, 1, 1.3),      # long filters: 576 words per filter
    (256, 9216, 1, 1, 512, 1, 1, 1, 0, None),  # FC-as-conv shape (fc6 rows)
]


@pytest.mark.parametrize("case", CASES)
def test_fused_quant_conv_equals_separate(case):
    N, C, H, W, K, R, S, st, pd, wscale = case
    g = inputs.generator(N * 17 + C * 3 + K + R)
    x = torch.randn(N, H, W, C, generator=g).to(torch.bfloat16).cuda()
    std = wscale if wscale is not None else (2.0 / (C * R * S)) ** 0.5
    Wt = inputs.normal((K, C, R, S), std, g)
    Wl = Wt.permute(0, 2, 3, 1).reshape(K, -1).contiguous().cuda()
    y, codes, alpha = tbn.tbn_conv2d_fwd_quant(x, Wl, K, R, S, (st, st), (pd, pd), relu=True)
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    codes_ref, alpha_ref = tbn.tbn_quantize_pack(Wl)
    y_ref = tbn.tbn_conv2d_fwd(x, codes_ref, alpha_ref, K, R, S, (st, st), (pd, pd),
                               layout=tbn.TBN_NHWC, relu=True, algo=tbn.TBN_CONV_IMPLICIT_GEMM)
    torch.cuda.synchronize()
    assert np.array_equal(u32(codes), u32(codes_ref))
    assert torch.equal(alpha, alpha_ref)
    assert torch.equal(y, y_ref)
    check_quantize(Wl.cpu(), codes, alpha)


def test_fused_quant_conv_matches_oracle():
    N, C, H, W, K = 2, 64, 10, 10, 96
    g = inputs.generator(77)
    x = torch.randn(N, C, H, W, generator=g)
    Wt = inputs.normal((K, C, 3, 3), 1.3, g)
    c = ConvCase(x, Wt, (1, 1), (1, 1))
    Wl = Wt.permute(0, 2, 3, 1).reshape(K, -1).contiguous().cuda()
    xin = x.to(torch.bfloat16).permute(0, 2, 3, 1).contiguous().cuda()
    y, codes, alpha = tbn.tbn_conv2d_fwd_quant(xin, Wl, K, 3, 3, (1, 1), (1, 1),
                                               out_dtype=torch.float32)
    torch.cuda.synchronize()
    check_quantize(Wl.cpu(), codes, alpha)
    y_orc, bound = c.oracle_full(torch.bfloat16)
    assert_within(y.cpu().permute(0, 3, 1, 2).numpy(), y_orc, bound, out_bf16=False,
                  what="fused quant conv")


def test_fused_quant_conv_repeats_with_the_same_workspace():
    # the barrier word is zeroed by every call: back-to-back calls (and a
    # CUDA graph replay) give the same result
    N, C, H, W, K = 2, 64, 8, 8, 128
    g = inputs.generator(78)
    x = torch.randn(N, H, W, C, generator=g).to(torch.bfloat16).cuda()
    Wl = inputs.normal((K, 9 * C), 1.3, g).cuda()
    ws = torch.empty(64, dtype=torch.uint8, device="cuda")
    y0, _, _ = tbn.tbn_conv2d_fwd_quant(x, Wl, K, 3, 3, (1, 1), (1, 1), workspace=ws)
    y1 = torch.empty_like(y0)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        tbn.tbn_conv2d_fwd_quant(x, Wl, K, 3, 3, (1, 1), (1, 1), workspace=ws, out=y1)
        torch.cuda.synchronize()
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr, stream=s):
            tbn.tbn_conv2d_fwd_quant(x, Wl, K, 3, 3, (1, 1), (1, 1), workspace=ws, out=y1)
    y1.zero_()
    for _ in range(3):
        gr.replay()
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    assert torch.equal(y0, y1)


@pytest.mark.parametrize("bad", [dict(C=8), dict(stride=3), dict(C=4096)])
def test_fused_quant_conv_refuses_unsupported(bad):
    # fused quantization takes the TMA activation modes only (C % 32 == 0,
    # stride <= 2) and at most 2048 words per filter
    C, st = bad.get("C", 64), bad.get("stride", 1)
    g = inputs.generator(79)
    x = torch.randn(1, 9, 9, C, generator=g).to(torch.bfloat16).cuda()
    Wl = inputs.normal((64, 9 * C), 1.0, g).cuda()
    with pytest.raises(tbn.TBNError):
        tbn.tbn_conv2d_fwd_quant(x, Wl, 64, 3, 3, (st, st), (1, 1))
