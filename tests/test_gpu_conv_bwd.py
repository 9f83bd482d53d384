"""GPU parity of Algorithm 1's TwoBitBackward through a two-bit convolution
(tbn_conv2d_bwd_data / tbn_conv2d_bwd_filter, NHWC bf16) against the
oracle's adjoint loops.  The input gradient runs on the forward kernels with
alpha*dy rounded to bf16, which adds up to 2^-9 relative per term to the
fp32 accumulation (the `extra` tolerance); the filter gradient sums exact
bf16 products in fp32."""
import numpy as np
import pytest
import torch

import oracle
import paper_1701_00485_gb300 as tbn
from paper_1701_00485_gb300 import inputs
from parity_util import assert_within

pytestmark = pytest.mark.gpu

BF16_TERM = 2.0 ** -9

CASES = [
    # N, C, H, W, K, R, S, stride, pad
    (2, 3, 9, 7, 5, 3, 3, (1, 1), (1, 1)),         # small-tap forward path for dx
    (2, 16, 10, 9, 24, 3, 3, (2, 2), (1, 1)),      # stride 2: dilated dy, ragged last row
    (1, 64, 8, 8, 64, 3, 3, (1, 1), (1, 1)),       # dx on the TMA implicit GEMM (K % 64 == 0)
    (2, 128, 8, 8, 128, 3, 3, (2, 2), (1, 1)),
    (1, 8, 12, 11, 16, 1, 1, (1, 1), (0, 0)),      # 1x1
    (1, 5, 13, 9, 7, 3, 2, (2, 1), (0, 1)),        # R != S, mixed stride / pad
    (1, 32, 9, 9, 40, 5, 5, (1, 1), (2, 2)),       # 5x5
]


def make(case, seed):
    N, C, H, W, K, R, S, st, pd = case
    g = inputs.generator(seed)
    x = torch.randn(N, C, H, W, generator=g).to(torch.bfloat16)
    Wt = inputs.normal((K, C, R, S), 1.2, g)
    P, Q = tbn.conv_out_hw(H, W, R, S, st, pd)
    dy = torch.randn(N, K, P, Q, generator=g).to(torch.bfloat16)
    Wl = Wt.permute(0, 2, 3, 1).reshape(K, -1).contiguous()       # (r, s, c) order
    codes, alpha = tbn.tbn_quantize_pack(Wl.cuda())
    wt, al = oracle.quantize(Wt.reshape(K, -1).numpy())
    return x, dy, codes, alpha, wt.reshape(K, C, R, S), al


@pytest.mark.parametrize("case", CASES)
@pytest.mark.parametrize("dxdt", [torch.float32, torch.bfloat16])
def test_bwd_data_matches_oracle(case, dxdt):
    N, C, H, W, K, R, S, st, pd = case
    x, dy, codes, alpha, wt, al = make(case, 9000 + sum(case[:7]))
    dy_nhwc = dy.permute(0, 2, 3, 1).contiguous().cuda()
    dx = tbn.tbn_conv2d_bwd_data(dy_nhwc, codes, alpha, C, (H, W), R, S, st, pd, out_dtype=dxdt)
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    dx_orc, bound = oracle.conv2d_bwd_data(dy.float().numpy(), wt, al, (H, W), st, pd)
    got = dx.float().cpu().permute(0, 3, 1, 2).numpy()
    assert_within(got, dx_orc, bound, out_bf16=dxdt == torch.bfloat16, extra=BF16_TERM,
                  what="bwd data %s" % (case,))


@pytest.mark.parametrize("case", CASES)
def test_bwd_filter_matches_oracle(case):
    N, C, H, W, K, R, S, st, pd = case
    x, dy, codes, alpha, wt, al = make(case, 9500 + sum(case[:7]))
    dw = tbn.tbn_conv2d_bwd_filter(x.permute(0, 2, 3, 1).contiguous().cuda(),
                                   dy.permute(0, 2, 3, 1).contiguous().cuda(), R, S, st, pd)
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    dw_orc, bound = oracle.conv2d_bwd_filter(x.float().numpy(), dy.float().numpy(), (R, S), st,
                                             pd)
    got = dw.cpu().reshape(K, R, S, C).permute(0, 3, 1, 2).numpy()
    assert_within(got, dw_orc, bound, out_bf16=False, what="bwd filter %s" % (case,))


@pytest.mark.parametrize("i", range(6))
def test_bwd_vgg_small_layer_geometry(i):
    """Each VGG-small convolution's shape (batch 2) through both gradients."""
    s = inputs.VGG_SMALL["convs"][i]
    hw = 32 >> (i // 2)
    case = (2, s.C, hw, hw, s.K, s.R, s.S, (s.stride, s.stride), (s.pad, s.pad))
    N, C, H, W, K, R, S, st, pd = case
    x, dy, codes, alpha, wt, al = make(case, 9900 + i)
    dy_nhwc = dy.permute(0, 2, 3, 1).contiguous().cuda()
    dx = tbn.tbn_conv2d_bwd_data(dy_nhwc, codes, alpha, C, (H, W), R, S, st, pd)
    dw = tbn.tbn_conv2d_bwd_filter(x.permute(0, 2, 3, 1).contiguous().cuda(), dy_nhwc, R, S, st,
                                   pd)
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    dx_orc, bx = oracle.conv2d_bwd_data(dy.float().numpy(), wt, al, (H, W), st, pd)
    assert_within(dx.float().cpu().permute(0, 3, 1, 2).numpy(), dx_orc, bx, out_bf16=True,
                  extra=BF16_TERM, what="vgg c%d bwd data" % (i + 1))
    dw_orc, bw = oracle.conv2d_bwd_filter(x.float().numpy(), dy.float().numpy(), (R, S), st, pd)
    assert_within(dw.cpu().reshape(K, R, S, C).permute(0, 3, 1, 2).numpy(), dw_orc, bw,
                  out_bf16=False, what="vgg c%d bwd filter" % (i + 1))


def test_bwd_is_reproducible_and_ignores_stale_workspace():
    case = (2, 128, 8, 8, 128, 3, 3, (1, 1), (1, 1))
    N, C, H, W, K, R, S, st, pd = case
    x, dy, codes, alpha, wt, al = make(case, 31)
    xn = x.permute(0, 2, 3, 1).contiguous().cuda()
    dyn = dy.permute(0, 2, 3, 1).contiguous().cuda()
    ws = torch.empty(max(tbn.lib().tbn_conv2d_bwd_data_workspace_bytes(N, C, H, W, K, R, S, 1, 1,
                                                                       1, 1),
                         tbn.lib().tbn_conv2d_bwd_filter_workspace_bytes(N, C, H, W, K, R, S, 1,
                                                                         1, 1, 1)),
                     dtype=torch.uint8, device="cuda")
    a1 = tbn.tbn_conv2d_bwd_data(dyn, codes, alpha, C, (H, W), R, S, st, pd, workspace=ws)
    b1 = tbn.tbn_conv2d_bwd_filter(xn, dyn, R, S, st, pd, workspace=ws)
    ws.fill_(0xA5)
    a2 = tbn.tbn_conv2d_bwd_data(dyn, codes, alpha, C, (H, W), R, S, st, pd, workspace=ws)
    ws.fill_(0x5A)
    b2 = tbn.tbn_conv2d_bwd_filter(xn, dyn, R, S, st, pd, workspace=ws)
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    assert torch.equal(a1, a2) and torch.equal(b1, b2)


def test_bwd_rejects_large_padding():
    dy = torch.zeros(1, 4, 4, 8, dtype=torch.bfloat16, device="cuda")
    codes = torch.zeros(8, 1, dtype=torch.int32, device="cuda")
    alpha = torch.ones(8, device="cuda")
    with pytest.raises(tbn.TBNError) as e:
        tbn.tbn_conv2d_bwd_data(dy, codes, alpha, 1, (2, 2), 1, 1, (1, 1), (1, 1))
    assert e.value.status in (tbn.TBN_ERR_UNSUPPORTED, tbn.TBN_ERR_INVALID_ARG)


@pytest.mark.parametrize("i", [1, 5])
def test_bwd_vgg_small_batch128_sampled(i):
    """Full-size VGG-small layers (batch 128, the backward workload's launch
    configuration): dx of three whole images and dW of a 3 x 3 block of
    (filter, channel) pairs, every tap, over the whole batch, against the
    oracle run on just those images / channels."""
    s = inputs.VGG_SMALL["convs"][i]
    hw = 32 >> (i // 2)
    case = (128, s.C, hw, hw, s.K, s.R, s.S, (s.stride, s.stride), (s.pad, s.pad))
    N, C, H, W, K, R, S, st, pd = case
    x, dy, codes, alpha, wt, al = make(case, 7700 + i)
    dy_nhwc = dy.permute(0, 2, 3, 1).contiguous().cuda()
    dx = tbn.tbn_conv2d_bwd_data(dy_nhwc, codes, alpha, C, (H, W), R, S, st, pd)
    dw = tbn.tbn_conv2d_bwd_filter(x.permute(0, 2, 3, 1).contiguous().cuda(), dy_nhwc, R, S, st,
                                   pd)
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    imgs = [0, 77, N - 1]
    dx_orc, bx = oracle.conv2d_bwd_data(dy[imgs].float().numpy(), wt, al, (H, W), st, pd)
    got_dx = dx[imgs].float().cpu().permute(0, 3, 1, 2).numpy()
    assert_within(got_dx, dx_orc, bx, out_bf16=True, extra=BF16_TERM,
                  what="vgg c%d b128 bwd data" % (i + 1))
    ks, cs = [0, 37, K - 1], [0, 53, C - 1]
    dw_orc, bw = oracle.conv2d_bwd_filter(x[:, cs].float().numpy(), dy[:, ks].float().numpy(),
                                          (R, S), st, pd)
    got_dw = dw.cpu().reshape(K, R, S, C).permute(0, 3, 1, 2)[ks][:, cs].numpy()
    assert_within(got_dw, dw_orc, bw, out_bf16=False, what="vgg c%d b128 bwd filter" % (i + 1))
