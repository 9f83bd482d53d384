"""GPU parity of tbn_linear_fwd (tensor-core GEMV for B <= 8, 1x1
convolution otherwise) and of the glue kernels, against the oracle."""
import numpy as np
import pytest
import torch

import oracle
import paper_1701_00485_gb300 as tbn
from paper_1701_00485_gb300 import inputs
from parity_util import assert_within, check_quantize

pytestmark = pytest.mark.gpu


def run_linear(W, x, out_dtype, relu=False, residual=None):
    codes, alpha = tbn.tbn_quantize_pack(W.cuda())
    check_quantize(W, codes, alpha)
    y = tbn.tbn_linear_fwd(x.cuda(), codes, alpha, W.shape[0], out_dtype=out_dtype, relu=relu,
                           residual=residual.cuda() if residual is not None else None)
    torch.cuda.synchronize()
    wt, al = oracle.quantize(W.numpy())
    y_orc, bound = oracle.linear(x.float().numpy(), wt, al)
    return y.float().cpu().numpy(), y_orc, bound


@pytest.mark.parametrize("B", [1, 2, 3, 8])
@pytest.mark.parametrize("K_in,K_out", [(64, 16), (256, 48), (1024, 100), (4096, 4096)])
def test_gemv_matches_oracle(B, K_in, K_out):
    g = inputs.generator(B * 131 + K_in + K_out)
    W = inputs.normal((K_out, K_in), 1.3, g)
    x = torch.randn(B, K_in, generator=g).to(torch.bfloat16)
    y, y_orc, bound = run_linear(W, x, torch.float32)
    assert_within(y, y_orc, bound, out_bf16=False, what="gemv")
    y, y_orc, bound = run_linear(W, x, torch.bfloat16)
    assert_within(y, y_orc, bound, out_bf16=True, what="gemv bf16")


@pytest.mark.parametrize("B,K_in,K_out", [
    (7, 64, 16),        # one stage, one tile
    (4, 3072, 33),      # one tile per band: six warps split K, fixed-order sum
    (5, 4160, 20000),   # nine tiles per band, ragged last stage
    (3, 1024, 38912),   # sixteen tiles per band
    (2, 576, 40000),    # two bands per CTA
    (1, 8192, 1000),    # K split over sixteen warps
    (8, 2048, 8192),    # four tiles per band, four warps per tile
])
def test_gemv_launch_shapes(B, K_in, K_out):
    """Shapes that exercise every branch of the GEMV work split."""
    g = inputs.generator(B * 7 + K_in * 3 + K_out)
    W = inputs.normal((K_out, K_in), 1.1, g)
    x = torch.randn(B, K_in, generator=g).to(torch.bfloat16)
    y, y_orc, bound = run_linear(W, x, torch.float32)
    assert_within(y, y_orc, bound, out_bf16=False, what="gemv shapes")


@pytest.mark.parametrize("K", inputs.GEMV_SIZES)
@pytest.mark.parametrize("B", inputs.GEMV_BATCHES)
def test_gemv_workload_full(K, B):
    """The GEMV workload at full size: every output compared with the oracle."""
    W, x = inputs.gemv_inputs(K, B)
    y, y_orc, bound = run_linear(W, x, torch.bfloat16)
    assert_within(y, y_orc, bound, out_bf16=True, what="gemv K=%d B=%d" % (K, B))


def test_gemv_epilogue():
    g = inputs.generator(99)
    W = inputs.normal((200, 512), 1.0, g)
    x = torch.randn(3, 512, generator=g).to(torch.bfloat16)
    res = torch.randn(3, 200, generator=g)
    y, y_orc, bound = run_linear(W, x, torch.float32, relu=True, residual=res)
    want = oracle.epilogue(y_orc, res.numpy(), relu=True)
    assert_within(y, want, bound, out_bf16=False, epilogue=True, what="gemv epilogue")


@pytest.mark.parametrize("B,K_in,K_out,xdt", [(16, 96, 40, torch.bfloat16),
                                              (256, 1024, 1000, torch.bfloat16),
                                              (4, 100, 30, torch.float32),
                                              (9, 64, 64, torch.bfloat16)])
def test_linear_as_conv_matches_oracle(B, K_in, K_out, xdt):
    g = inputs.generator(B + K_in)
    W = inputs.normal((K_out, K_in), 1.1, g)
    x = torch.randn(B, K_in, generator=g).to(xdt)
    y, y_orc, bound = run_linear(W, x, torch.float32)
    assert_within(y, y_orc, bound, out_bf16=False, what="linear-as-conv")


@pytest.mark.parametrize("shape,k,s,pd", [((2, 32, 32, 128), (2, 2), (2, 2), (0, 0)),
                                          ((3, 55, 55, 96), (3, 3), (2, 2), (0, 0)),
                                          ((1, 9, 8, 5), (2, 2), (2, 2), (0, 0)),
                                          ((2, 13, 13, 256), (3, 3), (2, 2), (0, 0)),
                                          ((2, 112, 112, 64), (3, 3), (2, 2), (1, 1)),
                                          ((1, 9, 7, 5), (3, 2), (2, 1), (1, 1))])
@pytest.mark.parametrize("dt", [torch.bfloat16, torch.float32])
def test_maxpool_matches_oracle(shape, k, s, pd, dt):
    g = inputs.generator(sum(shape))
    # shifted down so that every window is negative: a zero pad would win the max
    x = (torch.randn(*shape, generator=g) - 3.0).to(dt)
    y = tbn.tbn_maxpool2d_nhwc(x.cuda(), k, s, pad=pd).float().cpu().numpy()
    want = oracle.maxpool2d_nchw(x.float().permute(0, 3, 1, 2).numpy(), k, s, pd)
    assert np.array_equal(y, want.transpose(0, 2, 3, 1))


@pytest.mark.parametrize("dt", [torch.bfloat16, torch.float32])
def test_nchw_to_nhwc_padding(dt):
    g = inputs.generator(5)
    x = torch.randn(2, 3, 5, 7, generator=g).to(dt)
    y = tbn.tbn_nchw_to_nhwc(x.cuda(), C_pad=8).cpu()
    assert torch.equal(y[..., :3], x.permute(0, 2, 3, 1))
    assert torch.all(y[..., 3:] == 0)


@pytest.mark.parametrize("N,C,H,W,C_pad", [(3, 1, 8, 16, 1), (3, 3, 8, 16, 3), (2, 3, 4, 6, 4),
                                           (2, 2, 8, 8, 5), (3, 3, 8, 16, 8), (1, 7, 16, 8, 7),
                                           (2, 8, 8, 8, 8), (128, 3, 32, 32, 3),
                                           (2, 3, 5, 8, 3)])
def test_nchw_to_nhwc_vector_path(N, C, H, W, C_pad):
    """bf16 with H*W % 8 == 0 takes the 8-pixel vector kernel (C_pad <= 8):
    every element and the zero padding, exactly."""
    g = inputs.generator(N * 100 + C * 10 + C_pad)
    x = torch.randn(N, C, H, W, generator=g).to(torch.bfloat16)
    y = tbn.tbn_nchw_to_nhwc(x.cuda(), C_pad=C_pad).cpu()
    want = torch.zeros(N, H, W, C_pad, dtype=torch.bfloat16)
    want[..., :C] = x.permute(0, 2, 3, 1)
    assert torch.equal(y, want)


def test_device_error_word_is_clear():
    assert tbn.tbn_device_error() == 0


@pytest.mark.parametrize("N,C,H,W,C_pad", [(2, 3, 227, 227, 3), (1, 3, 33, 35, 4), (3, 1, 7, 5, 1),
                                           (2, 5, 31, 33, 12), (1, 3, 3, 3, 16)])
def test_nchw_to_nhwc_tiled_path(N, C, H, W, C_pad):
    """bf16 with H*W % 8 != 0 (AlexNet's 227 x 227 input) or C_pad > 8 takes
    the shared-memory tiled kernel: every element and the zero padding,
    exactly, including images that end inside a tile."""
    g = inputs.generator(N * 1000 + C * 10 + H)
    x = torch.randn(N, C, H, W, generator=g).to(torch.bfloat16)
    y = tbn.tbn_nchw_to_nhwc(x.cuda(), C_pad=C_pad).cpu()
    want = torch.zeros(N, H, W, C_pad, dtype=torch.bfloat16)
    want[..., :C] = x.permute(0, 2, 3, 1)
    assert torch.equal(y, want)


@pytest.mark.parametrize("B,K_in,K_out,relu,res", [(256, 9216, 4096, True, False),
                                                   (256, 4096, 1000, False, False),
                                                   (64, 2048, 300, True, True)])
def test_linear_split_k_matches_oracle(B, K_in, K_out, relu, res):
    """A fully-connected layer whose output tiles leave SMs idle (AlexNet's FC
    layers at batch 256) runs with split K when given the workspace the query
    asks for: every output within the bound, and the same results as the
    unsplit call within the bound (the sum order differs)."""
    ws_bytes = tbn.tbn_linear_workspace_bytes(B, K_in, K_out)
    assert ws_bytes >= 4 * B * K_out * 2      # at least two K ranges of fp32 partial sums
    g = inputs.generator(B + K_in + K_out)
    W = inputs.normal((K_out, K_in), 1.1, g)
    x = torch.randn(B, K_in, generator=g).to(torch.bfloat16)
    r = torch.randn(B, K_out, generator=g).to(torch.bfloat16) if res else None
    codes, alpha = tbn.tbn_quantize_pack(W.cuda())
    ws = torch.full((ws_bytes,), 0xFF, dtype=torch.uint8, device="cuda")   # stale contents
    y = tbn.tbn_linear_fwd_ws(x.cuda(), codes, alpha, K_out, ws, relu=relu,
                              residual=r.cuda() if res else None)
    y1 = tbn.tbn_linear_fwd(x.cuda(), codes, alpha, K_out, relu=relu,
                            residual=r.cuda() if res else None)
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    wt, al = oracle.quantize(W.numpy())
    y_orc, bound = oracle.linear(x.float().numpy(), wt, al)
    want = oracle.epilogue(y_orc, r.float().numpy() if res else None, relu=relu)
    for got, what in ((y, "split K"), (y1, "unsplit")):
        assert_within(got.float().cpu().numpy(), want, bound, out_bf16=True, epilogue=True,
                      what="linear %s %s" % (what, (B, K_in, K_out)))
