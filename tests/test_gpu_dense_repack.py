"""GPU parity of the canonical <-> byte-planar repack and of the
full-precision layers a network keeps around its two-bit layers (the
ResNet-18 first convolution, global average pool and last FC), against the
oracle.

Tolerances of the full-precision layers (fp32 products, fp32 sums of n
terms; the oracle is exact to fp64):
  |y - y_oracle| <= n * 2^-24 * bound + (bf16 output: 2^-8 |y_oracle|)
with bound = sum of |x * w| over the n terms (the classical worst case of an
n-term fp32 sum, n u with u = 2^-24); the average pool adds its one scaling
rounding, 2^-24 |y|.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_1701_00485_gb300 as tbn
from paper_1701_00485_gb300 import inputs
from parity_util import u32

pytestmark = pytest.mark.gpu

U = 2.0 ** -24


@pytest.mark.parametrize("K,n", [(1, 8), (3, 4), (5, 17), (96, 363), (64, 2400), (7, 16384)])
def test_repack_matches_oracle_layouts(K, n):
    rng = np.random.default_rng(K * 1000 + n)
    codes = rng.choice(np.array([-2, -1, 1, 2], dtype=np.int8), size=(K, n))
    planar = oracle.pack(codes)
    canon = oracle.pack_canonical(codes)
    p_gpu = torch.from_numpy(planar.view(np.int32)).cuda()
    c_gpu = torch.from_numpy(canon.view(np.int32)).cuda()
    got_c = tbn.tbn_repack(p_gpu, n, tbn.TBN_REPACK_PLANAR_TO_CANONICAL)
    got_p = tbn.tbn_repack(c_gpu, n, tbn.TBN_REPACK_CANONICAL_TO_PLANAR)
    torch.cuda.synchronize()
    assert np.array_equal(u32(got_c), canon)
    assert np.array_equal(u32(got_p), planar)
    # in place, both ways
    t = p_gpu.clone()
    tbn.tbn_repack(t, n, tbn.TBN_REPACK_PLANAR_TO_CANONICAL, out=t)
    tbn.tbn_repack(t, n, tbn.TBN_REPACK_CANONICAL_TO_PLANAR, out=t)
    torch.cuda.synchronize()
    assert torch.equal(t, p_gpu)


def test_repack_worked_example_words():
    """The hand-derived words of the worked example: 0x03080309 byte-planar,
    0x000050AB canonical."""
    W = torch.tensor([[-1.5, -1.0, -0.25, 0.0, 0.5, 1.0, 1.25, 3.0]], device="cuda")
    codes, _ = tbn.tbn_quantize_pack(W)
    canon = tbn.tbn_repack(codes, 8, tbn.TBN_REPACK_PLANAR_TO_CANONICAL)
    torch.cuda.synchronize()
    assert int(u32(codes)[0, 0]) == 0x03080309
    assert int(u32(canon)[0, 0]) == 0x000050AB


def test_quantize_then_canonical_equals_oracle_canonical():
    W = inputs.scaled_weights((33, 300), 71)
    codes, _ = tbn.tbn_quantize_pack(W.cuda())
    canon = tbn.tbn_repack(codes, 300, tbn.TBN_REPACK_PLANAR_TO_CANONICAL)
    torch.cuda.synchronize()
    wt, _ = oracle.quantize(W.numpy())
    assert np.array_equal(u32(canon), oracle.pack_canonical(wt))


DENSE_CASES = [
    # N, C, H, W, K, R, S, stride, pad, layout
    (2, 3, 37, 35, 64, 7, 7, (2, 2), (3, 3), tbn.TBN_NCHW_NHWC),
    (1, 5, 9, 40, 70, 3, 3, (1, 1), (1, 1), tbn.TBN_NCHW),
    (2, 8, 11, 12, 16, 3, 2, (2, 1), (0, 1), tbn.TBN_NHWC),
    (1, 3, 6, 6, 4, 1, 1, (1, 1), (0, 0), tbn.TBN_NCHW_NHWC),
]


@pytest.mark.parametrize("case", DENSE_CASES)
@pytest.mark.parametrize("xdt,ydt", [(torch.bfloat16, torch.bfloat16),
                                     (torch.float32, torch.float32)])
def test_dense_conv_matches_oracle(case, xdt, ydt):
    N, C, H, W, K, R, S, st, pd, layout = case
    g = inputs.generator(N * 1000 + C * 100 + K)
    x = torch.randn(N, C, H, W, generator=g).to(xdt)
    w = inputs.he_normal(K, C, R, S, g)
    xin = x.permute(0, 2, 3, 1).contiguous() if layout == tbn.TBN_NHWC else x
    for relu in (False, True):
        y = tbn.tbn_dense_conv2d_fwd(xin.cuda(), w.cuda(), st, pd, layout=layout, out_dtype=ydt,
                                     relu=relu)
        torch.cuda.synchronize()
        y = y.float().cpu()
        if layout != tbn.TBN_NCHW:
            y = y.permute(0, 3, 1, 2)
        want, bound = oracle.dense_conv2d_nchw(x.float().numpy(), w.numpy(), st, pd)
        if relu:
            want = np.maximum(want, 0.0)
        tol = C * R * S * U * bound
        if ydt == torch.bfloat16:
            tol = tol + 2.0 ** -8 * np.abs(want)
        err = np.abs(y.numpy().astype(np.float64) - want)
        assert np.all(err <= tol), float(np.max(err - tol))


@pytest.mark.parametrize("N,H,W,C", [(2, 7, 7, 512), (3, 5, 4, 33), (1, 1, 1, 8)])
@pytest.mark.parametrize("xdt", [torch.bfloat16, torch.float32])
def test_global_avgpool_matches_oracle(N, H, W, C, xdt):
    g = inputs.generator(N + H + C)
    x = torch.randn(N, H, W, C, generator=g).to(xdt)
    y = tbn.tbn_avgpool2d_global_nhwc(x.cuda())
    torch.cuda.synchronize()
    want = oracle.avgpool_global_nchw(x.float().permute(0, 3, 1, 2).numpy())
    mag = np.abs(x.float().numpy()).mean(axis=(1, 2))
    tol = H * W * U * mag + U * np.abs(want)
    assert np.all(np.abs(y.cpu().numpy().astype(np.float64) - want) <= tol)


@pytest.mark.parametrize("B,K_in,K_out", [(128, 512, 1000), (3, 37, 65), (70, 100, 9)])
def test_dense_linear_matches_oracle(B, K_in, K_out):
    g = inputs.generator(B + K_in + K_out)
    x = torch.randn(B, K_in, generator=g)
    w = inputs.he_normal(K_out, K_in, 1, 1, g).reshape(K_out, K_in)
    for relu, ydt in ((False, torch.float32), (True, torch.bfloat16)):
        y = tbn.tbn_dense_linear_fwd(x.cuda(), w.cuda(), out_dtype=ydt, relu=relu)
        torch.cuda.synchronize()
        want, bound = oracle.dense_linear(x.numpy(), w.numpy())
        if relu:
            want = np.maximum(want, 0.0)
        tol = K_in * U * bound
        if ydt == torch.bfloat16:
            tol = tol + 2.0 ** -8 * np.abs(want)
        assert np.all(np.abs(y.float().cpu().numpy().astype(np.float64) - want) <= tol)
