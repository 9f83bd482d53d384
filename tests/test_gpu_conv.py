"""GPU parity of tbn_conv2d_fwd (direct and tcgen05 implicit-GEMM kernels)
against the oracle's seven-loop convolution, per output:
|y_gpu - y_orc| <= 2e-3 * |alpha| * sum|x| (fp32 output), plus the bf16
output rounding for bf16 output."""
import zlib

import numpy as np
import pytest
import torch

import paper_1701_00485_gb300 as tbn
from paper_1701_00485_gb300 import inputs
from parity_util import ConvCase, assert_within, random_sites

pytestmark = pytest.mark.gpu


def make_case(N, C, H, W, K, R, S, stride, pad, seed, wscale=None, xdist="normal"):
    g = inputs.generator(seed)
    if xdist == "normal":
        x = torch.randn(N, C, H, W, generator=g)
    else:
        x = torch.rand(N, C, H, W, generator=g)
    std = wscale if wscale is not None else (2.0 / (C * R * S)) ** 0.5
    Wt = inputs.normal((K, C, R, S), std, g)
    return ConvCase(x, Wt, stride, pad)


# ---------------------------------------------------------------- direct kernel
DIRECT = [
    # N, C, H, W, K, R, S, stride, pad
    (2, 3, 9, 7, 5, 3, 3, (1, 1), (1, 1)),
    (1, 1, 28, 28, 20, 5, 5, (1, 1), (0, 0)),
    (3, 4, 11, 10, 33, 5, 5, (2, 2), (2, 2)),
    (2, 8, 6, 6, 7, 1, 1, (1, 1), (0, 0)),
    (1, 3, 23, 23, 40, 11, 11, (4, 4), (0, 0)),
    (1, 5, 9, 7, 3, 3, 1, (1, 2), (0, 1)),
    (2, 70, 5, 5, 65, 3, 3, (1, 1), (1, 1)),
]


@pytest.mark.parametrize("case", DIRECT)
@pytest.mark.parametrize("layout", [tbn.TBN_NCHW, tbn.TBN_NHWC])
@pytest.mark.parametrize("xdt", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("ydt", [torch.float32, torch.bfloat16])
def test_direct_conv_matches_oracle(case, layout, xdt, ydt):
    c = make_case(*case, seed=sum(case[:7]), wscale=1.3)
    y = c.run_gpu(layout, xdt, ydt, algo=tbn.TBN_CONV_DIRECT)
    y_orc, bound = c.oracle_full(xdt)
    assert_within(y, y_orc, bound, out_bf16=(ydt == torch.bfloat16), what="direct %s" % (case,))


def test_lenet_layer_full():
    # the LeNet-like workload: fp32 input U(0,1), W ~ N(0, 0.1), quantize + conv
    x, W = inputs.lenet_inputs(0)
    c = ConvCase(x, W, (1, 1), (0, 0))
    y = c.run_gpu(tbn.TBN_NCHW, torch.float32, torch.float32)
    y_orc, bound = c.oracle_full(torch.float32)
    assert_within(y, y_orc, bound, out_bf16=False, what="lenet")


# ---------------------------------------------------------------- implicit GEMM
IGEMM = [
    # N, C, H, W, K, R, S, stride, pad    (all NHWC bf16, C % 32 == 0, stride <= 2)
    (1, 64, 8, 8, 128, 3, 3, (1, 1), (1, 1)),       # one tile, exact
    (2, 64, 8, 8, 128, 1, 1, (1, 1), (0, 0)),       # 1x1
    (3, 128, 16, 16, 256, 3, 3, (1, 1), (1, 1)),    # two filter tiles
    (2, 64, 32, 32, 128, 3, 3, (1, 1), (1, 1)),     # 32-wide rows, 8-row tiles
    (5, 64, 7, 7, 200, 3, 3, (1, 1), (1, 1)),       # ragged K and image packing
    (3, 64, 13, 13, 96, 3, 3, (1, 1), (1, 1)),      # N = 176 tile, K < 128
    (2, 128, 28, 28, 64, 3, 3, (1, 1), (1, 1)),     # balanced row tiles
    (2, 64, 9, 11, 130, 3, 3, (1, 1), (0, 0)),      # valid conv, odd sizes
    (2, 64, 14, 14, 128, 3, 3, (2, 2), (1, 1)),     # stride 2
    (2, 64, 15, 15, 128, 1, 1, (2, 2), (0, 0)),     # 1x1 stride 2 projection
    (1, 192, 6, 5, 136, 2, 3, (1, 1), (1, 0)),      # R != S, asymmetric pad
    (1, 64, 300, 4, 128, 3, 3, (1, 1), (1, 1)),     # Q < P, tall image
    (1, 64, 3, 300, 128, 3, 3, (1, 1), (1, 1)),     # Q > 256: several q tiles
    # C % 32 == 0, not % 64: two 32-channel boxes per K block (64-byte swizzle)
    (2, 96, 13, 13, 128, 5, 5, (1, 1), (2, 2)),     # AlexNet conv2 taps, n % 64 == 32
    (2, 32, 9, 9, 64, 3, 3, (1, 1), (1, 1)),        # one box per tap, ragged last block
    (2, 160, 8, 8, 128, 1, 1, (1, 1), (0, 0)),      # 1x1, n = 160
    (2, 96, 14, 14, 128, 3, 3, (2, 2), (1, 1)),     # stride 2
    (1, 96, 27, 27, 256, 5, 5, (1, 1), (2, 2)),     # AlexNet conv2 image, two filter tiles
]


@pytest.mark.parametrize("case", IGEMM)
def test_igemm_conv_matches_oracle_fp32_out(case):
    c = make_case(*case, seed=1000 + sum(case[:7]), wscale=1.2)
    algo = tbn.tbn_conv2d_select_algo(torch.bfloat16, tbn.TBN_NHWC, *case[:7], case[7], case[8])
    assert algo == tbn.TBN_CONV_IMPLICIT_GEMM
    y = c.run_gpu(tbn.TBN_NHWC, torch.bfloat16, torch.float32, algo=tbn.TBN_CONV_IMPLICIT_GEMM)
    y_orc, bound = c.oracle_full(torch.bfloat16)
    assert_within(y, y_orc, bound, out_bf16=False, what="igemm %s" % (case,))


GATHER = [
    # C % 32 != 0 (activations gathered by threads) or stride > 2
    (2, 3, 32, 32, 128, 3, 3, (1, 1), (1, 1)),      # VGG first layer shape (C=3)
    (1, 1, 28, 28, 20, 5, 5, (1, 1), (0, 0)),       # C=1
    (1, 3, 35, 35, 96, 11, 11, (4, 4), (0, 0)),     # AlexNet conv1 geometry
    (2, 40, 13, 13, 128, 5, 5, (1, 1), (2, 2)),     # C % 8 == 0, not % 32 (vector gather)
    (2, 5, 9, 7, 70, 3, 3, (1, 1), (1, 1)),         # odd C, ragged K
    (1, 16, 12, 12, 64, 3, 3, (2, 2), (1, 1)),      # stride 2 gathered
    (1, 64, 20, 20, 128, 3, 3, (3, 3), (1, 1)),     # C % 64 == 0 but stride 3
    (3, 24, 6, 6, 40, 1, 1, (1, 1), (0, 0)),        # 1x1, C=24
]


@pytest.mark.parametrize("case", GATHER)
def test_igemm_gather_conv_matches_oracle(case):
    c = make_case(*case, seed=4000 + sum(case[:7]), wscale=1.2)
    algo = tbn.tbn_conv2d_select_algo(torch.bfloat16, tbn.TBN_NHWC, *case[:7], case[7], case[8])
    short = case[1] * case[5] * case[6] <= 64
    assert algo == (tbn.TBN_CONV_SMALL_TAPS if short else tbn.TBN_CONV_IMPLICIT_GEMM)
    y = c.run_gpu(tbn.TBN_NHWC, torch.bfloat16, torch.float32, algo=tbn.TBN_CONV_IMPLICIT_GEMM)
    y_orc, bound = c.oracle_full(torch.bfloat16)
    assert_within(y, y_orc, bound, out_bf16=False, what="gather %s" % (case,))


# ---------------------------------------------------------------- small-tap kernel
SMALLTAP = [
    # N, C, H, W, K, R, S, stride, pad    (bf16 x, C*R*S <= 64)
    (2, 3, 32, 32, 128, 3, 3, (1, 1), (1, 1)),      # VGG first layer geometry, n = 27
    (1, 1, 28, 28, 20, 5, 5, (1, 1), (0, 0)),       # C = 1, 5x5, K < 128
    (2, 7, 10, 9, 200, 3, 3, (1, 1), (1, 1)),       # n = 63 (64-code rows), two filter tiles
    (1, 2, 17, 300, 24, 3, 3, (1, 1), (1, 1)),      # Q > 256: column tiles
    (3, 4, 15, 13, 37, 3, 3, (2, 2), (1, 1)),       # stride 2, odd K
    (1, 16, 9, 9, 64, 2, 2, (1, 1), (0, 0)),        # n = 64 exactly
    (2, 3, 20, 20, 16, 1, 1, (1, 1), (0, 0)),       # 1x1
    (1, 5, 12, 7, 130, 3, 1, (1, 2), (0, 1)),       # R != S, mixed stride / pad
]


@pytest.mark.parametrize("case", SMALLTAP)
@pytest.mark.parametrize("layout", [tbn.TBN_NCHW, tbn.TBN_NHWC])
def test_smalltap_conv_matches_oracle(case, layout):
    c = make_case(*case, seed=6000 + sum(case[:7]), wscale=1.2)
    algo = tbn.tbn_conv2d_select_algo(torch.bfloat16, layout, *case[:7], case[7], case[8])
    assert algo == tbn.TBN_CONV_SMALL_TAPS
    y_orc, bound = c.oracle_full(torch.bfloat16)
    y = c.run_gpu(layout, torch.bfloat16, torch.float32, algo=tbn.TBN_CONV_SMALL_TAPS)
    assert_within(y, y_orc, bound, out_bf16=False, what="smalltap %s" % (case,))
    yb = c.run_gpu(layout, torch.bfloat16, torch.bfloat16, algo=tbn.TBN_CONV_SMALL_TAPS)
    assert_within(yb, y_orc, bound, out_bf16=True, what="smalltap bf16 %s" % (case,))


@pytest.mark.parametrize("case", SMALLTAP[:3])
@pytest.mark.parametrize("layout", [tbn.TBN_NCHW, tbn.TBN_NHWC])
@pytest.mark.parametrize("ydt", [torch.float32, torch.bfloat16])
def test_smalltap_conv_epilogue(case, layout, ydt):
    import oracle
    c = make_case(*case, seed=6500 + sum(case[:7]))
    y_orc, bound = c.oracle_full(torch.bfloat16)
    g = inputs.generator(17)
    res = torch.randn(*y_orc.shape, generator=g).to(ydt)
    want = oracle.epilogue(y_orc, res.float().numpy(), relu=True)
    y = c.run_gpu(layout, torch.bfloat16, ydt, algo=tbn.TBN_CONV_SMALL_TAPS, relu=True,
                  residual=res)
    assert_within(y, want, bound, out_bf16=(ydt == torch.bfloat16), epilogue=True,
                  what="smalltap epi %s" % (case,))


@pytest.mark.parametrize("case", SMALLTAP)
def test_smalltap_nchw_in_nhwc_out_matches_oracle(case):
    """TBN_NCHW_NHWC (NCHW x, NHWC y, codes in (r, s, c) order) on the
    mma.sync small-tap kernel: bf16 and fp32 output, the residual epilogue."""
    c = make_case(*case, seed=6700 + sum(case[:7]), wscale=1.2)
    algo = tbn.tbn_conv2d_select_algo(torch.bfloat16, tbn.TBN_NCHW_NHWC, *case[:7], case[7],
                                      case[8])
    assert algo == tbn.TBN_CONV_SMALL_TAPS
    y_orc, bound = c.oracle_full(torch.bfloat16)
    yb = c.run_gpu(tbn.TBN_NCHW_NHWC, torch.bfloat16, torch.bfloat16)
    assert_within(yb, y_orc, bound, out_bf16=True, what="smalltap nchw->nhwc bf16 %s" % (case,))
    y = c.run_gpu(tbn.TBN_NCHW_NHWC, torch.bfloat16, torch.float32)
    assert_within(y, y_orc, bound, out_bf16=False, what="smalltap nchw->nhwc %s" % (case,))
    import oracle
    g = inputs.generator(99)
    res = torch.randn(*y_orc.shape, generator=g).to(torch.bfloat16)
    want = oracle.epilogue(y_orc, res.float().numpy(), relu=True)
    ye = c.run_gpu(tbn.TBN_NCHW_NHWC, torch.bfloat16, torch.bfloat16, relu=True, residual=res)
    assert_within(ye, want, bound, out_bf16=True, epilogue=True,
                  what="smalltap nchw->nhwc epi %s" % (case,))


@pytest.mark.parametrize("case", DIRECT[:4])
@pytest.mark.parametrize("xdt", [torch.float32, torch.bfloat16])
def test_direct_nchw_in_nhwc_out_matches_oracle(case, xdt):
    c = make_case(*case, seed=7100 + sum(case[:7]), wscale=1.3)
    y = c.run_gpu(tbn.TBN_NCHW_NHWC, xdt, torch.float32, algo=tbn.TBN_CONV_DIRECT)
    y_orc, bound = c.oracle_full(xdt)
    assert_within(y, y_orc, bound, out_bf16=False, what="direct nchw->nhwc %s" % (case,))


def test_nchw_in_nhwc_out_auto_falls_back_to_direct():
    """Long filters with the mixed layout have no tensor-core kernel: AUTO
    takes the direct kernel, the implicit GEMM refuses."""
    case = (2, 8, 9, 9, 24, 3, 3, (1, 1), (1, 1))   # C*R*S = 72
    assert tbn.tbn_conv2d_select_algo(torch.bfloat16, tbn.TBN_NCHW_NHWC, *case[:7], case[7],
                                      case[8]) == tbn.TBN_CONV_DIRECT
    c = make_case(*case, seed=71)
    y_orc, bound = c.oracle_full(torch.bfloat16)
    y = c.run_gpu(tbn.TBN_NCHW_NHWC, torch.bfloat16, torch.bfloat16, relu=True)
    assert_within(y, oracle_relu(y_orc), bound, out_bf16=True, epilogue=True, what="auto mixed")
    with pytest.raises(tbn.TBNError):
        c.run_gpu(tbn.TBN_NCHW_NHWC, torch.bfloat16, torch.bfloat16,
                  algo=tbn.TBN_CONV_IMPLICIT_GEMM)


def oracle_relu(y):
    import oracle
    return oracle.epilogue(y, None, relu=True)


def test_smalltap_rejects_long_filters_and_pool():
    c = make_case(1, 8, 6, 6, 16, 3, 3, (1, 1), (1, 1), seed=5)   # n = 72
    with pytest.raises(tbn.TBNError):
        c.run_gpu(tbn.TBN_NHWC, torch.bfloat16, torch.float32, algo=tbn.TBN_CONV_SMALL_TAPS)
    assert tbn.tbn_conv2d_select_algo(torch.float32, tbn.TBN_NHWC, 1, 3, 8, 8, 16, 3, 3) != \
        tbn.TBN_CONV_SMALL_TAPS


POOL = [
    # N, C, H, W, K, R, S, stride, pad  -> conv + ReLU + 2x2/2 max pool fused
    (2, 64, 32, 32, 128, 3, 3, (1, 1), (1, 1)),     # VGG c2 geometry (8-row tiles)
    (4, 128, 8, 8, 256, 3, 3, (1, 1), (1, 1)),      # several images per tile
    (3, 128, 16, 16, 200, 3, 3, (1, 1), (1, 1)),    # 16-wide rows, ragged K
    (2, 3, 32, 32, 128, 3, 3, (1, 1), (1, 1)),      # gathered activations
    (5, 64, 9, 8, 64, 3, 3, (1, 1), (1, 1)),        # odd P (floor), images per tile
    (2, 96, 16, 16, 128, 3, 3, (1, 1), (1, 1)),     # 32-channel boxes
]
POOL_OTHER = [
    (1, 64, 13, 11, 72, 3, 3, (1, 1), (1, 1)),      # odd P, Q: direct kernel
    (1, 64, 60, 60, 128, 3, 3, (1, 1), (1, 1)),     # 60-wide rows: direct kernel
]


def _pooled_oracle(c, x_dtype):
    import oracle
    y, bound = c.oracle_full(x_dtype)
    y = oracle.epilogue(y, None, relu=True)
    P2, Q2 = y.shape[2] // 2, y.shape[3] // 2
    yp = oracle.maxpool2d_nchw(y, (2, 2), (2, 2))
    # the tolerance of a pooled output: the largest bound in its window
    bw = bound[:, :, :2 * P2, :2 * Q2].reshape(bound.shape[0], bound.shape[1], P2, 2, Q2, 2)
    return yp, bw.max(axis=(3, 5))


def _run_pooled(c, layout, x_dtype, y_dtype, algo):
    Wl, codes, alpha = c.quantize_gpu(layout)
    x = c.x.to(x_dtype)
    if layout == tbn.TBN_NHWC:
        x = x.permute(0, 2, 3, 1).contiguous()
    y = tbn.tbn_conv2d_fwd(x.cuda(), codes, alpha, c.K, c.R, c.S, c.stride, c.pad, layout=layout,
                           out_dtype=y_dtype, relu=True, pool=2, algo=algo)
    y = y.float().cpu()
    if layout == tbn.TBN_NHWC:
        y = y.permute(0, 3, 1, 2)
    return y.numpy()


@pytest.mark.parametrize("case", POOL)
@pytest.mark.parametrize("algo", [tbn.TBN_CONV_IMPLICIT_GEMM, tbn.TBN_CONV_DIRECT])
def test_fused_relu_pool_matches_oracle(case, algo):
    c = make_case(*case, seed=5000 + sum(case[:7]))
    want, bound = _pooled_oracle(c, torch.bfloat16)
    y = _run_pooled(c, tbn.TBN_NHWC, torch.bfloat16, torch.float32, algo)
    assert y.shape == want.shape
    assert_within(y, want, bound, out_bf16=False, epilogue=True, what="pool %s" % (case,))
    yb = _run_pooled(c, tbn.TBN_NHWC, torch.bfloat16, torch.bfloat16, algo)
    assert_within(yb, want, bound, out_bf16=True, epilogue=True, what="pool bf16 %s" % (case,))


@pytest.mark.parametrize("case", POOL_OTHER)
def test_fused_pool_other_widths_auto(case):
    c = make_case(*case, seed=5100 + sum(case[:7]))
    want, bound = _pooled_oracle(c, torch.bfloat16)
    y = _run_pooled(c, tbn.TBN_NHWC, torch.bfloat16, torch.float32, tbn.TBN_CONV_AUTO)
    assert_within(y, want, bound, out_bf16=False, epilogue=True, what="pool auto %s" % (case,))
    with pytest.raises(tbn.TBNError):
        _run_pooled(c, tbn.TBN_NHWC, torch.bfloat16, torch.float32, tbn.TBN_CONV_IMPLICIT_GEMM)


@pytest.mark.parametrize("case", IGEMM[3:6] + GATHER[:2])
def test_igemm_persistent_many_tiles_per_cta(case):
    """Batches large enough that every CTA of the persistent kernel walks
    several tiles (accumulator reuse across tiles)."""
    N = case[0] * 40
    c = make_case(N, *case[1:], seed=6000 + sum(case[:7]))
    y = c.run_gpu(tbn.TBN_NHWC, torch.bfloat16, torch.bfloat16, algo=tbn.TBN_CONV_IMPLICIT_GEMM)
    sites = random_sites(y.shape, 4000, seed=N)
    y_orc, bound = c.oracle_sites(torch.bfloat16, sites)
    assert_within(y[tuple(sites.T)], y_orc, bound, out_bf16=True, what="persistent %s" % (case,))


def test_fused_pool_nchw_direct():
    c = make_case(2, 3, 10, 12, 9, 3, 3, (1, 1), (1, 1), seed=77)
    want, bound = _pooled_oracle(c, torch.float32)
    y = _run_pooled(c, tbn.TBN_NCHW, torch.float32, torch.float32, tbn.TBN_CONV_DIRECT)
    assert_within(y, want, bound, out_bf16=False, epilogue=True, what="pool nchw")


@pytest.mark.parametrize("case", IGEMM[:6])
def test_igemm_conv_bf16_out_and_epilogue(case):
    c = make_case(*case, seed=2000 + sum(case[:7]))
    y_orc, bound = c.oracle_full(torch.bfloat16)
    y = c.run_gpu(tbn.TBN_NHWC, torch.bfloat16, torch.bfloat16, algo=tbn.TBN_CONV_IMPLICIT_GEMM)
    assert_within(y, y_orc, bound, out_bf16=True, what="igemm bf16 %s" % (case,))
    # fused residual + ReLU, checked against the oracle's epilogue
    import oracle
    g = inputs.generator(7)
    res = torch.randn(*y_orc.shape, generator=g).to(torch.bfloat16)
    want = oracle.epilogue(y_orc, res.float().numpy(), relu=True)
    y2 = c.run_gpu(tbn.TBN_NHWC, torch.bfloat16, torch.bfloat16, algo=tbn.TBN_CONV_IMPLICIT_GEMM,
                   relu=True, residual=res)
    assert_within(y2, want, bound, out_bf16=True, epilogue=True, what="igemm epi %s" % (case,))


@pytest.mark.parametrize("case", IGEMM[2:5])
def test_igemm_equals_direct_kernel(case):
    c = make_case(*case, seed=3000 + sum(case[:7]))
    y1 = c.run_gpu(tbn.TBN_NHWC, torch.bfloat16, torch.float32, algo=tbn.TBN_CONV_IMPLICIT_GEMM)
    y2 = c.run_gpu(tbn.TBN_NHWC, torch.bfloat16, torch.float32, algo=tbn.TBN_CONV_DIRECT)
    _, bound = c.oracle_full(torch.bfloat16)
    assert np.all(np.abs(y1 - y2) <= 4e-3 * bound + 1e-30)


# ------------------------------------------------------ workload layers, full size
def _workload_layers():
    out = []
    for i, s in enumerate(inputs.VGG_SMALL["convs"]):
        hw = 32 >> (i // 2)
        out.append(("vgg_c%d" % (i + 1), 128, s, hw))
    a = inputs.ALEXNET["convs"]
    out += [("alex_conv1", 256, a[0], 227), ("alex_conv2", 256, a[1], 27),
            ("alex_conv3", 256, a[2], 13), ("alex_conv4", 256, a[3], 13),
            ("alex_conv5", 256, a[4], 13)]
    # input size of each ResNet-18 conv (224 -> stem /2 -> pool /2 = 56)
    stage_hw = {"l1": 56, "l2": 28, "l3": 14, "l4": 7}
    prev_hw = {"l1": 56, "l2": 56, "l3": 28, "l4": 14}
    for name, s in inputs.resnet18_convs():
        stage = name[:2]
        h = prev_hw[stage] if (s.stride == 2) else stage_hw[stage]
        out.append(("resnet_" + name, 128, s, h))
    return out


WORKLOAD = _workload_layers()


@pytest.mark.parametrize("name,N,spec,hw", WORKLOAD, ids=[w[0] for w in WORKLOAD])
def test_workload_layer_sampled(name, N, spec, hw):
    """Each conv layer of the VGG-small / AlexNet / ResNet-18 workloads at its
    full batch and size, in the launch configuration the networks use
    (NHWC bf16 in, bf16 out, AUTO algorithm), checked at sampled outputs."""
    g = inputs.generator(zlib.crc32(name.encode()) % 100000)
    x = torch.randn(N, spec.C, hw, hw, generator=g).to(torch.bfloat16)
    W = inputs.he_normal(spec.K, spec.C, spec.R, spec.S, g)
    c = ConvCase(x, W, (spec.stride, spec.stride), (spec.pad, spec.pad))
    y = c.run_gpu(tbn.TBN_NHWC, torch.bfloat16, torch.bfloat16)
    sites = random_sites(y.shape, 3000, seed=len(name))
    y_orc, bound = c.oracle_sites(torch.bfloat16, sites)
    assert_within(y[tuple(sites.T)], y_orc, bound, out_bf16=True, what=name)
