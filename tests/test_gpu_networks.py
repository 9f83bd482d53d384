"""Full-size network forwards (AlexNet b256, ResNet-18 b128), checked layer by
layer against the oracle on each layer's actual input.

Multi-layer workloads compound their errors and carry glue the paper does
not define, so parity is per layer: the oracle takes the bf16 tensor the GPU
fed to that layer (exact in fp64), quantizes the same fp32 weights (codes
bit-exact, alpha within 1e-6 relative) and computes the layer; the GPU output
must lie within the benchmark spec's bound 2e-3 * |alpha| * sum|x| plus the bf16
rounding of the output (and 2^-22 |y| for a fused residual / ReLU).
Convolutions are compared at sampled output sites (plus the corners), the
fully-connected layers at every output, max pools and the layer wiring
exactly.  The full-precision ResNet-18 stem, average pool and FC use the
fp32 tolerance of test_gpu_dense_repack.py.
"""
import zlib

import numpy as np
import pytest
import torch

import oracle
import paper_1701_00485_gb300 as tbn
from paper_1701_00485_gb300 import nets
from parity_util import assert_within, check_quantize, random_sites

pytestmark = pytest.mark.gpu

U = 2.0 ** -24


def _nchw(t: torch.Tensor) -> np.ndarray:
    return t.float().permute(0, 3, 1, 2).contiguous().cpu().numpy()


def _kcrs(W_rsc: torch.Tensor, spec) -> np.ndarray:
    """fp32 weights stored (r, s, c)-ordered back in [K, C, R, S]."""
    K = W_rsc.shape[0]
    return W_rsc.cpu().reshape(K, spec.R, spec.S, spec.C).permute(0, 3, 1, 2).contiguous().numpy()


def _check_conv_sites(name, x_nhwc, W_rsc, codes, alpha, spec, y_nhwc, residual=None,
                      relu=True, count=2000):
    """One two-bit convolution of a network at sampled sites of its output."""
    check_quantize(W_rsc.cpu(), codes, alpha)
    Wk = _kcrs(W_rsc, spec)
    wt, al = oracle.quantize(Wk.reshape(spec.K, -1))
    y = _nchw(y_nhwc)
    sites = random_sites(y.shape, count, seed=zlib.crc32(name.encode()) % 100000)
    y_orc, bound = oracle.conv2d_sites(_nchw(x_nhwc), wt.reshape(Wk.shape), al, sites,
                                       (spec.stride,) * 2, (spec.pad,) * 2)
    res = None
    if residual is not None:
        res = _nchw(residual)[tuple(sites.T)]
    want = oracle.epilogue(y_orc, res, relu=relu)
    assert_within(y[tuple(sites.T)], want, bound, out_bf16=True, epilogue=True, what=name)


@pytest.fixture(scope="module")
def alexnet():
    net = nets.alexnet()
    net.forward(requantize=True)
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    return net


def test_alexnet_b256_conv_layers(alexnet):
    net = alexnet
    # conv1 runs on the space-to-depth form of the input; the oracle sees
    # the original input
    assert net.features.s2d
    h = net.x_in.permute(0, 2, 3, 1).contiguous()
    for i, l in enumerate(net.features.layers):
        _check_conv_sites("alexnet conv%d" % (i + 1), h, l.W, l.codes, l.alpha, l.spec, l.y)
        h = l.y
        if l.pooled is not None:
            k, st = l.spec.pool
            want = oracle.maxpool2d_nchw(_nchw(l.y), (k, k), (st, st))
            assert np.array_equal(_nchw(l.pooled), want), "alexnet pool after conv%d" % (i + 1)
            h = l.pooled
    assert tuple(h.shape) == (256, 6, 6, 256)


def test_alexnet_b256_fc_layers(alexnet):
    """FC 9216-4096-4096-1000 at batch 256, every output, each on the GPU's
    own input (the NHWC flattening of the last pooled map for fc6)."""
    net = alexnet
    h = net.features.out.reshape(net.N, -1)
    assert h.shape == (256, 9216)
    for i, (W, codes, alpha, relu, y) in enumerate(net.classifier.layers):
        check_quantize(W.cpu(), codes, alpha)
        wt, al = oracle.quantize(W.cpu().numpy())
        y_orc, bound = oracle.linear(h.float().cpu().numpy(), wt, al)
        want = oracle.epilogue(y_orc, None, relu=relu)
        assert_within(y.float().cpu().numpy(), want, bound, out_bf16=True, epilogue=True,
                      what="alexnet fc%d" % (i + 6))
        h = y
    assert net.out.shape == (256, 1000)


def test_alexnet_graph_replay_is_bitwise_stable(alexnet):
    net = alexnet
    ref = net.out.clone()
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        net.forward(requantize=True)
        torch.cuda.synchronize()
        with torch.cuda.graph(g, stream=s):
            net.forward(requantize=True)
    net.out.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(net.out, ref)


@pytest.fixture(scope="module")
def resnet():
    net = nets.resnet18()
    net.forward(requantize=True)
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    return net


def test_resnet18_b128_stem_and_pool(resnet):
    """fp32 7x7/2 first convolution (ReLU, bf16 out) on three whole images, and
    the 3x3/2 pad-1 max pool exactly."""
    net = resnet
    imgs = [0, 77, 127]
    x = net.x_in[imgs].float().cpu().numpy()
    want, bound = oracle.dense_conv2d_nchw(x, net.stem_w.cpu().numpy(), (2, 2), (3, 3))
    want = np.maximum(want, 0.0)
    got = _nchw(net.stem_y[imgs])
    tol = 3 * 49 * U * bound + 2.0 ** -8 * np.abs(want)
    assert np.all(np.abs(got - want) <= tol), float(np.max(np.abs(got - want) - tol))
    pooled = oracle.maxpool2d_nchw(_nchw(net.stem_y), (3, 3), (2, 2), (1, 1))
    assert np.array_equal(_nchw(net.pool_y), pooled)


def test_resnet18_b128_basic_blocks(resnet):
    """Every two-bit convolution of the eight basic blocks on its own input:
    a (3x3, ReLU), the 1x1/2 projection d (no ReLU) and b (3x3 + shortcut,
    then ReLU; the shortcut is d's output or the block input)."""
    net = resnet
    h = net.pool_y
    for a, b, d in net.blocks:
        _check_conv_sites("resnet " + a.name, h, a.W, a.codes, a.alpha, a.spec, a.y)
        if d is not None:
            _check_conv_sites("resnet " + d.name, h, d.W, d.codes, d.alpha, d.spec, d.y,
                              relu=False)
        res = d.y if d is not None else h
        _check_conv_sites("resnet " + b.name, a.y, b.W, b.codes, b.alpha, b.spec, b.y,
                          residual=res, relu=True)
        h = b.y
    assert tuple(h.shape) == (128, 7, 7, 512)


def test_resnet18_b128_head(resnet):
    """Global average pool and the fp32 FC 512 -> 1000, every output."""
    net = resnet
    last = net.blocks[-1][1].y
    want = oracle.avgpool_global_nchw(_nchw(last))
    mag = np.abs(last.float().cpu().numpy()).mean(axis=(1, 2))
    tol = 49 * U * mag + U * np.abs(want)
    assert np.all(np.abs(net.feat.cpu().numpy().astype(np.float64) - want) <= tol)
    y, bound = oracle.dense_linear(net.feat.cpu().numpy(), net.fc_w.cpu().numpy())
    assert np.all(np.abs(net.logits.cpu().numpy().astype(np.float64) - y) <= 512 * U * bound)
