"""The network forward (re-quantization, input layout change, convolutions
with fused epilogues, run eagerly and from a captured CUDA graph) gives
bitwise the outputs of the same library calls issued one by one, and its
first layer matches the oracle."""
import numpy as np
import pytest
import torch

import oracle
import paper_1701_00485_gb300 as tbn
from paper_1701_00485_gb300 import inputs, nets
from parity_util import assert_within

pytestmark = pytest.mark.gpu


def sequential_forward(net):
    """Every launch of the forward on the current stream, in order."""
    net.quantize()
    tbn.tbn_nchw_to_nhwc(net.x_in, out=net.x_nhwc)
    h = net.x_nhwc
    for l in net.layers:
        s = l.spec
        tbn.tbn_conv2d_fwd(h, l.codes, l.alpha, s.K, s.R, s.S, (s.stride, s.stride),
                           (s.pad, s.pad), layout=tbn.TBN_NHWC, relu=s.relu, out=l.y,
                           pool=2 if s.pool == (2, 2) else 0)
        h = l.y
        if l.pooled is not None:
            k, st = s.pool
            tbn.tbn_maxpool2d_nhwc(h, (k, k), (st, st), out=l.pooled)
            h = l.pooled
    return h


def test_forward_matches_sequential_launches():
    net = nets.vgg_small(batch=8)
    ref = sequential_forward(net).clone()
    firsts = [l.y.clone() for l in net.layers]
    for l in net.layers:
        l.y.zero_()
        l.codes.zero_()
    out = net.forward(requantize=True)
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    assert torch.equal(out, ref)
    for l, y0 in zip(net.layers, firsts):
        assert torch.equal(l.y, y0)
    # captured in a graph and replayed, still the same
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        net.forward(requantize=True)
        torch.cuda.synchronize()
        with torch.cuda.graph(g, stream=s):
            net.forward(requantize=True)
    for _ in range(2):
        net.layers[-1].y.zero_()
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(net.out, ref)


def test_network_first_layer_matches_oracle():
    net = nets.vgg_small(batch=2)
    net.forward(requantize=True)
    torch.cuda.synchronize()
    l = net.layers[0]
    K, n = l.W.shape
    s = l.spec
    W_kcrs = l.W.cpu().reshape(K, s.R, s.S, s.C).permute(0, 3, 1, 2).contiguous()
    wt, al = oracle.quantize(W_kcrs.reshape(K, -1).numpy())
    y_orc, bound = oracle.conv2d_nchw(net.x_in.float().cpu().numpy(),
                                      wt.reshape(K, s.C, s.R, s.S), al, (s.stride, s.stride),
                                      (s.pad, s.pad))
    y_orc = oracle.epilogue(y_orc, None, relu=True)   # the layer's fused ReLU
    y = l.y.float().cpu().permute(0, 3, 1, 2).numpy()
    assert_within(y, y_orc, bound, out_bf16=True, epilogue=True, what="network c1")
