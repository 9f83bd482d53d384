"""Two-bit network forward passes built from the C-ABI calls: VGG-small,
AlexNet and ResNet-18 shaped networks.

A network object owns its device buffers (fp32 real-valued weights, packed
codes, alpha, activations) so that one forward pass is a fixed sequence of
library launches on one stream -- capturable in a CUDA graph.  Weights are
kept as real values and re-quantized at every forward (Algorithm 1: the
quantization loop runs before TwoBitForward), with one grouped
tbn_quantize_pack_group launch for all layers; ``requantize=False`` runs the
inference form (codes + alpha only, Section 3).

Activations are NHWC bf16 between layers; the input batch arrives NCHW and
is converted by tbn_nchw_to_nhwc, or, for a strided first layer over few
channels (AlexNet's 11x11/4), by tbn_space_to_depth into the input of that
layer's space-to-depth convolution.  Weights of an NHWC layer are packed in
(r, s, c) order: the fp32 [K, C, R, S] weights are permuted once at build
time (quantization is elementwise and alpha is order-independent).
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

from . import (TBN_NCHW, TBN_NHWC, TBN_NCHW_NHWC, TBN_S2D_NHWC, tbn_conv2d_fwd,
               tbn_space_to_depth, space_to_depth_shape, tbn_linear_fwd_ws,
               tbn_linear_workspace_bytes, tbn_maxpool2d_nhwc,
               tbn_nchw_to_nhwc, tbn_quantize_pack_group, tbn_dense_conv2d_fwd,
               tbn_avgpool2d_global_nhwc, tbn_dense_linear_fwd, packed_words, conv_out_hw)
from . import inputs as _inputs


@dataclass
class ConvLayer:
    spec: _inputs.ConvSpec
    W: torch.Tensor          # fp32 [K, R*S*C] in (r, s, c) order, device
    codes: torch.Tensor      # int32 [K, ceil(n/16)]
    alpha: torch.Tensor      # fp32 [K]
    in_hw: tuple
    out_hw: tuple
    y: torch.Tensor          # NHWC bf16 output
    pooled: torch.Tensor | None

    @property
    def flops_per_image(self) -> int:
        s = self.spec
        return 2 * s.K * self.out_hw[0] * self.out_hw[1] * s.C * s.R * s.S


class ConvStack:
    """A chain of TBN conv layers (ReLU and max pooling fused/glued as the
    specs say), e.g. the VGG-small and AlexNet feature extractors."""

    def __init__(self, specs, x_nchw: torch.Tensor, weights, device="cuda"):
        self.device = torch.device(device)
        N, C, H, W = x_nchw.shape
        self.N = N
        self.x_in = x_nchw.to(self.device).contiguous()
        self.in_chw = (C, H, W)
        s0 = specs[0]
        # a strided first layer over few channels runs on its space-to-depth
        # input (the implicit GEMM with the filter resident in tensor memory)
        # instead of an NHWC copy of the input
        self.s2d = (self.x_in.dtype == torch.bfloat16 and s0.stride >= 2 and
                    s0.stride * s0.stride * C <= 64 and s0.K <= 128 and s0.pool != (2, 2) and
                    -(-s0.R // s0.stride) * -(-s0.S // s0.stride) <= 9)
        if self.s2d:
            self.x_s2d = torch.empty(space_to_depth_shape(N, C, H, W, s0.R, s0.S,
                                                          (s0.stride,) * 2, (s0.pad,) * 2),
                                     dtype=torch.bfloat16, device=self.device)
        else:
            self.x_nhwc = torch.empty((N, H, W, C), dtype=torch.bfloat16, device=self.device)
        self.layers = []
        hw = (H, W)
        for spec, Wt in zip(specs, weights):
            K, Cc, R, S = Wt.shape
            assert (K, Cc, R, S) == (spec.K, spec.C, spec.R, spec.S)
            Wl = Wt.permute(0, 2, 3, 1).reshape(K, -1).contiguous().to(self.device)
            n = Wl.shape[1]
            codes = torch.empty((K, packed_words(n)), dtype=torch.int32, device=self.device)
            alpha = torch.empty((K,), dtype=torch.float32, device=self.device)
            ohw = conv_out_hw(hw[0], hw[1], R, S, (spec.stride, spec.stride), (spec.pad, spec.pad))
            pooled = None
            nhw = ohw
            fused = spec.pool == (2, 2)
            if spec.pool is not None:
                k, st = spec.pool
                nhw = ((ohw[0] - k) // st + 1, (ohw[1] - k) // st + 1)
            if fused:
                # 2x2/2 max pool fused into the convolution's epilogue
                y = torch.empty((N, nhw[0], nhw[1], K), dtype=torch.bfloat16, device=self.device)
            else:
                y = torch.empty((N, ohw[0], ohw[1], K), dtype=torch.bfloat16, device=self.device)
                if spec.pool is not None:
                    pooled = torch.empty((N, nhw[0], nhw[1], K), dtype=torch.bfloat16,
                                         device=self.device)
            self.layers.append(ConvLayer(spec, Wl, codes, alpha, hw, ohw, y, pooled))
            hw = nhw
        last = self.layers[-1]
        self.out = last.pooled if last.pooled is not None else last.y

    @property
    def flops(self) -> int:
        """Algorithmic flops of the TBN convolutions for one batch."""
        return self.N * sum(l.flops_per_image for l in self.layers)

    def quantize(self):
        jobs = [(l.W, l.codes, l.alpha) for l in self.layers]
        for i in range(0, len(jobs), 16):
            tbn_quantize_pack_group(jobs[i:i + 16])

    def forward(self, requantize: bool = True, conv_hook=None):
        """One forward pass on the current stream; returns the output tensor.
        conv_hook(i, layer, when) is called before/after each conv launch, and
        once as conv_hook(-1, None, "quantized") after the re-quantization
        (used by the benchmark to record timing events)."""
        if requantize:
            self.quantize()
        if conv_hook:
            conv_hook(-1, None, "quantized")
        if self.s2d:
            s0 = self.layers[0].spec
            tbn_space_to_depth(self.x_in, s0.R, s0.S, (s0.stride,) * 2, (s0.pad,) * 2,
                               layout=TBN_NCHW, out=self.x_s2d)
            h = self.x_s2d
        else:
            tbn_nchw_to_nhwc(self.x_in, out=self.x_nhwc)
            h = self.x_nhwc
        for i, l in enumerate(self.layers):
            s = l.spec
            if conv_hook:
                conv_hook(i, l, "before")
            s2d = i == 0 and self.s2d
            tbn_conv2d_fwd(h, l.codes, l.alpha, s.K, s.R, s.S, (s.stride, s.stride),
                           (s.pad, s.pad), layout=TBN_S2D_NHWC if s2d else TBN_NHWC,
                           relu=s.relu, out=l.y, pool=2 if s.pool == (2, 2) else 0,
                           in_chw=self.in_chw if s2d else None)
            if conv_hook:
                conv_hook(i, l, "after")
            h = l.y
            if l.pooled is not None:
                k, st = s.pool
                tbn_maxpool2d_nhwc(h, (k, k), (st, st), out=l.pooled)
                h = l.pooled
        return h

    def launches_per_forward(self, requantize: bool = True) -> int:
        # the input layout change, one launch per conv, one per pool that is not fused
        n = 1 + len(self.layers) + sum(1 for l in self.layers if l.pooled is not None)
        if requantize:
            n += (len(self.layers) + 15) // 16
        return n


def vgg_small(batch: int | None = None, seed: int = 1, device="cuda") -> ConvStack:
    x, Ws = _inputs.vgg_small_inputs(seed, batch)
    return ConvStack(_inputs.VGG_SMALL["convs"], x, Ws, device)


class FCStack:
    """Fully-connected TBN layers (Section 3), ReLU between them.  One device
    workspace, sized by tbn_linear_workspace_bytes for the largest layer and
    shared by all (they run one after another on the stream), lets a layer
    whose output tiles leave SMs idle split its K dimension over them."""

    def __init__(self, fcs, weights, batch, device="cuda"):
        self.device = torch.device(device)
        self.layers = []
        self.launches = 0
        ws = 0
        for (kin, kout, relu), W in zip(fcs, weights):
            W = W.contiguous().to(self.device)
            codes = torch.empty((kout, packed_words(kin)), dtype=torch.int32, device=self.device)
            alpha = torch.empty((kout,), dtype=torch.float32, device=self.device)
            y = torch.empty((batch, kout), dtype=torch.bfloat16, device=self.device)
            self.layers.append((W, codes, alpha, relu, y))
            need = tbn_linear_workspace_bytes(batch, kin, kout)
            self.launches += 2 if need > 0 else 1     # split K adds the ordered sum
            ws = max(ws, need)
        self.workspace = (torch.empty(ws, dtype=torch.uint8, device=self.device)
                          if ws > 0 else None)

    def quantize(self):
        tbn_quantize_pack_group([(W, c, a) for (W, c, a, _, _) in self.layers])

    def forward(self, x, requantize: bool = False):
        if requantize:
            self.quantize()
        h = x
        for (W, codes, alpha, relu, y) in self.layers:
            tbn_linear_fwd_ws(h, codes, alpha, codes.shape[0], self.workspace, relu=relu, out=y)
            h = y
        return h

    @property
    def flops_per_image(self) -> int:
        return sum(2 * codes.shape[0] * W.shape[1] for (W, codes, _, _, _) in self.layers)


def _quantize_all(jobs):
    for i in range(0, len(jobs), 16):
        tbn_quantize_pack_group(jobs[i:i + 16])


class AlexNet:
    """AlexNet-shaped TBN network (every convolution and fully-connected
    layer two-bit, per-output-neuron alpha): the conv stack with 3x3/2 max
    pools, the NHWC flattening of the last pooled map, FC 9216-4096-4096-1000
    with ReLU between them."""

    def __init__(self, batch: int | None = None, seed: int = 2, device="cuda"):
        x, Ws, Wfc = _inputs.alexnet_inputs(seed, batch)
        self.features = ConvStack(_inputs.ALEXNET["convs"], x, Ws, device)
        self.N = self.features.N
        self.classifier = FCStack(_inputs.ALEXNET["fcs"], Wfc, self.N, device)
        self.x_in = self.features.x_in
        self.out = self.classifier.layers[-1][4]
        # re-quantization runs beside the input's layout change (both read
        # HBM, neither fills it; only the first convolution needs both)
        self.quant_stream = torch.cuda.Stream(device=self.features.device)

    @property
    def conv_flops(self) -> int:
        return self.features.flops

    @property
    def fc_flops(self) -> int:
        return self.N * self.classifier.flops_per_image

    @property
    def flops(self) -> int:
        """Algorithmic flops of all TBN layers (convolutions and FC) per batch."""
        return self.conv_flops + self.fc_flops

    def quantize(self):
        _quantize_all([(l.W, l.codes, l.alpha) for l in self.features.layers] +
                      [(W, c, a) for (W, c, a, _, _) in self.classifier.layers])

    def forward(self, requantize: bool = False, conv_hook=None):
        """One forward pass on the current stream.  With requantize, the
        grouped quantizer runs on a second stream while the input's layout
        change runs on this one; the streams join before the first
        convolution (every launch keeps its order and inputs)."""
        hook = conv_hook
        if requantize:
            cur = torch.cuda.current_stream(self.features.device)
            qs = self.quant_stream
            qs.wait_stream(cur)
            with torch.cuda.stream(qs):
                self.quantize()
            joined = [False]

            def hook(i, layer, when):
                if not joined[0] and i == 0 and when == "before":
                    cur.wait_stream(qs)   # codes and alpha of every layer are ready
                    joined[0] = True
                if conv_hook:
                    conv_hook(i, layer, when)
        h = self.features.forward(requantize=False, conv_hook=hook)
        return self.classifier.forward(h.reshape(self.N, -1))

    def launches_per_forward(self, requantize: bool = False) -> int:
        n = self.features.launches_per_forward(False) + self.classifier.launches
        return n + (1 if requantize else 0)


def alexnet(batch: int | None = None, seed: int = 2, device="cuda") -> AlexNet:
    return AlexNet(batch, seed, device)


@dataclass
class TbnConv:
    name: str
    spec: _inputs.ConvSpec
    W: torch.Tensor          # fp32 [K, R*S*C] in (r, s, c) order
    codes: torch.Tensor
    alpha: torch.Tensor
    in_hw: tuple
    out_hw: tuple
    y: torch.Tensor          # NHWC bf16

    @property
    def flops_per_image(self) -> int:
        s = self.spec
        return 2 * s.K * self.out_hw[0] * self.out_hw[1] * s.C * s.R * s.S

    def run(self, x, residual=None, relu=None):
        s = self.spec
        tbn_conv2d_fwd(x, self.codes, self.alpha, s.K, s.R, s.S, (s.stride, s.stride),
                       (s.pad, s.pad), layout=TBN_NHWC, relu=s.relu if relu is None else relu,
                       residual=residual, out=self.y)
        return self.y


class ResNet18:
    """ResNet-18-shaped network: a full-precision 7x7/2 first convolution
    (fp32 weights, ReLU) and 3x3/2 max pool (pad 1), eight basic blocks of
    two-bit 3x3 convolutions (64/128/256/512 channels; the first block of
    stages 2-4 has stride 2 and a two-bit 1x1/2 projection shortcut), the
    residual added in the second convolution's fused epilogue before its
    ReLU, then a global average pool and a full-precision FC 512 -> 1000.
    Batch norm is the identity (synthetic weights carry no statistics)."""

    def __init__(self, batch: int | None = None, seed: int = 3, device="cuda"):
        self.device = torch.device(device)
        x, stem, convs, fc = _inputs.resnet18_inputs(seed, batch)
        dev = self.device
        self.N = N = x.shape[0]
        self.x_in = x.to(dev).contiguous()
        self.stem_w = stem.to(dev).contiguous()
        H, W = x.shape[2], x.shape[3]
        self.stem_hw = conv_out_hw(H, W, 7, 7, (2, 2), (3, 3))
        self.stem_y = torch.empty((N, self.stem_hw[0], self.stem_hw[1], 64), dtype=torch.bfloat16,
                                  device=dev)
        self.pool_hw = conv_out_hw(self.stem_hw[0], self.stem_hw[1], 3, 3, (2, 2), (1, 1))
        self.pool_y = torch.empty((N, self.pool_hw[0], self.pool_hw[1], 64), dtype=torch.bfloat16,
                                  device=dev)
        self.convs = {}
        hw = self.pool_hw
        stage_in = {}
        for name, spec, Wt in convs:
            blk = name[:4]
            if blk not in stage_in:
                stage_in[blk] = hw
            ihw = stage_in[blk] if name[-1] in "ad" else self.convs[blk + "a"].out_hw
            ohw = conv_out_hw(ihw[0], ihw[1], spec.R, spec.S, (spec.stride,) * 2, (spec.pad,) * 2)
            K = spec.K
            Wl = Wt.permute(0, 2, 3, 1).reshape(K, -1).contiguous().to(dev)
            codes = torch.empty((K, packed_words(Wl.shape[1])), dtype=torch.int32, device=dev)
            alpha = torch.empty((K,), dtype=torch.float32, device=dev)
            y = torch.empty((N, ohw[0], ohw[1], K), dtype=torch.bfloat16, device=dev)
            self.convs[name] = TbnConv(name, spec, Wl, codes, alpha, ihw, ohw, y)
            if name[-1] == "b":
                hw = ohw
        self.blocks = []
        for name in self.convs:
            if name[-1] == "a":
                blk = name[:4]
                self.blocks.append((self.convs[blk + "a"], self.convs[blk + "b"],
                                    self.convs.get(blk + "d")))
        self.feat_hw = hw
        self.feat = torch.empty((N, 512), dtype=torch.float32, device=dev)
        self.fc_w = fc.to(dev).contiguous()
        self.logits = torch.empty((N, self.fc_w.shape[0]), dtype=torch.float32, device=dev)
        self.out = self.logits

    @property
    def tbn_flops(self) -> int:
        """Algorithmic flops of the 19 two-bit convolutions per batch."""
        return self.N * sum(c.flops_per_image for c in self.convs.values())

    @property
    def dense_flops(self) -> int:
        """Flops of the full-precision first convolution and FC per batch."""
        P, Q = self.stem_hw
        return self.N * (2 * 64 * P * Q * 3 * 49 + 2 * self.fc_w.shape[0] * self.fc_w.shape[1])

    def quantize(self):
        _quantize_all([(c.W, c.codes, c.alpha) for c in self.convs.values()])

    def stem(self):
        tbn_dense_conv2d_fwd(self.x_in, self.stem_w, (2, 2), (3, 3), layout=TBN_NCHW_NHWC,
                             out_dtype=torch.bfloat16, relu=True, out=self.stem_y)
        tbn_maxpool2d_nhwc(self.stem_y, (3, 3), (2, 2), out=self.pool_y, pad=(1, 1))
        return self.pool_y

    def body(self, h):
        """The two-bit basic blocks from the pooled stem output."""
        for a, b, d in self.blocks:
            a.run(h)
            res = d.run(h) if d is not None else h
            b.run(a.y, residual=res, relu=True)
            h = b.y
        return h

    def head(self, h):
        tbn_avgpool2d_global_nhwc(h, out=self.feat)
        tbn_dense_linear_fwd(self.feat, self.fc_w, out=self.logits)
        return self.logits

    def forward(self, requantize: bool = False, conv_hook=None):
        """conv_hook(0, None, "before") is called once, after the stem has
        read the input (the benchmark copies the next batch from then on)."""
        if requantize:
            self.quantize()
        h = self.stem()
        if conv_hook:
            conv_hook(0, None, "before")
        return self.head(self.body(h))

    def launches_per_forward(self, requantize: bool = False) -> int:
        n = 2 + len(self.convs) + 2
        return n + ((len(self.convs) + 15) // 16 if requantize else 0)


def resnet18(batch: int | None = None, seed: int = 3, device="cuda") -> ResNet18:
    return ResNet18(batch, seed, device)
