"""Two-bit network forward passes built from the C-ABI calls.

A network object owns its device buffers (fp32 real-valued weights, packed
codes, alpha, activations) so that one forward pass is a fixed sequence of
library launches on one stream -- capturable in a CUDA graph.  Weights are
kept as real values and re-quantized at every forward (Algorithm 1: the
quantization loop runs before TwoBitForward), with one grouped
tbn_quantize_pack_group launch for all layers; ``requantize=False`` runs the
inference form (codes + alpha only, Section 3).

Activations are NHWC bf16 between layers; the input batch arrives NCHW and
is converted by tbn_nchw_to_nhwc.  Weights of an NHWC layer are packed in
(r, s, c) order: the fp32 [K, C, R, S] weights are permuted once at build
time (quantization is elementwise and alpha is order-independent).
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

from . import (TBN_NHWC, tbn_conv2d_fwd, tbn_linear_fwd, tbn_maxpool2d_nhwc, tbn_nchw_to_nhwc,
               tbn_quantize_pack_group, packed_words, conv_out_hw)
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
        tbn_nchw_to_nhwc(self.x_in, out=self.x_nhwc)
        h = self.x_nhwc
        for i, l in enumerate(self.layers):
            s = l.spec
            if conv_hook:
                conv_hook(i, l, "before")
            tbn_conv2d_fwd(h, l.codes, l.alpha, s.K, s.R, s.S, (s.stride, s.stride),
                           (s.pad, s.pad), layout=TBN_NHWC, relu=s.relu, out=l.y,
                           pool=2 if s.pool == (2, 2) else 0)
            if conv_hook:
                conv_hook(i, l, "after")
            h = l.y
            if l.pooled is not None:
                k, st = s.pool
                tbn_maxpool2d_nhwc(h, (k, k), (st, st), out=l.pooled)
                h = l.pooled
        return h

    def launches_per_forward(self, requantize: bool = True) -> int:
        # NCHW->NHWC, one launch per conv, one per pool that is not fused
        n = 1 + len(self.layers) + sum(1 for l in self.layers if l.pooled is not None)
        if requantize:
            n += (len(self.layers) + 15) // 16
        return n


def vgg_small(batch: int | None = None, seed: int = 1, device="cuda") -> ConvStack:
    x, Ws = _inputs.vgg_small_inputs(seed, batch)
    return ConvStack(_inputs.VGG_SMALL["convs"], x, Ws, device)


class FCStack:
    """Fully-connected TBN layers (Section 3), ReLU between them."""

    def __init__(self, fcs, weights, batch, device="cuda"):
        self.device = torch.device(device)
        self.layers = []
        for (kin, kout, relu), W in zip(fcs, weights):
            W = W.contiguous().to(self.device)
            codes = torch.empty((kout, packed_words(kin)), dtype=torch.int32, device=self.device)
            alpha = torch.empty((kout,), dtype=torch.float32, device=self.device)
            y = torch.empty((batch, kout), dtype=torch.bfloat16, device=self.device)
            self.layers.append((W, codes, alpha, relu, y))

    def quantize(self):
        tbn_quantize_pack_group([(W, c, a) for (W, c, a, _, _) in self.layers])

    def forward(self, x, requantize: bool = False):
        if requantize:
            self.quantize()
        h = x
        for (W, codes, alpha, relu, y) in self.layers:
            tbn_linear_fwd(h, codes, alpha, codes.shape[0], relu=relu, out=y)
            h = y
        return h
