"""Seeded synthetic inputs for the TBN workloads.

Shared by the tests, the benchmark and the smoke check, and by both the CUDA
path and the CPU oracle.  It holds no arithmetic of the method: it only
draws tensors (torch CPU generator, so a seed gives the same values on every
machine running the same torch build) with the shapes and distributions of
the five workloads:

  lenet      x fp32 U(0,1) [16,1,28,28]; W fp32 N(0, 0.1) [20,1,5,5]; seed 0
  vgg_small  x bf16 N(0,1) [128,3,32,32]; six 3x3/p1 layers 128-128-256-256-512-512,
             He-normal W, 2x2 max pool after every second layer; seed 1
  alexnet    x bf16 N(0,1) [256,3,227,227]; conv 96x11x11/s4, 256x5x5/p2,
             384x3x3/p1, 384x3x3/p1, 256x3x3/p1 with 3x3/s2 pools; FC
             9216-4096-4096-1000; He-normal W; seed 2
  resnet18   x bf16 N(0,1) [128,3,224,224]; basic-block ResNet-18 convs; seed 3
  gemv       W He-normal [K,K] for K in {4096, 8192, 16384}; x bf16 N(0,1) [B,K],
             B in {1, 8}; seed 4

"He-normal" is N(0, sqrt(2 / fan_in)) with fan_in = C*R*S (the std is the
second parameter).  Weights are returned as fp32 [K, C, R, S] (PyTorch's
order); callers permute to the order their activation layout reads.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import torch


def generator(seed: int) -> torch.Generator:
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed))
    return g


def normal(shape, std: float, g: torch.Generator) -> torch.Tensor:
    return torch.randn(*shape, generator=g, dtype=torch.float32) * float(std)


def uniform01(shape, g: torch.Generator) -> torch.Tensor:
    return torch.rand(*shape, generator=g, dtype=torch.float32)


def he_normal(K, C, R, S, g) -> torch.Tensor:
    return normal((K, C, R, S), math.sqrt(2.0 / (C * R * S)), g)


@dataclass(frozen=True)
class ConvSpec:
    """One TBN convolution: C -> K channels, R x S kernel, stride, padding,
    followed by ReLU (relu) and an optional max pool (pool = (k, stride))."""
    C: int
    K: int
    R: int
    S: int
    stride: int = 1
    pad: int = 0
    relu: bool = True
    pool: tuple | None = None


LENET = dict(N=16, C=1, H=28, W=28, conv=ConvSpec(1, 20, 5, 5, 1, 0, relu=False))

VGG_SMALL = dict(N=128, C=3, H=32, W=32, convs=[
    ConvSpec(3, 128, 3, 3, 1, 1),
    ConvSpec(128, 128, 3, 3, 1, 1, pool=(2, 2)),
    ConvSpec(128, 256, 3, 3, 1, 1),
    ConvSpec(256, 256, 3, 3, 1, 1, pool=(2, 2)),
    ConvSpec(256, 512, 3, 3, 1, 1),
    ConvSpec(512, 512, 3, 3, 1, 1, pool=(2, 2)),
])

ALEXNET = dict(N=256, C=3, H=227, W=227, convs=[
    ConvSpec(3, 96, 11, 11, 4, 0, pool=(3, 2)),
    ConvSpec(96, 256, 5, 5, 1, 2, pool=(3, 2)),
    ConvSpec(256, 384, 3, 3, 1, 1),
    ConvSpec(384, 384, 3, 3, 1, 1),
    ConvSpec(384, 256, 3, 3, 1, 1, pool=(3, 2)),
], fcs=[(9216, 4096, True), (4096, 4096, True), (4096, 1000, False)])


def resnet18_convs():
    """(name, spec) for the TBN convolutions of ResNet-18 after the stem
    (3x3 basic-block convs and the three 1x1/2 projection shortcuts)."""
    out = []
    cin = 64
    for stage, cout in enumerate((64, 128, 256, 512)):
        for blk in range(2):
            stride = 2 if (stage > 0 and blk == 0) else 1
            out.append(("l%db%da" % (stage + 1, blk), ConvSpec(cin, cout, 3, 3, stride, 1)))
            out.append(("l%db%db" % (stage + 1, blk), ConvSpec(cout, cout, 3, 3, 1, 1)))
            if stride != 1 or cin != cout:
                out.append(("l%db%dd" % (stage + 1, blk),
                            ConvSpec(cin, cout, 1, 1, stride, 0, relu=False)))
            cin = cout
    return out


RESNET18 = dict(N=128, C=3, H=224, W=224)

GEMV_SIZES = (4096, 8192, 16384)
GEMV_BATCHES = (1, 8)


def lenet_inputs(seed: int = 0):
    g = generator(seed)
    cfg = LENET
    x = uniform01((cfg["N"], cfg["C"], cfg["H"], cfg["W"]), g)
    c = cfg["conv"]
    W = normal((c.K, c.C, c.R, c.S), 0.1, g)
    return x, W


def conv_stack_inputs(cfg, seed: int, batch: int | None = None):
    """x bf16 NCHW N(0,1) and He-normal fp32 weights [K,C,R,S] per conv."""
    g = generator(seed)
    N = cfg["N"] if batch is None else batch
    x = torch.randn(N, cfg["C"], cfg["H"], cfg["W"], generator=g, dtype=torch.float32)
    x = x.to(torch.bfloat16)
    Ws = [he_normal(c.K, c.C, c.R, c.S, g) for c in cfg["convs"]]
    Wfc = [he_normal(o, i, 1, 1, g).reshape(o, i) for (i, o, _) in cfg.get("fcs", [])]
    return x, Ws, Wfc


def vgg_small_inputs(seed: int = 1, batch: int | None = None):
    x, Ws, _ = conv_stack_inputs(VGG_SMALL, seed, batch)
    return x, Ws


def alexnet_inputs(seed: int = 2, batch: int | None = None):
    return conv_stack_inputs(ALEXNET, seed, batch)


def resnet18_inputs(seed: int = 3, batch: int | None = None):
    g = generator(seed)
    N = RESNET18["N"] if batch is None else batch
    x = torch.randn(N, 3, 224, 224, generator=g, dtype=torch.float32).to(torch.bfloat16)
    stem = he_normal(64, 3, 7, 7, g)
    convs = [(name, spec, he_normal(spec.K, spec.C, spec.R, spec.S, g))
             for name, spec in resnet18_convs()]
    fc = he_normal(1000, 512, 1, 1, g).reshape(1000, 512)
    return x, stem, convs, fc


def gemv_inputs(K: int, B: int, seed: int = 4):
    g = generator(seed * 1000003 + K * 31 + B)
    W = normal((K, K), math.sqrt(2.0 / K), g)
    x = torch.randn(B, K, generator=g, dtype=torch.float32).to(torch.bfloat16)
    return W, x


def scaled_weights(shape, seed: int, scale: float = 1.5):
    """Weights spread so that all four codes occur (|W| > 1 is common)."""
    g = generator(seed)
    return normal(shape, scale, g)
