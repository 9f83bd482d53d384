"""Model memory of Two-Bit Networks against full-precision weights.

The comparison of Fig. 2 (Section 4: TBN storage against double-precision
weights for AlexNet, ResNet-18 and VGG-19), recomputed from the layer shapes;
the paper prints no values for it.  A TBN layer stores, per filter (output
neuron) of n weights, tbn_packed_words(n) 32-bit words of two-bit codes and
one fp32 alpha (Eq. 5); a full-precision layer stores n values per filter.
Every convolution and fully-connected weight is counted (biases and batch
normalisation, which the TBN method does not quantize, are not).

Run ``python -m paper_1701_00485_gb300.memory`` for the table.
"""
from __future__ import annotations

from . import packed_words
from .inputs import ALEXNET, resnet18_convs

# VGG-19 (configuration E): 16 3x3 convolutions, then 25088 -> 4096 -> 4096
# -> 1000 fully-connected layers.
VGG19_CONV_CHANNELS = [(3, 64), (64, 64), (64, 128), (128, 128), (128, 256), (256, 256),
                       (256, 256), (256, 256), (256, 512), (512, 512), (512, 512), (512, 512),
                       (512, 512), (512, 512), (512, 512), (512, 512)]
VGG19_FCS = [(25088, 4096), (4096, 4096), (4096, 1000)]


def layers(net: str) -> list[tuple[str, int, int]]:
    """(name, filters K, weights per filter n) of every weight layer."""
    if net == "alexnet":
        out = [("conv%d" % (i + 1), s.K, s.C * s.R * s.S) for i, s in enumerate(ALEXNET["convs"])]
        out += [("fc%d" % (i + 6), o, i_) for i, (i_, o, _) in enumerate(ALEXNET["fcs"])]
        return out
    if net == "resnet18":
        out = [("stem", 64, 3 * 7 * 7)]
        out += [(name, s.K, s.C * s.R * s.S) for name, s in resnet18_convs()]
        out.append(("fc", 1000, 512))
        return out
    if net == "vgg19":
        out = [("conv%d" % (i + 1), co, ci * 9) for i, (ci, co) in enumerate(VGG19_CONV_CHANNELS)]
        out += [("fc%d" % (i + 1), o, i_) for i, (i_, o) in enumerate(VGG19_FCS)]
        return out
    raise ValueError("unknown network %r" % net)


def report(net: str) -> dict:
    """Weights and bytes of the network in fp64, fp32 and TBN form."""
    ls = layers(net)
    weights = sum(K * n for _, K, n in ls)
    tbn_codes = sum(K * packed_words(n) * 4 for _, K, n in ls)
    tbn_alpha = sum(K * 4 for _, K, _ in ls)
    tbn = tbn_codes + tbn_alpha
    return {"net": net, "weights": weights, "fp64_bytes": 8 * weights, "fp32_bytes": 4 * weights,
            "tbn_code_bytes": tbn_codes, "tbn_alpha_bytes": tbn_alpha, "tbn_bytes": tbn,
            "ratio_fp64": 8 * weights / tbn, "ratio_fp32": 4 * weights / tbn}


def main() -> None:
    print("%-9s %12s %12s %12s %12s %9s %9s" % ("network", "weights", "fp64 MB", "fp32 MB",
                                                "TBN MB", "fp64/TBN", "fp32/TBN"))
    for net in ("alexnet", "resnet18", "vgg19"):
        r = report(net)
        print("%-9s %12d %12.2f %12.2f %12.2f %9.2f %9.2f" % (
            net, r["weights"], r["fp64_bytes"] / 1e6, r["fp32_bytes"] / 1e6, r["tbn_bytes"] / 1e6,
            r["ratio_fp64"], r["ratio_fp32"]))


if __name__ == "__main__":
    main()
