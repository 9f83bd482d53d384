"""The Fig. 2 memory comparison (TBN storage against full-precision weights
for AlexNet, ResNet-18 and VGG-19), pinned to numbers fixed outside the
report: per-layer weight counts written out by hand, the size Section 1
prints for AlexNet with floating-point weights (249 MB), and the published
parameter totals of VGG-19 and ResNet-18 less their biases and batch-norm
parameters."""
from paper_1701_00485_gb300 import memory


def test_alexnet_weights_and_section1_size():
    hand = (96 * 3 * 11 * 11 + 256 * 96 * 5 * 5 + 384 * 256 * 9 + 384 * 384 * 9 + 256 * 384 * 9 +
            4096 * 9216 + 4096 * 4096 + 1000 * 4096)
    r = memory.report("alexnet")
    assert r["weights"] == hand == 62_367_776
    # Section 1: "249MB of memory with floating point weights"
    assert abs(r["fp32_bytes"] / 1e6 - 249.0) < 0.5


def test_vgg19_and_resnet18_weight_counts():
    # VGG-19: 143,667,240 parameters, of which 14,696 are biases
    assert memory.report("vgg19")["weights"] == 143_667_240 - 14_696
    # ResNet-18: 11,689,512 parameters, less 4,800 batch-norm channels x 2
    # and the 1,000 classifier biases
    assert memory.report("resnet18")["weights"] == 11_689_512 - 9_600 - 1_000


def test_tbn_bytes_are_codes_plus_alpha_per_filter():
    for net in ("alexnet", "resnet18", "vgg19"):
        r = memory.report(net)
        want = sum(K * (4 * (-(-n // 16)) + 4) for _, K, n in memory.layers(net))
        assert r["tbn_bytes"] == want
        # two bits instead of 64 is 32x, less the alpha and the word padding
        assert 31.5 < r["ratio_fp64"] < 32.0
        assert r["fp64_bytes"] == 2 * r["fp32_bytes"] == 8 * r["weights"]
