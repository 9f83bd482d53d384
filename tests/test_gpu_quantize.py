"""GPU parity of tbn_quantize_pack / tbn_quantize_pack_group / tbn_unpack
against the oracle (codes bit-exact, alpha within 1e-6 relative)."""
import numpy as np
import pytest
import torch

import oracle
import paper_1701_00485_gb300 as tbn
from paper_1701_00485_gb300 import inputs
from parity_util import check_quantize, u32

pytestmark = pytest.mark.gpu

SHAPES = [(1, 1), (3, 15), (5, 16), (7, 17), (20, 25), (128, 27), (9, 31), (64, 363),
          (33, 1152), (16, 4100), (8, 4608), (3, 16384), (2, 40000), (300, 64)]


def _weights(K, n, dist, seed):
    g = inputs.generator(seed)
    if dist == "small":
        return inputs.normal((K, n), 0.1, g)
    if dist == "wide":
        return inputs.normal((K, n), 1.5, g)
    return (inputs.uniform01((K, n), g) * 6.0 - 3.0)


@pytest.mark.parametrize("K,n", SHAPES)
@pytest.mark.parametrize("dist", ["small", "wide", "uniform3"])
def test_quantize_matches_oracle(K, n, dist):
    W = _weights(K, n, dist, seed=K * 7919 + n)
    codes, alpha = tbn.tbn_quantize_pack(W.cuda())
    torch.cuda.synchronize()
    assert codes.shape == (K, (n + 15) // 16)
    check_quantize(W, codes, alpha)


def test_quantize_boundary_values():
    f = np.float32
    vals = [-1.0, -0.0, 0.0, 1.0, float(np.nextafter(f(1), f(2))), float(np.nextafter(f(1), f(0))),
            float(np.nextafter(f(-1), f(-2))), float(np.nextafter(f(-1), f(0))),
            float(np.nextafter(f(0), f(1))), -float(np.nextafter(f(0), f(1))), 3e38, -3e38,
            1e-38, -2.5, 2.5, 0.5, -0.5]
    row = torch.tensor(vals * 3, dtype=torch.float32)
    W = torch.stack([row, row.flip(0), row.roll(5)])
    codes, alpha = tbn.tbn_quantize_pack(W.cuda())
    check_quantize(W, codes, alpha)


def test_quantize_all_zero_filter_and_special_cases():
    W = torch.zeros(2, 20)
    a0 = np.float32(2.0 / 3.0)
    W[1, :4] = torch.tensor([a0, -a0, 2 * a0, -2 * a0])
    W[1, 4:] = torch.tensor([a0] * 16)
    codes, alpha = tbn.tbn_quantize_pack(W.cuda())
    check_quantize(W, codes, alpha)
    al = alpha.cpu().numpy()
    assert al[0] == 0.0
    assert abs(float(al[1]) - float(a0)) <= 1e-6 * float(a0)


def test_quantize_unaligned_rows_take_scalar_path():
    base = _weights(10, 1154, "wide", seed=5).cuda()
    W = base.reshape(-1)[1:1 + 10 * 1153].reshape(10, 1153)  # 4-byte aligned only
    codes = torch.empty((10, 73), dtype=torch.int32, device="cuda")
    alpha = torch.empty((10,), dtype=torch.float32, device="cuda")
    st = tbn.lib().tbn_quantize_pack(W.data_ptr(), 10, 1153, codes.data_ptr(), alpha.data_ptr(),
                                     None)
    assert st == 0
    torch.cuda.synchronize()
    check_quantize(W.cpu(), codes, alpha)


def test_quantize_group_matches_single_calls():
    shapes = [(128, 27), (128, 1152), (256, 1152), (256, 2304), (512, 2304), (512, 4608),
              (20, 25), (3, 17)]
    jobs, cpu = [], []
    for i, (K, n) in enumerate(shapes):
        W = _weights(K, n, "wide" if i % 2 else "small", seed=100 + i)
        cpu.append(W)
        jobs.append((W.cuda(), torch.empty((K, (n + 15) // 16), dtype=torch.int32, device="cuda"),
                     torch.empty((K,), dtype=torch.float32, device="cuda")))
    tbn.tbn_quantize_pack_group(jobs)
    torch.cuda.synchronize()
    for W, (_, codes, alpha) in zip(cpu, jobs):
        check_quantize(W, codes, alpha)
        c1, a1 = tbn.tbn_quantize_pack(W.cuda())
        assert torch.equal(c1, codes) and torch.equal(a1, alpha)


@pytest.mark.parametrize("K", [16384])
def test_quantize_full_size_sampled_rows(K):
    # the 16384 x 16384 matrix of the GEMV workload: every row quantized on
    # the GPU, 96 sampled rows (and the first/last) compared with the oracle
    W, _ = inputs.gemv_inputs(K, 1)
    Wd = W.cuda()
    codes, alpha = tbn.tbn_quantize_pack(Wd)
    torch.cuda.synchronize()
    rng = np.random.default_rng(7)
    rows = np.unique(np.concatenate([[0, K - 1], rng.integers(0, K, size=96)]))
    check_quantize(W, codes, alpha, rows=rows)


@pytest.mark.parametrize("K,n", [(1, 1), (5, 17), (64, 363), (7, 4608)])
def test_unpack_formats(K, n):
    W = _weights(K, n, "wide", seed=K + n)
    codes, alpha = tbn.tbn_quantize_pack(W.cuda())
    wt, al = oracle.quantize(W.numpy())
    i8 = tbn.tbn_unpack(codes, None, n, tbn.TBN_UNPACK_I8).cpu().numpy()
    assert np.array_equal(i8, wt)
    assert np.array_equal(oracle.unpack(u32(codes), n), wt)
    f32 = tbn.tbn_unpack(codes, alpha, n, tbn.TBN_UNPACK_F32).cpu().numpy()
    a = alpha.cpu().numpy()
    assert np.array_equal(f32, (a[:, None] * wt.astype(np.float32)).astype(np.float32))
    bf = tbn.tbn_unpack(codes, alpha, n, tbn.TBN_UNPACK_BF16).cpu()
    want = torch.from_numpy(a[:, None] * wt.astype(np.float32)).to(torch.bfloat16)
    assert torch.equal(bf, want)


def test_no_device_error_recorded():
    assert tbn.tbn_device_error() == 0
