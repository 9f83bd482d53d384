"""GPU parity of the batch-1 fp8 tensor-core linear layer (tbn_linear_prepare_f8
+ tbn_linear_fwd_f8) against the oracle's linear layer, per output:
|y_gpu - y_orc| <= 2e-3 * |alpha| * sum|x| (fp32 output; bf16 adds its
rounding), and the prepared code layout bit-exact against its definition."""
import numpy as np
import pytest
import torch

import oracle
import paper_1701_00485_gb300 as tbn
from paper_1701_00485_gb300 import inputs
from parity_util import assert_within, check_quantize, u32

pytestmark = pytest.mark.gpu


def e4m3_planar_reference(words: np.ndarray) -> np.ndarray:
    """Byte-planar code l = 2p + h (m at bit 16h + p, s at 16h + 8 + p) moved
    to e4m3-planar code l = 4j + b (m at bit 8b + j, s at 8b + 4 + j)."""
    w = words.astype(np.uint64)
    out = np.zeros_like(w)
    for l in range(16):
        src = 16 * (l & 1) + (l >> 1)
        dst = 8 * (l & 3) + (l >> 2)
        out |= ((w >> src) & 1) << dst
        out |= ((w >> (src + 8)) & 1) << (dst + 4)
    return out.astype(np.uint32)


def prepared_reference(words: np.ndarray, K_in: int) -> np.ndarray:
    """Blocked layout [tiles][K_in / 512][128 rows][32 words]: word w of row r
    of a block at position 4 ((w / 4) ^ (r % 8)) + w % 4; rows past K_out 0."""
    K_out = words.shape[0]
    tiles, nks = -(-K_out // 128), K_in // 512
    e = np.zeros((tiles * 128, K_in // 16), dtype=np.uint32)
    e[:K_out] = e4m3_planar_reference(words)
    blk = e.reshape(tiles, 128, nks, 32).transpose(0, 2, 1, 3).copy()   # [t][ks][r][w]
    out = np.empty_like(blk)
    for r in range(128):
        for wp in range(32):
            w = (((wp >> 2) ^ (r & 7)) << 2) | (wp & 3)
            out[:, :, r, wp] = blk[:, :, r, w]
    return out.reshape(-1)


@pytest.mark.parametrize("K_out,K_in", [(4, 512), (7, 1024), (130, 4096)])
def test_prepare_f8_layout_is_bit_exact(K_out, K_in):
    g = inputs.generator(K_out * 7 + K_in)
    W = inputs.normal((K_out, K_in), 1.5, g)
    codes, _ = tbn.tbn_quantize_pack(W.cuda())
    prep = tbn.tbn_linear_prepare_f8(codes, K_in)
    torch.cuda.synchronize()
    assert prep.numel() == tbn.tbn_linear_f8_prepared_words(K_out, K_in)
    assert np.array_equal(u32(prep), prepared_reference(u32(codes), K_in))
    assert tbn.tbn_linear_f8_prepared_words(K_out, 1000) == -1


def run_f8(W, x, out_dtype, relu=False, residual=None):
    K_out, K_in = W.shape
    codes, alpha = tbn.tbn_quantize_pack(W.cuda())
    check_quantize(W, codes, alpha)
    prep = tbn.tbn_linear_prepare_f8(codes, K_in)
    ws = torch.empty(tbn.tbn_linear_f8_workspace_bytes(1, K_in, K_out), dtype=torch.uint8,
                     device="cuda")
    y = tbn.tbn_linear_fwd_f8(x.cuda(), prep, alpha, K_out, ws, out_dtype=out_dtype, relu=relu,
                              residual=residual.cuda() if residual is not None else None)
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    wt, al = oracle.quantize(W.numpy())
    y_orc, bound = oracle.linear(x.float().numpy(), wt, al)
    return y.float().cpu().numpy(), y_orc, bound


SHAPES = [
    # K_in, K_out: stream-K ranges that start and end inside tiles, ragged last tile
    (512, 128),       # one unit
    (512, 100),       # one ragged tile
    (1024, 1000),     # ranges of one unit, eight tiles
    (4096, 4096),     # 32 tiles x 8 stages over the grid
    (8192, 1000),     # 8 tiles x 16 stages: several CTAs per tile
    (16384, 384),     # 3 tiles x 32 stages: long segments split between CTAs
    (2560, 4100),     # ragged tile, 5 stages per tile
]


@pytest.mark.parametrize("K_in,K_out", SHAPES)
def test_f8_linear_matches_oracle(K_in, K_out):
    g = inputs.generator(K_in * 3 + K_out)
    W = inputs.normal((K_out, K_in), 1.3, g)
    x = torch.randn(1, K_in, generator=g).to(torch.bfloat16)
    y, y_orc, bound = run_f8(W, x, torch.float32)
    assert_within(y, y_orc, bound, out_bf16=False, what="f8 %d x %d" % (K_out, K_in))
    y, y_orc, bound = run_f8(W, x, torch.bfloat16)
    assert_within(y, y_orc, bound, out_bf16=True, what="f8 bf16 %d x %d" % (K_out, K_in))


@pytest.mark.parametrize("case", ["wide", "spike", "zeros", "tiny", "huge"])
def test_f8_linear_input_ranges(case):
    """The exact three-term split of x under one scale: inputs spanning many
    binades, one large element among small ones, all zeros, and vectors
    scaled near the bottom and the top of the bf16 range."""
    K_in, K_out = 4096, 256
    g = inputs.generator(11)
    W = inputs.normal((K_out, K_in), 1.3, g)
    x = torch.randn(1, K_in, generator=g)
    if case == "wide":
        x = x * torch.pow(2.0, torch.randint(-30, 30, (1, K_in), generator=g).float())
    elif case == "spike":
        x = x * 1e-6
        x[0, 17] = 1e4
    elif case == "zeros":
        x = torch.zeros(1, K_in)
    elif case == "tiny":
        x = x * 1e-30
    else:
        x = x * 1e30
    x = x.to(torch.bfloat16)
    y, y_orc, bound = run_f8(W, x, torch.float32)
    assert_within(y, y_orc, bound, out_bf16=False, what="f8 %s" % case)
    if case == "zeros":
        assert np.all(y == 0.0)


def test_f8_linear_epilogue():
    K_in, K_out = 2048, 700
    g = inputs.generator(12)
    W = inputs.normal((K_out, K_in), 1.3, g)
    x = torch.randn(1, K_in, generator=g).to(torch.bfloat16)
    res = torch.randn(1, K_out, generator=g)
    y, y_orc, bound = run_f8(W, x, torch.float32, relu=True, residual=res)
    want = oracle.epilogue(y_orc, res.numpy().astype(np.float64), relu=True)
    assert_within(y, want, bound, out_bf16=False, epilogue=True, what="f8 epilogue")


@pytest.mark.parametrize("K", [4096, 8192, 16384])
def test_f8_gemv_workload_full(K):
    """The GEMV workload's batch-1 inputs at full size, every output."""
    W, x = inputs.gemv_inputs(K, 1)
    y, y_orc, bound = run_f8(W, x.to(torch.bfloat16), torch.float32)
    assert_within(y, y_orc, bound, out_bf16=False, what="f8 gemv %d" % K)


def test_f8_is_bitwise_reproducible():
    K_in, K_out = 8192, 2048
    g = inputs.generator(13)
    W = inputs.normal((K_out, K_in), 1.3, g).cuda()
    x = torch.randn(1, K_in, generator=g).to(torch.bfloat16).cuda()
    codes, alpha = tbn.tbn_quantize_pack(W)
    prep = tbn.tbn_linear_prepare_f8(codes, K_in)
    ws = torch.empty(tbn.tbn_linear_f8_workspace_bytes(1, K_in, K_out), dtype=torch.uint8,
                     device="cuda")
    a = tbn.tbn_linear_fwd_f8(x, prep, alpha, K_out, ws, out_dtype=torch.float32)
    ws.fill_(0xAB)
    b = tbn.tbn_linear_fwd_f8(x, prep, alpha, K_out, ws, out_dtype=torch.float32)
    torch.cuda.synchronize()
    assert torch.equal(a, b)


def test_f8_refuses_unsupported_shapes():
    g = inputs.generator(14)
    W = inputs.normal((64, 1000), 1.0, g).cuda()
    codes, alpha = tbn.tbn_quantize_pack(W)
    x = torch.randn(1, 1000, generator=g).to(torch.bfloat16).cuda()
    ws = torch.empty(1 << 20, dtype=torch.uint8, device="cuda")
    with pytest.raises(tbn.TBNError):
        tbn.tbn_linear_fwd_f8(x, codes, alpha, 64, ws)   # K_in not a multiple of 512
    assert tbn.tbn_linear_f8_workspace_bytes(2, 4096, 64) == 0
    assert tbn.tbn_linear_f8_workspace_bytes(1, 32768, 64) == 0
