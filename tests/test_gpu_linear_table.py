"""GPU parity of the batch-1 table-lookup GEMV for fp32 activations
(tbn_linear_fwd_ws with a workspace) against the oracle: chunking of the
input into 512-column table sets, ragged row blocks, bf16 and fp32 outputs,
the fused epilogue, the GEMV workload sizes, and bitwise reproducibility."""
import numpy as np
import pytest
import torch

import oracle
import paper_1701_00485_gb300 as tbn
from paper_1701_00485_gb300 import inputs
from parity_util import assert_within, check_quantize

pytestmark = pytest.mark.gpu


def workspace_for(K_in, K_out):
    n = tbn.tbn_linear_workspace_bytes(1, K_in, K_out, torch.float32)
    return torch.empty(max(n, 256), dtype=torch.uint8, device="cuda"), n


def run_table(W, x, out_dtype, relu=False, residual=None, ws=None):
    assert x.dtype == torch.float32 and x.shape[0] == 1
    codes, alpha = tbn.tbn_quantize_pack(W.cuda())
    check_quantize(W, codes, alpha)
    if ws is None:
        ws, _ = workspace_for(W.shape[1], W.shape[0])
    y = tbn.tbn_linear_fwd_ws(x.cuda(), codes, alpha, W.shape[0], ws, out_dtype=out_dtype,
                              relu=relu,
                              residual=residual.cuda() if residual is not None else None)
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    wt, al = oracle.quantize(W.numpy())
    y_orc, bound = oracle.linear(x.numpy().astype(np.float64), wt, al)
    return y.float().cpu().numpy(), y_orc, bound


@pytest.mark.parametrize("K_in,K_out", [
    (64, 16),        # one chunk, one partial row block: results written directly
    (512, 1000),     # one full chunk, ragged last row block
    (576, 33),       # two chunks, the second 64 columns wide
    (1024, 100),
    (4160, 20000),   # nine chunks, ragged chunk and row block
    (8192, 1000),
    (16384, 257),    # 32 chunks over a few row blocks
])
def test_table_gemv_matches_oracle(K_in, K_out):
    g = inputs.generator(K_in * 5 + K_out)
    W = inputs.normal((K_out, K_in), 1.3, g)
    x = torch.randn(1, K_in, generator=g)
    y, y_orc, bound = run_table(W, x, torch.float32)
    assert_within(y, y_orc, bound, out_bf16=False, what="table gemv")
    y, y_orc, bound = run_table(W, x, torch.bfloat16)
    assert_within(y, y_orc, bound, out_bf16=True, what="table gemv bf16 out")


def test_table_gemv_uniform_codes_and_wide_inputs():
    """U(-3, 3) weights give all four codes in equal measure (every table
    entry is hit); inputs with exact zeros and a wide exponent range."""
    g = inputs.generator(4242)
    W = inputs.uniform01((3000, 2048), g) * 6.0 - 3.0
    x = torch.randn(1, 2048, generator=g)
    x = x * torch.exp2(torch.randint(-20, 20, (1, 2048), generator=g).float())
    x[0, ::7] = 0.0
    y, y_orc, bound = run_table(W, x, torch.float32)
    assert_within(y, y_orc, bound, out_bf16=False, what="table gemv wide x")


def test_table_gemv_epilogue():
    g = inputs.generator(77)
    W = inputs.normal((700, 1536), 1.0, g)
    x = torch.randn(1, 1536, generator=g)
    for out_dtype in (torch.float32, torch.bfloat16):
        res = torch.randn(1, 700, generator=g).to(out_dtype)
        y, y_orc, bound = run_table(W, x, out_dtype, relu=True, residual=res)
        want = oracle.epilogue(y_orc, res.float().numpy(), relu=True)
        assert_within(y, want, bound, out_bf16=out_dtype == torch.bfloat16, epilogue=True,
                      what="table gemv epilogue")


def test_table_gemv_is_reproducible_and_ignores_stale_workspace():
    """Chunk partials are added in chunk order whichever CTA finishes first,
    and every partial is written before it is read: a workspace left by a
    call of another shape, or filled with garbage, gives bitwise the same
    result."""
    g = inputs.generator(31337)
    W = inputs.normal((4096, 4096), 1.2, g)
    x = torch.randn(1, 4096, generator=g).cuda()
    codes, alpha = tbn.tbn_quantize_pack(W.cuda())
    ws, n = workspace_for(8192, 8192)
    assert n >= tbn.tbn_linear_workspace_bytes(1, 4096, 4096, torch.float32) > 0
    y1 = tbn.tbn_linear_fwd_ws(x, codes, alpha, 4096, ws, out_dtype=torch.float32)
    W2 = inputs.normal((1000, 8192), 1.0, g).cuda()
    c2, a2 = tbn.tbn_quantize_pack(W2)
    tbn.tbn_linear_fwd_ws(torch.randn(1, 8192, device="cuda"), c2, a2, 1000, ws)
    y2 = tbn.tbn_linear_fwd_ws(x, codes, alpha, 4096, ws, out_dtype=torch.float32)
    ws.fill_(0xA5)
    y3 = tbn.tbn_linear_fwd_ws(x, codes, alpha, 4096, ws, out_dtype=torch.float32)
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    assert torch.equal(y1, y2) and torch.equal(y1, y3)


def test_batch1_fp32_without_enough_workspace_is_refused():
    """A batch-1 fp32 layer of the table kernel's shape runs only there: with
    a workspace smaller than the query asks for (or none) the call returns
    TBN_ERR_UNSUPPORTED instead of taking the CUDA-core 1x1 convolution,
    and launches nothing."""
    g = inputs.generator(8)
    W = inputs.normal((300, 2048), 1.2, g)
    codes, alpha = tbn.tbn_quantize_pack(W.cuda())
    x = torch.randn(1, 2048, generator=g).cuda()
    small = torch.empty(64, dtype=torch.uint8, device="cuda")
    y = torch.full((1, 300), 7.0, device="cuda")
    for ws in (small, None):
        with pytest.raises(tbn.TBNError) as e:
            tbn.tbn_linear_fwd_ws(x, codes, alpha, 300, ws, out=y)
        assert e.value.status == tbn.TBN_ERR_UNSUPPORTED
    with pytest.raises(tbn.TBNError) as e:
        tbn.tbn_linear_fwd(x, codes, alpha, 300, out=y)
    assert e.value.status == tbn.TBN_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert torch.all(y == 7.0)
    # one chunk (K_in <= 512) needs no workspace
    x2 = torch.randn(1, 512, generator=g).cuda()
    c2, a2 = tbn.tbn_quantize_pack(inputs.normal((40, 512), 1.2, g).cuda())
    tbn.tbn_linear_fwd(x2, c2, a2, 40)


@pytest.mark.parametrize("K", inputs.GEMV_SIZES)
def test_table_gemv_workload_full(K):
    """The GEMV workload's weights at full size with fp32 activations, every
    output compared with the oracle."""
    W, x = inputs.gemv_inputs(K, 1)
    y, y_orc, bound = run_table(W, x.float(), torch.float32)
    assert_within(y, y_orc, bound, out_bf16=False, what="table gemv K=%d" % K)
    assert np.isfinite(y).all()
