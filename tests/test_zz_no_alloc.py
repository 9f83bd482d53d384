"""tbn_linear_fwd_noalloc: the batch-1 fp32 table GEMV with its scratch in a
file-scope device array of the library.  Collected last on purpose: it must
pass alone and after every other test, whatever those left on the device."""
import pytest
import torch

import paper_1701_00485_gb300 as tbn
from paper_1701_00485_gb300 import inputs

pytestmark = pytest.mark.gpu


def _layer(K_in, K_out, seed):
    g = inputs.generator(seed)
    W = inputs.normal((K_out, K_in), 1.3, g).cuda()
    codes, alpha = tbn.tbn_quantize_pack(W)
    x = torch.randn(1, K_in, generator=g).cuda()
    return x, codes, alpha


@pytest.mark.parametrize("K_in,K_out", [(64, 16), (576, 33), (4160, 20000), (16384, 16384),
                                        (16384, 32768)])
def test_noalloc_matches_the_workspace_entry_point_twice(K_in, K_out):
    """Two calls in a row of each entry point give bitwise the same outputs
    (the static scratch needs no clearing between calls)."""
    x, codes, alpha = _layer(K_in, K_out, K_in + 3 * K_out)
    ws = torch.empty(max(tbn.tbn_linear_workspace_bytes(1, K_in, K_out, torch.float32), 256),
                     dtype=torch.uint8, device="cuda")
    ref = [tbn.tbn_linear_fwd_ws(x, codes, alpha, K_out, ws, out_dtype=torch.float32)
           for _ in range(2)]
    got = [tbn.tbn_linear_fwd_noalloc(x, codes, alpha, K_out, out_dtype=torch.float32)
           for _ in range(2)]
    torch.cuda.synchronize()
    assert tbn.tbn_device_error() == 0
    assert torch.equal(ref[0], ref[1])
    assert torch.equal(got[0], ref[0]) and torch.equal(got[1], ref[0])


def test_noalloc_epilogue_matches():
    x, codes, alpha = _layer(2048, 700, 5)
    res = torch.randn(1, 700, device="cuda").to(torch.bfloat16)
    ws = torch.empty(tbn.tbn_linear_workspace_bytes(1, 2048, 700, torch.float32),
                     dtype=torch.uint8, device="cuda")
    ref = tbn.tbn_linear_fwd_ws(x, codes, alpha, 700, ws, out_dtype=torch.bfloat16, relu=True,
                                residual=res)
    got = tbn.tbn_linear_fwd_noalloc(x, codes, alpha, 700, out_dtype=torch.bfloat16, relu=True,
                                     residual=res)
    torch.cuda.synchronize()
    assert torch.equal(got, ref)


def test_noalloc_rejects_oversize_and_other_shapes():
    """More than 4 MiB of scratch (16384 inputs, 32769 outputs), bf16
    activations and batches above one are refused before any launch."""
    dummy = torch.zeros(16, dtype=torch.int32, device="cuda")
    alpha = torch.ones(32769, device="cuda")
    with pytest.raises(tbn.TBNError) as e:
        tbn.tbn_linear_fwd_noalloc(torch.zeros(1, 16384, device="cuda"), dummy, alpha, 32769)
    assert e.value.status == tbn.TBN_ERR_UNSUPPORTED
    with pytest.raises(tbn.TBNError) as e:
        tbn.tbn_linear_fwd_noalloc(torch.zeros(1, 64, device="cuda").to(torch.bfloat16), dummy,
                                   alpha, 16)
    assert e.value.status == tbn.TBN_ERR_UNSUPPORTED
    with pytest.raises(tbn.TBNError) as e:
        tbn.tbn_linear_fwd_noalloc(torch.zeros(2, 64, device="cuda"), dummy, alpha, 16)
    assert e.value.status == tbn.TBN_ERR_UNSUPPORTED
    assert tbn.tbn_device_error() == 0
