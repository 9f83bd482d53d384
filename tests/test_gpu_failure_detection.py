"""Failure detection without a fault: a bounded kernel wait that nothing
ends runs out, records the timeout in the device error word, returns, and
the device keeps computing correctly afterwards."""
import time

import pytest
import torch

import paper_1701_00485_gb300 as tbn
from paper_1701_00485_gb300 import inputs
from parity_util import check_quantize

pytestmark = pytest.mark.gpu


def test_bounded_wait_runs_out_and_is_reported():
    tbn.tbn_device_error()                         # start from a clear word
    t0 = time.perf_counter()
    tbn.tbn_selftest_wait_timeout(2000)            # 2 ms
    flags = tbn.tbn_device_error()                 # synchronizes
    elapsed = time.perf_counter() - t0
    assert flags & tbn.TBN_DEVERR_TIMEOUT
    assert elapsed >= 0.002
    assert tbn.tbn_device_error() == 0             # reading cleared the word
    # the context is still usable: a quantization right after it is exact
    W = inputs.normal((64, 300), 1.3, inputs.generator(77))
    codes, alpha = tbn.tbn_quantize_pack(W.cuda())
    torch.cuda.synchronize()
    check_quantize(W, codes, alpha)
    assert tbn.tbn_device_error() == 0
