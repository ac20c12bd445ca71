"""Failure detection without a GPU fault: a kernel wait that runs out is
reported through the device status word, and the context stays usable."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from tests.gpu_helpers import assert_close, bf16_to_f64, host_case, to_device

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def test_bounded_wait_reports_timeout_and_context_survives():
    from paper_2608_30877_gb300 import w4a16 as W
    assert W.get_device_error() == W.OK
    W.selftest_wait_timeout(2_000_000)  # 2 ms, on a barrier nothing arrives on
    assert W.get_device_error() == W.ERR_TIMEOUT
    assert W.get_device_error() == W.OK  # read-and-clear
    # the context is still usable: a linear right after matches the oracle
    x, xb, packed, scales = host_case(40, 256, 512, 128, 21, 22)
    xd, wd, sd = to_device(x, packed, scales)
    out = W.linear(xd, wd, sd, 128)
    torch.cuda.synchronize()
    ref = O.linear_rows(xb, packed, scales, 256, 512, 128)
    assert_close(bf16_to_f64(out), ref, "after timeout")
    assert W.get_device_error() == W.OK


def test_selftest_rejects_bad_limit():
    from paper_2608_30877_gb300 import w4a16 as W
    assert W.lib().w4a16_selftest_wait_timeout(10, None) == W.ERR_INVALID_ARG
    assert W.lib().w4a16_selftest_wait_timeout(10**10, None) == W.ERR_INVALID_ARG
