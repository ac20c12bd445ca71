"""Failure detection without a GPU fault: a kernel wait that runs out is
reported through the device status word, and the context stays usable.

Two forms.  The self test runs the kernels' own wait helpers on a barrier
that nothing arrives on.  The abort-path tests lower the wait limit of the
real kernels (w4a16_selftest_set_wait_limit) so that their first wait that
does not complete at once gives up: the kernel records the timeout, drains
the copies and MMAs it has in flight, frees its tensor memory and returns.
A correct linear right after shows that the context survived."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2608_30877_gb300 import synthetic as S
from tests.gpu_helpers import assert_close, bf16_to_f64, host_case, to_device

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _W():
    from paper_2608_30877_gb300 import w4a16 as W
    return W


def _linear_still_correct(M=40, g=128):
    W = _W()
    x, xb, packed, scales = host_case(M, 256, 512, g, 21, 22)
    xd, wd, sd = to_device(x, packed, scales)
    out = W.linear(xd, wd, sd, g)
    torch.cuda.synchronize()
    ref = O.linear_rows(xb, packed, scales, 256, 512, g)
    assert_close(bf16_to_f64(out), ref, "after timeout")
    assert W.get_device_error() == W.OK


def test_bounded_wait_reports_timeout_and_context_survives():
    W = _W()
    assert W.get_device_error() == W.OK
    # 1 ms on a barrier nothing arrives on; the second waiter leaves through
    # the abort flag (else the kernel records INVALID_ARG instead)
    W.selftest_wait_timeout(1_000_000)
    assert W.get_device_error() == W.ERR_TIMEOUT
    assert W.get_device_error() == W.OK  # read-and-clear
    _linear_still_correct()


def test_selftest_rejects_bad_limit():
    W = _W()
    assert W.lib().w4a16_selftest_wait_timeout(10, None) == W.ERR_INVALID_ARG
    assert W.lib().w4a16_selftest_wait_timeout(10**7, None) == W.ERR_INVALID_ARG
    assert W.lib().w4a16_selftest_set_wait_limit(-1) == W.ERR_INVALID_ARG
    assert W.lib().w4a16_selftest_set_wait_limit(5 * 10**9) == W.ERR_INVALID_ARG


@pytest.fixture
def short_waits():
    W = _W()
    assert W.get_device_error() == W.OK
    W.set_wait_limit(1)
    try:
        yield W
    finally:
        W.set_wait_limit(0)


# (M, N, K, g): large-M tcgen05 GEMM on CTA pairs (several tiles per pair),
# the warp-level small-M streaming kernel, the tcgen05 small-M streaming
# kernel with 32, 64 and 128 token columns, the 32-token tcgen05 tiles (g = 64)
ABORT_CASES = [(600, 128 * 400, 2048, 128), (8, 8192, 4096, 128), (24, 8192, 4096, 128),
               (48, 8192, 4096, 128), (96, 8192, 4096, 128),
               (16, 4096, 1024, 64)]


@pytest.mark.parametrize("M,N,K,g", ABORT_CASES)
def test_linear_abort_path_under_short_waits(short_waits, M, N, K, g):
    W = short_waits
    x = S.make_x(M, K, 3, "cuda")
    w = torch.zeros((N, K // 2), dtype=torch.uint8, device="cuda")
    s = torch.zeros((N, K // g), dtype=torch.bfloat16, device="cuda")
    W.linear(x, w, s, g)
    assert W.get_device_error() == W.ERR_TIMEOUT
    W.set_wait_limit(0)
    _linear_still_correct(M=M if M <= 128 else 200, g=g)


def test_fused_abort_path_under_short_waits(short_waits):
    W = short_waits
    M, N, K = 300, 128 * 200, 2048
    x = S.make_x(M, K, 3, "cuda")
    w = torch.zeros((N, K // 2), dtype=torch.uint8, device="cuda")
    s = torch.zeros((N, K // 128), dtype=torch.bfloat16, device="cuda")
    res = torch.zeros((M, N // 2), dtype=torch.bfloat16, device="cuda")
    W.linear_fused(x, w, s, 128, act=W.ACT_SWIGLU, residual=res, out=res)
    assert W.get_device_error() == W.ERR_TIMEOUT
    W.set_wait_limit(0)
    _linear_still_correct()


def test_attention_abort_path_under_short_waits(short_waits):
    W = short_waits
    H, L, nseq = 8, 1024, 4
    qkv = S.make_x(L * nseq, 3 * H * 128, 9, "cuda")
    st = torch.arange(0, L * nseq + 1, L, dtype=torch.int32, device="cuda")
    W.attention_prefill(qkv, st, H, 32768)
    assert W.get_device_error() == W.ERR_TIMEOUT
    W.set_wait_limit(0)
    _linear_still_correct()


def test_first_error_is_kept():
    """A bad gather index after a timeout does not overwrite the timeout."""
    W = _W()
    assert W.get_device_error() == W.OK
    W.selftest_wait_timeout(1_000_000)
    src = torch.zeros((4, 64), dtype=torch.bfloat16, device="cuda")
    idx = torch.tensor([0, 7], dtype=torch.int32, device="cuda")
    W.gather_rows(src, idx)
    assert W.get_device_error() == W.ERR_TIMEOUT
    W.gather_rows(src, idx)
    assert W.get_device_error() == W.ERR_INVALID_ARG
    assert W.get_device_error() == W.OK
