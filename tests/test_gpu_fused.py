"""Parity of the fused epilogue (w4a16_linear_fused) with the oracle:
act(x W^T + bias) + residual for every activation, with and without bias and
residual (also in place), on the small-M streaming kernel (g = 128), the
32-token tcgen05 tiles (small M, g = 64) and the large-M tcgen05 GEMM."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2608_30877_gb300 import synthetic as S
from tests.gpu_helpers import assert_close_fused, bf16_to_f64, host_case, to_device

pytestmark = pytest.mark.gpu


def _W():
    from paper_2608_30877_gb300 import w4a16 as W
    return W


def _case(M, N, K, g, seed, act, with_bias, with_res):
    W = _W()
    x, xb, packed, scales = host_case(M, N, K, g, seed, seed + 1)
    xd, wd, sd = to_device(x, packed, scales)
    n_out = N // 2 if act == W.ACT_SWIGLU else N
    rng = np.random.default_rng(seed + 2)
    bf16 = lambda a: S.bf16_bits(torch.from_numpy(a.astype(np.float32)).to(torch.bfloat16))
    bias = bf16(0.5 * rng.normal(size=N)) if with_bias else None
    res = bf16(0.5 * rng.normal(size=(M, n_out))) if with_res else None
    y = O.linear_rows(xb, packed, scales, N, K, g, nthreads=O.max_threads())
    ref = O.epilogue_rows(y, act, bias=bias, residual=res)
    to_dev = lambda b: torch.from_numpy(b.view(np.int16)).view(torch.bfloat16).cuda()
    return (xd, wd, sd, (None if bias is None else to_dev(bias)),
            (None if res is None else to_dev(res)), ref, y, bias)


SHAPES = [  # (M, N, K, g): streaming kernel, 32-token tcgen05 tiles, large-M GEMM
    (8, 1000, 1024, 128), (16, 4096, 512, 128), (24, 1234, 384, 128), (5, 200, 256, 64),
    (300, 1000, 1024, 128), (40, 258, 512, 128),
]


@pytest.mark.parametrize("M,N,K,g", SHAPES)
@pytest.mark.parametrize("act", [0, 1, 2])
def test_fused_activation_bias_residual(M, N, K, g, act):
    W = _W()
    for with_bias, with_res in ((False, False), (True, False), (True, True), (False, True)):
        xd, wd, sd, bias, res, ref, y, bias_bits = _case(M, N, K, g, 17 * M + N + act, act,
                                                         with_bias, with_res)
        out = W.linear_fused(xd, wd, sd, g, act=act, bias=bias, residual=res)
        torch.cuda.synchronize()
        assert_close_fused(bf16_to_f64(out), y, ref, act, bias_bits,
                           f"{M}x{K}x{N} g{g} act{act} b{with_bias} r{with_res}")


@pytest.mark.parametrize("M", [8, 300])
def test_fused_residual_in_place(M):
    W = _W()
    N, K, g = 512, 1024, 128
    xd, wd, sd, bias, res, ref, y, bias_bits = _case(M, N, K, g, 99 + M, W.ACT_GELU, True, True)
    buf = res.clone()
    W.linear_fused(xd, wd, sd, g, act=W.ACT_GELU, bias=bias, residual=buf, out=buf)
    torch.cuda.synchronize()
    assert_close_fused(bf16_to_f64(buf), y, ref, W.ACT_GELU, bias_bits, f"in-place residual M={M}")


def test_fused_none_equals_plain_linear():
    W = _W()
    M, N, K, g = 64, 1024, 512, 128
    x, xb, packed, scales = host_case(M, N, K, g, 5, 6)
    xd, wd, sd = to_device(x, packed, scales)
    a = W.linear(xd, wd, sd, g)
    b = W.linear_fused(xd, wd, sd, g)
    torch.cuda.synchronize()
    assert torch.equal(a, b)
