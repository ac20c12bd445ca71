"""Parity of the fused epilogue (w4a16_linear_fused) with the oracle:
act(x W^T + bias) + residual for every activation, with and without bias and
residual (also in place), on the small-M streaming kernel (g = 128), the
32-token tcgen05 tiles (small M, g = 64) and the large-M tcgen05 GEMM."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2608_30877_gb300 import synthetic as S
from tests.gpu_helpers import assert_close_fused, bf16_to_f64, host_case, prepare_weights, to_device

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
    (300, 1000, 1024, 128), (40, 258, 512, 128), (64, 1000, 1024, 128),
    (100, 1000, 1024, 128),
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


def _rows(M):
    rng = np.random.default_rng(M + 1)
    r = {0, 255, 256, M - 1, M // 2}
    r.update(int(v) for v in rng.integers(0, M, size=5))
    return np.array(sorted(r), dtype=np.int64)


@pytest.mark.slow
def test_fused_swiglu_bias_fullsize_sampled():
    """SwiGLU + bias on the benched gate/up shape (8192 tokens x K 12288 x
    2 x 49152 interleaved rows): the persistent, raster-grouped GEMM over
    many waves, on sampled token rows (all outputs) and output columns (all
    tokens)."""
    W = _W()
    c = S.MLP_SWIGLU
    packed, scales, wd, sd = prepare_weights(c.N, c.K, c.g, c.w_seed)
    x = S.make_x(c.M, c.K, c.x_seed, "cuda")
    rng = np.random.default_rng(11)
    bias = S.bf16_bits(torch.from_numpy((0.5 * rng.normal(size=c.N)).astype(np.float32))
                       .to(torch.bfloat16))
    bias_d = torch.from_numpy(bias.view(np.int16)).view(torch.bfloat16).cuda()
    out = W.linear_fused(x, wd, sd, c.g, act=W.ACT_SWIGLU, bias=bias_d)
    torch.cuda.synchronize()
    nth = O.max_threads()
    rows = _rows(c.M)
    ridx = torch.from_numpy(rows).cuda()
    y = O.linear_rows(S.bf16_bits(x[ridx]), packed, scales, c.N, c.K, c.g, nthreads=nth)
    ref = O.epilogue_rows(y, W.ACT_SWIGLU, bias=bias)
    assert_close_fused(bf16_to_f64(out[ridx]), y, ref, W.ACT_SWIGLU, bias, "swiglu rows")
    n_out = c.N // 2
    cols = np.array(sorted({0, n_out // 3, n_out - 1}), dtype=np.int64)
    wrows = np.stack([2 * cols, 2 * cols + 1], axis=1).ravel()      # (gate, up) per column
    mi = np.repeat(np.arange(c.M, dtype=np.int64), len(wrows))
    ni = np.tile(wrows, c.M)
    yc = O.linear_points(S.bf16_bits(x), packed, scales, c.N, c.K, c.g, mi, ni,
                         nthreads=nth).reshape(c.M, len(wrows))
    refc = O.epilogue_rows(yc, W.ACT_SWIGLU, bias=bias[wrows])
    gotc = bf16_to_f64(out[:, torch.from_numpy(cols).cuda()])
    assert_close_fused(gotc, yc, refc, W.ACT_SWIGLU, bias[wrows], "swiglu columns")
    assert W.get_device_error() == W.OK


@pytest.mark.slow
def test_fused_gelu_bias_residual_in_place_fullsize_sampled():
    """GELU + bias + residual added in place at 8192 tokens x 12288 x 12288
    (the persistent GEMM over many waves), on sampled rows and columns."""
    W = _W()
    M, N, K, g = 8192, 12288, 12288, 128
    packed, scales, wd, sd = prepare_weights(N, K, g, 5)
    x = S.make_x(M, K, 6, "cuda")
    rng = np.random.default_rng(12)
    bf = lambda a: S.bf16_bits(torch.from_numpy(a.astype(np.float32)).to(torch.bfloat16))
    bias = bf(0.5 * rng.normal(size=N))
    res = S.make_x(M, N, 13, "cuda")
    res_bits = S.bf16_bits(res)
    bias_d = torch.from_numpy(bias.view(np.int16)).view(torch.bfloat16).cuda()
    W.linear_fused(x, wd, sd, g, act=W.ACT_GELU, bias=bias_d, residual=res, out=res)
    torch.cuda.synchronize()
    nth = O.max_threads()
    rows = _rows(M)
    ridx = torch.from_numpy(rows).cuda()
    y = O.linear_rows(S.bf16_bits(x[ridx]), packed, scales, N, K, g, nthreads=nth)
    ref = O.epilogue_rows(y, W.ACT_GELU, bias=bias, residual=res_bits, rows=rows)
    assert_close_fused(bf16_to_f64(res[ridx]), y, ref, W.ACT_GELU, bias, "gelu rows")
    cols = np.array(sorted({0, N // 3, N - 1}), dtype=np.int64)
    mi = np.repeat(np.arange(M, dtype=np.int64), len(cols))
    ni = np.tile(cols, M)
    yc = O.linear_points(S.bf16_bits(x), packed, scales, N, K, g, mi, ni,
                         nthreads=nth).reshape(M, len(cols))
    refc = O.epilogue_rows(yc, W.ACT_GELU, bias=bias[cols],
                           residual=np.ascontiguousarray(res_bits[:, cols]))
    gotc = bf16_to_f64(res[:, torch.from_numpy(cols).cuda()])
    assert_close_fused(gotc, yc, refc, W.ACT_GELU, bias[cols], "gelu columns")
    assert W.get_device_error() == W.OK


@pytest.mark.slow
@pytest.mark.parametrize("M", [8, 24])
def test_fused_swiglu_small_m_readout_scale(M):
    """SwiGLU + bias + residual on the small-M streaming kernels (warp-level
    at M = 8, tensor-core at M = 24) over the full gate/up weights (K 12288 x
    2 x 49152 interleaved rows: more row chunks than SMs), on sampled output
    columns for every token."""
    W = _W()
    c = S.MLP_SWIGLU
    packed, scales, wd, sd = prepare_weights(c.N, c.K, c.g, c.w_seed)
    x = S.make_x(M, c.K, 700 + M, "cuda")
    n_out = c.N // 2
    rng = np.random.default_rng(13 + M)
    bf16 = lambda a: S.bf16_bits(torch.from_numpy(a.astype(np.float32)).to(torch.bfloat16))
    bias = bf16(0.5 * rng.normal(size=c.N))
    res = bf16(0.5 * rng.normal(size=(M, n_out)))
    to_dev = lambda b: torch.from_numpy(b.view(np.int16)).view(torch.bfloat16).cuda()
    out = W.linear_fused(x, wd, sd, c.g, act=W.ACT_SWIGLU, bias=to_dev(bias), residual=to_dev(res))
    torch.cuda.synchronize()
    cols = {0, 161, 162, 191, 192, n_out // 3, n_out // 2 + 7, n_out - 1}
    cols.update(int(v) for v in rng.integers(0, n_out, size=8))
    cols = np.array(sorted(cols), dtype=np.int64)
    wrows = np.stack([2 * cols, 2 * cols + 1], axis=1).ravel()      # (gate, up) per column
    mi = np.repeat(np.arange(M, dtype=np.int64), len(wrows))
    ni = np.tile(wrows, M)
    y = O.linear_points(S.bf16_bits(x), packed, scales, c.N, c.K, c.g, mi, ni,
                        nthreads=O.max_threads()).reshape(M, len(wrows))
    ref = O.epilogue_rows(y, W.ACT_SWIGLU, bias=bias[wrows], residual=res[:, cols])
    got = bf16_to_f64(out[:, torch.from_numpy(cols).cuda()])
    assert_close_fused(got, y, ref, W.ACT_SWIGLU, bias[wrows], f"swiglu small M={M}")
    assert W.get_device_error() == W.OK
