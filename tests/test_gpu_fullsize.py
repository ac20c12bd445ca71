"""Full-size parity, in the launch configuration bench.py times.

Each workload is generated on the GPU from its seeds (fp32 master weights
N(0, 0.02), bf16 activations N(0, 1)).  The oracle quantises the same master
weights on the CPU; the library's quantiser must produce the same bytes, and
the library's linear (fed those bytes) is checked against the oracle's fp64
result on sampled outputs: whole rows (every n for a token) and whole
columns (every token for an n), including the last token and the last row so
that ragged tiles are covered."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2608_30877_gb300 import synthetic as S
from tests.gpu_helpers import assert_close, bf16_to_f64, prepare_weights

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_30877_gb300 import w4a16 as W
    W.lib()
    yield
    assert W.get_device_error() == W.OK


def _W():
    from paper_2608_30877_gb300 import w4a16 as W
    return W


def _prepare(N, K, g, w_seed):
    return prepare_weights(N, K, g, w_seed)


def _sample_rows(M, k=6):
    rows = {0, M - 1, M // 2, min(M - 1, 255), min(M - 1, 257)}
    rng = np.random.default_rng(M)
    rows.update(int(v) for v in rng.integers(0, M, size=k))
    return np.array(sorted(rows), dtype=np.int64)


def _check_linear(M, N, K, g, w_seed, x_seed, what, col_samples=3):
    W = _W()
    packed, scales, wd, sd = _prepare(N, K, g, w_seed)
    x = S.make_x(M, K, x_seed, "cuda")
    out = W.linear(x, wd, sd, g)
    torch.cuda.synchronize()
    nth = O.max_threads()
    rows = _sample_rows(M)
    xb_rows = S.bf16_bits(x[torch.from_numpy(rows).cuda()])
    ref = O.linear_rows(xb_rows, packed, scales, N, K, g, nthreads=nth)
    got = bf16_to_f64(out[torch.from_numpy(rows).cuda()])
    for i in range(len(rows)):
        assert_close(got[i], ref[i], f"{what} row {rows[i]}")
    if col_samples:
        cols = np.array(sorted({0, N - 1, N // 3}))[:col_samples]
        xb = S.bf16_bits(x)
        mi = np.repeat(np.arange(M, dtype=np.int64), len(cols))
        ni = np.tile(cols, M)
        refc = O.linear_points(xb, packed, scales, N, K, g, mi, ni, nthreads=nth).reshape(M, -1)
        gotc = bf16_to_f64(out[:, torch.from_numpy(cols).cuda()])
        for j in range(len(cols)):
            assert_close(gotc[:, j], refc[:, j], f"{what} column {cols[j]}")
    del out, x, wd, sd
    torch.cuda.empty_cache()


def test_qkv_prefill_4096x12288x36864():
    c = S.QKV_PREFILL
    _check_linear(c.M, c.N, c.K, c.g, c.w_seed, c.x_seed, c.name)


def test_mlp_up_8192x12288x49152():
    c = S.MLP_UP
    _check_linear(c.M, c.N, c.K, c.g, c.w_seed, c.x_seed, c.name, col_samples=2)


def test_mlp_down_8192x49152x12288():
    c = S.MLP_DOWN
    _check_linear(c.M, c.N, c.K, c.g, c.w_seed, c.x_seed, c.name, col_samples=2)


def test_small_m_all_outputs():
    W = _W()
    c = S.gemv_case(32)
    packed, scales, wd, sd = _prepare(c.N, c.K, c.g, c.w_seed)
    x = S.make_x(32, c.K, c.x_seed, "cuda")
    ref = O.linear_rows(S.bf16_bits(x), packed, scales, c.N, c.K, c.g, nthreads=O.max_threads())
    for M in S.GEMV_MS + (3, 17):
        out = W.linear(x[:M].contiguous(), wd, sd, c.g)
        torch.cuda.synchronize()
        assert_close(bf16_to_f64(out), ref[:M], f"small-M M={M}")


@pytest.mark.parametrize("layer", [0, 95])
def test_stack_layer_sampled_rows(layer):
    """One layer of the 175B-class stack (M = 65536), each linear against the
    oracle on sampled token rows, run through w4a16_linear_stack."""
    W = _W()
    M = S.STACK_M
    layers, preps, xs = [], [], []
    for j in range(4):
        c = S.stack_case(layer, j)
        packed, scales, wd, sd = _prepare(c.N, c.K, c.g, c.w_seed)
        x = S.make_x(M, c.K, c.x_seed, "cuda")
        out = torch.empty((M, c.N), dtype=torch.bfloat16, device="cuda")
        layers.append((x, wd, sd, out))
        preps.append((c, packed, scales))
    W.linear_stack(layers, M, 128)
    torch.cuda.synchronize()
    rows = _sample_rows(M, k=3)
    ridx = torch.from_numpy(rows).cuda()
    for (x, _, _, out), (c, packed, scales) in zip(layers, preps):
        ref = O.linear_rows(S.bf16_bits(x[ridx]), packed, scales, c.N, c.K, c.g,
                            nthreads=O.max_threads())
        got = bf16_to_f64(out[ridx])
        for i in range(len(rows)):
            assert_close(got[i], ref[i], f"{c.name} row {rows[i]}")
    del layers
    torch.cuda.empty_cache()
