"""Parity of the scoring readout with the oracle: gather of one hidden state
per pair, the int4 affinity head (w4a16_linear_fused with a bias), and the
top-k of the predicted affinities (bit-exact indices and scores)."""
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


def _topk_check(scores_np, k, bf16=False):
    W = _W()
    if bf16:
        t = torch.from_numpy(scores_np.astype(np.float32)).to(torch.bfloat16)
        ref_in = O.bf16_bits_to_f32(S.bf16_bits(t))
        t = t.cuda()
    else:
        ref_in = scores_np.astype(np.float32)
        t = torch.from_numpy(ref_in).cuda()
    idx, val = W.topk_smallest(t, k)
    torch.cuda.synchronize()
    ridx, rval = O.topk_smallest(ref_in, k)
    assert idx.cpu().numpy().tolist() == ridx.tolist()
    assert val.cpu().numpy().tobytes() == rval.tobytes()


@pytest.mark.parametrize("n,k", [(1, 1), (7, 7), (8, 3), (1000, 1000), (1023, 17), (10000, 100),
                                 (200000, 1024), (200003, 1), (65536, 513)])
def test_topk_random(n, k):
    rng = np.random.default_rng(n + k)
    _topk_check((rng.normal(size=n) * 3 - 8).astype(np.float32), k)


def test_topk_ties_zeros_infinities_nan():
    rng = np.random.default_rng(3)
    s = np.round(rng.normal(size=50000), 1).astype(np.float32)    # heavy ties
    s[rng.integers(0, 50000, 200)] = -0.0
    s[rng.integers(0, 50000, 200)] = 0.0
    s[rng.integers(0, 50000, 50)] = np.inf
    s[rng.integers(0, 50000, 50)] = -np.inf
    s[rng.integers(0, 50000, 50)] = np.nan
    for k in (1, 64, 1000, 1024):
        _topk_check(s, k)
    _topk_check(np.full(5000, 2.5, dtype=np.float32), 1024)     # all equal: first k indices
    nan_tail = np.full(100, np.nan, dtype=np.float32)
    nan_tail[[5, 50]] = [1.0, -1.0]
    _topk_check(nan_tail, 10)                                     # NaNs after the numbers


def test_topk_bf16_scores():
    rng = np.random.default_rng(9)
    _topk_check((rng.normal(size=30000) - 6).astype(np.float32), 200, bf16=True)


def test_gather_rows_and_bad_index_status():
    W = _W()
    rng = np.random.default_rng(4)
    src = torch.from_numpy(rng.normal(size=(300, 520)).astype(np.float32)).to(torch.bfloat16)
    idx = np.array([299, 0, 17, 17, 150], dtype=np.int32)
    out = W.gather_rows(src.cuda(), torch.from_numpy(idx).cuda())
    torch.cuda.synchronize()
    ref, ok = O.gather_rows(S.bf16_bits(src), idx)
    assert ok and (S.bf16_bits(out) == ref).all()
    src2 = src[:, :13].contiguous()          # rows of 26 bytes: the 2-byte path
    out2 = W.gather_rows(src2.cuda(), torch.from_numpy(idx).cuda())
    torch.cuda.synchronize()
    assert (S.bf16_bits(out2) == O.gather_rows(S.bf16_bits(src2), idx)[0]).all()
    assert W.get_device_error() == W.OK
    bad = np.array([1, 300, -2], dtype=np.int32)
    out3 = W.gather_rows(src.cuda(), torch.from_numpy(bad).cuda())
    assert W.get_device_error() == W.ERR_INVALID_ARG        # recorded, then cleared
    assert W.get_device_error() == W.OK
    ref3, ok3 = O.gather_rows(S.bf16_bits(src), bad)
    assert not ok3 and (S.bf16_bits(out3) == ref3).all()


def test_scoring_readout_end_to_end():
    """Packed batch of pairs -> last token of each pair -> int4 head with a
    bias -> the k best (smallest) affinities."""
    W = _W()
    pairs, D, k = 64, 1024, 10
    rng = np.random.default_rng(12)
    lengths = rng.integers(200, 1025, size=pairs)
    last = (np.cumsum(lengths) - 1).astype(np.int32)
    M = int(lengths.sum())
    hidden = S.make_x(M, D, 21, "cpu")
    # head: 2 output rows (affinity, a second readout), int4 like every weight
    _, _, packed, scales = host_case(1, 2, D, 128, 22, 23)
    bias_bits = S.bf16_bits(torch.tensor([-7.0, 0.5]).to(torch.bfloat16))
    xd, wd, sd = to_device(hidden, packed, scales)
    g = W.gather_rows(xd, torch.from_numpy(last).cuda())
    bias = torch.from_numpy(bias_bits.view(np.int16)).view(torch.bfloat16).cuda()
    head = W.linear_fused(g, wd, sd, 128, bias=bias)
    aff = head[:, 0].contiguous()
    idx, val = W.topk_smallest(aff, k)
    torch.cuda.synchronize()
    # oracle chain
    gx, ok = O.gather_rows(S.bf16_bits(hidden), last)
    y = O.linear_rows(gx, packed, scales, 2, D, 128)
    ref = O.epilogue_rows(y, O.ACT_NONE, bias=bias_bits)
    assert_close_fused(bf16_to_f64(head), y, ref, O.ACT_NONE, bias_bits, "affinity head")
    # the top-k of the GPU's own (bf16) affinities is exact
    ridx, rval = O.topk_smallest(bf16_to_f64(aff).astype(np.float32), k)
    assert idx.cpu().numpy().tolist() == ridx.tolist()
    assert val.cpu().numpy().tobytes() == rval.tobytes()
