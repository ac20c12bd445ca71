"""Parity of the attention prefill (w4a16_attention_prefill) with the oracle:
causal sliding-window attention over packed sequences, d = 128, on ragged
sequence lengths (partial query and key blocks), small and large windows,
tokens outside every sequence, a bad sequence table, and the full-size
workload (64 pairs x 1024 tokens x 96 heads) on sampled query rows."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2608_30877_gb300 import synthetic as S

pytestmark = pytest.mark.gpu

D = 128


def _W():
    from paper_2608_30877_gb300 import w4a16 as W
    return W


def _check(gpu, ref, v_rms, what):
    """P is rounded to bf16 for the PV product (relative 2^-9 per weight), so
    an output moves by up to ~2^-9 rms(v); the store adds half an ulp
    (2^-9 |ref|).  Bound per element: 2^-8 |ref| + 2^-7 rms(v); Frobenius:
    ||gpu - ref|| / sqrt(n) <= 2^-9 (rms(v) + rms(ref))."""
    assert np.isfinite(gpu).all(), what
    err = np.abs(gpu - ref)
    bound = 2.0 ** -8 * np.abs(ref) + 2.0 ** -7 * v_rms
    worst = float(np.max(err / bound))
    assert worst <= 1.0, f"{what}: worst/bound {worst:.3f}, max err {err.max():.3g}"
    fro = float(np.sqrt(np.mean(err * err)))
    assert fro <= 2.0 ** -9 * (v_rms + float(np.sqrt(np.mean(ref * ref)))), f"{what}: fro {fro:.3g}"


def _case(lengths, H, window, seed, extra_tokens=0):
    W = _W()
    st = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int32)
    M = int(st[-1]) + extra_tokens
    g = torch.Generator(device="cpu").manual_seed(seed)
    qkv = torch.randn((M, 3 * H * D), generator=g).to(torch.bfloat16)
    bits = S.bf16_bits(qkv)
    out = torch.full((M, H * D), -7.0, dtype=torch.bfloat16, device="cuda")
    W.attention_prefill(qkv.cuda(), torch.from_numpy(st).cuda(), H, window, out=out)
    torch.cuda.synchronize()
    assert W.get_device_error() == W.OK
    gpu = out.float().cpu().numpy().astype(np.float64)
    v = O.bf16_bits_to_f32(bits[:, 2 * H * D:]).astype(np.float64)
    return gpu, bits, st, M, float(np.sqrt(np.mean(v * v)))


@pytest.mark.parametrize("lengths,window", [
    ([1], 32768), ([128], 32768), ([129, 5], 32768), ([300, 1, 127, 256], 32768),
    ([300, 200], 1), ([300, 200], 17), ([700], 200), ([512, 333], 128),
])
def test_attention_ragged_sequences(lengths, window):
    H = 2
    gpu, bits, st, M, v_rms = _case(lengths, H, window, sum(lengths) + window, extra_tokens=3)
    n = int(st[-1])
    ref = O.attention_rows(bits, H, D, st, window, rows=np.arange(n))
    _check(gpu[:n], ref, v_rms, f"lengths {lengths} window {window}")
    assert (gpu[n:] == -7.0).all()            # tokens outside every sequence are untouched


def test_attention_bad_sequence_table_writes_nothing():
    W = _W()
    H, M = 1, 64
    qkv = torch.randn((M, 3 * H * D), device="cuda").to(torch.bfloat16)
    out = torch.full((M, H * D), 3.0, dtype=torch.bfloat16, device="cuda")
    st = torch.tensor([0, 40, 20, 64], dtype=torch.int32, device="cuda")   # decreasing
    W.attention_prefill(qkv, st, H, 1024, out=out)
    assert W.get_device_error() == W.ERR_INVALID_ARG
    assert (out == 3.0).all()


def test_attention_full_size_sampled_rows():
    """64 pairs x 1024 tokens, 96 heads, window 32K: sampled query rows."""
    W = _W()
    H, pairs, L = 96, 64, 1024
    M = pairs * L
    st = np.arange(0, M + 1, L, dtype=np.int32)
    qkv = S.make_x(M, 3 * H * D, 77, "cuda")
    out = W.attention_prefill(qkv, torch.from_numpy(st).cuda(), H, 32768)
    torch.cuda.synchronize()
    assert W.get_device_error() == W.OK
    rows = np.array([0, 1, 127, 128, 1023, 1024, 5 * L + 517, M - 1], dtype=np.int64)
    bits = S.bf16_bits(qkv)
    ref = O.attention_rows(bits, H, D, st, 32768, rows=rows)
    gpu = out[torch.from_numpy(rows).cuda()].float().cpu().numpy().astype(np.float64)
    v = O.bf16_bits_to_f32(bits[:, 2 * H * D:]).astype(np.float64)
    _check(gpu, ref, float(np.sqrt(np.mean(v * v))), "full size")


@pytest.mark.parametrize("window", [100, 64, 32768])
def test_attention_many_short_jobs(window):
    """Hundreds of sequences of random lengths (1 to 700 tokens) and 4 heads:
    more jobs than the persistent grid has CTAs, so every CTA runs many jobs
    back to back, many of them with one or two key blocks, and the pipeline's
    barrier phases carry across job boundaries; sampled query rows of every
    length class against the oracle."""
    W = _W()
    H = 4
    rng = np.random.default_rng(window)
    lengths = rng.integers(1, 701, size=300)
    lengths[:8] = [1, 2, 63, 64, 65, 127, 128, 129]
    st = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int32)
    M = int(st[-1])
    qkv = S.make_x(M, 3 * H * D, 300 + window, "cuda")
    out = W.attention_prefill(qkv, torch.from_numpy(st).cuda(), H, window)
    torch.cuda.synchronize()
    assert W.get_device_error() == W.OK
    # the first and last rows of every eighth sequence, and random rows
    seq_rows = np.concatenate([[st[s], st[s + 1] - 1] for s in range(0, 300, 8)])
    rows = np.unique(np.concatenate([seq_rows, rng.integers(0, M, size=600)])).astype(np.int64)
    bits = S.bf16_bits(qkv)
    ref = O.attention_rows(bits, H, D, st, window, rows=rows)
    gpu = out[torch.from_numpy(rows).cuda()].float().cpu().numpy().astype(np.float64)
    v = O.bf16_bits_to_f32(bits[:, 2 * H * D:]).astype(np.float64)
    _check(gpu, ref, float(np.sqrt(np.mean(v * v))), f"many short jobs, window {window}")
