"""Shared helpers for the GPU parity tests: seeded inputs from the synthetic
generator, oracle-side quantisation on the CPU, device uploads, tolerances."""
from __future__ import annotations

import numpy as np
import torch

from oracle import oracle as O
from paper_2608_30877_gb300 import synthetic as S

# Tolerances for one output matrix (or a sample of one), fp32 accumulation
# followed by one bf16 rounding of the output.
MAX_ERR_OVER_RMS = 2e-2
REL_FRO = 5e-3


def host_case(M, N, K, g, w_seed, x_seed):
    """CPU-generated inputs, quantised by the oracle."""
    w = S.make_w_master(N, K, w_seed, "cpu").numpy()
    x = S.make_x(M, K, x_seed, "cpu")
    packed, scales = O.quantize(w, g)
    return x, S.bf16_bits(x), packed, scales


def to_device(x_bf16, packed, scales):
    dev = torch.device("cuda")
    xd = x_bf16.to(dev)
    wd = torch.from_numpy(packed).to(dev)
    sd = torch.from_numpy(scales.view(np.int16)).view(torch.bfloat16).to(dev)
    return xd, wd, sd


def prepare_weights(N, K, g, w_seed):
    """Master weights from the generator (on the GPU), quantised on both
    sides: the oracle's bytes are the reference (and the tensors handed to
    the library), the library's quantiser must produce the same bytes."""
    from paper_2608_30877_gb300 import w4a16 as W
    master = S.make_w_master(N, K, w_seed, "cuda")
    packed_gpu, scales_gpu = W.quantize(master, g)
    host = master.cpu().numpy()
    del master
    packed, scales = O.quantize(host, g)
    del host
    assert np.array_equal(packed_gpu.cpu().numpy(), packed), "quantiser bytes differ"
    assert np.array_equal(scales_gpu.cpu().view(torch.int16).numpy().view(np.uint16), scales), \
        "quantiser scales differ"
    return packed, scales, packed_gpu, scales_gpu


def oracle_chain(x_bits, weights, g, nthreads=None):
    """The oracle's own layer chain: layer i reads the bf16 rounding (the
    oracle's RNE of the fp32 value) of the fp64 output of layer i - 1.
    weights: [(packed, scales, N, K)]; returns the fp64 outputs per layer."""
    nth = O.max_threads() if nthreads is None else nthreads
    refs, xin = [], x_bits
    for packed, scales, N, K in weights:
        ref = O.linear_rows(xin, packed, scales, N, K, g, nthreads=nth)
        refs.append(ref)
        xin = O.bf16_rne_array(ref.astype(np.float32))
    return refs


def bf16_to_f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def assert_close(gpu: np.ndarray, ref: np.ndarray, what: str = ""):
    m = O.error_metrics(gpu, ref)
    assert np.isfinite(gpu).all(), f"{what}: non-finite output"
    assert m["max_err_over_rms"] <= MAX_ERR_OVER_RMS, f"{what}: {m}"
    assert m["rel_fro"] <= REL_FRO, f"{what}: {m}"
    return m


def assert_close_chain(gpu: np.ndarray, ref: np.ndarray, depth: int, what: str = ""):
    """Layer `depth` (0-based) of a chained stack against the oracle's own
    chain.  Each layer adds its own error (the single-layer bounds) to the
    error of its input, and a layer of random N(0, 0.02) weights maps a
    relative input perturbation to about the same relative output
    perturbation, so the relative errors add: the bounds are the
    single-layer ones times depth + 1."""
    m = O.error_metrics(gpu, ref)
    assert np.isfinite(gpu).all(), f"{what}: non-finite output"
    assert m["max_err_over_rms"] <= MAX_ERR_OVER_RMS * (depth + 1), f"{what}: {m}"
    assert m["rel_fro"] <= REL_FRO * (depth + 1), f"{what}: {m}"
    return m


def assert_close_fused(gpu: np.ndarray, y: np.ndarray, ref: np.ndarray, act: int,
                       bias=None, what: str = ""):
    """Tolerance for fused-epilogue outputs h = act(y + bias) + residual.

    The plain-linear bound allows the pre-activation y an error of up to
    MAX_ERR_OVER_RMS * rms(y) per element (fp32 accumulation in any order, and
    in the small-M kernel the scale applied per group in fp32 instead of a
    bf16 rounding of every (q - 8) s).  The activation carries that error
    scaled by its derivative: 1 (none), |GELU'(z)|, and for SwiGLU
    |silu'(g) u| + |silu(g)| (gate g, up u).  On top comes the bf16 store,
    half an ulp, i.e. at most 2^-9 |ref|; the bound takes twice each term.
    The Frobenius bound is the plain one."""
    from math import sqrt
    y = np.asarray(y, dtype=np.float64)
    z = y + (0.0 if bias is None else O.bf16_bits_to_f32(np.asarray(bias)).astype(np.float64))
    eps = 2.0 * MAX_ERR_OVER_RMS * float(np.sqrt(np.mean(y * y)))
    if act == 1:
        gate, up = z[:, 0::2], z[:, 1::2]
        sig = 1.0 / (1.0 + np.exp(-gate))
        gain = np.abs(sig * (1.0 + gate * (1.0 - sig)) * up) + np.abs(gate * sig)
    elif act == 2:
        from scipy.special import erf
        gain = np.abs(0.5 * (1.0 + erf(z / sqrt(2.0))) + z * np.exp(-0.5 * z * z) / sqrt(2.0 * np.pi))
    else:
        gain = np.ones_like(z)
    m = O.error_metrics(gpu, ref)
    assert np.isfinite(gpu).all(), f"{what}: non-finite output"
    bound = 2.0 ** -8 * np.abs(ref) + eps * gain + 1e-30
    worst = float(np.max(np.abs(gpu - ref) / bound)) if ref.size else 0.0
    assert worst <= 1.0, f"{what}: worst error / bound = {worst:.3f}, {m}"
    assert m["rel_fro"] <= REL_FRO, f"{what}: {m}"
    return m
