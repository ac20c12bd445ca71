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


def bf16_to_f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def assert_close(gpu: np.ndarray, ref: np.ndarray, what: str = ""):
    m = O.error_metrics(gpu, ref)
    assert np.isfinite(gpu).all(), f"{what}: non-finite output"
    assert m["max_err_over_rms"] <= MAX_ERR_OVER_RMS, f"{what}: {m}"
    assert m["rel_fro"] <= REL_FRO, f"{what}: {m}"
    return m
