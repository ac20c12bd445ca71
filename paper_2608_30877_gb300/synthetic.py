"""Seeded synthetic workloads for the W4A16 linear layers.

This module draws random inputs only: bf16 activations ~ N(0, 1) and fp32
master weights ~ N(0, 0.02).  It holds none of the method's arithmetic
(no quantisation, no dequantisation, no matmul), so both the CUDA library's
tests and the CPU oracle can take their inputs from it.

The paper's workload (Sec. 3.3, Sec. 4.1) is batched scoring of packed
protein-ligand token sequences through a 175B-class decoder; its dataset,
tokenizer and weights are not available, and the linear layers are token-wise,
so only the shapes and value distributions below matter.
"""
from __future__ import annotations

import dataclasses

import torch

D_MODEL = 12288
D_FF = 4 * D_MODEL
N_LAYERS = 96
GROUP = 128

# The four int4 linears of one decoder layer: (name, K, N).
LAYER_LINEARS = (
    ("qkv", D_MODEL, 3 * D_MODEL),
    ("o", D_MODEL, D_MODEL),
    ("up", D_MODEL, D_FF),
    ("down", D_FF, D_MODEL),
)


@dataclasses.dataclass(frozen=True)
class LinearCase:
    name: str
    M: int
    N: int
    K: int
    g: int
    w_seed: int
    x_seed: int


# Named workloads.  Seeds: the tiny case uses seed 0; the others use their
# index; the full stack uses 1000 + 4*layer + j for weights and
# 2000 + 4*layer + j for activations (j = 0..3 over qkv, o, up, down).
TINY = LinearCase("tiny_64x512x1024", 64, 1024, 512, GROUP, 0, 0)
QKV_PREFILL = LinearCase("qkv_prefill_4096x12288x36864", 4096, 3 * D_MODEL, D_MODEL, GROUP, 1, 1)
MLP_UP = LinearCase("mlp_up_8192x12288x49152", 8192, D_FF, D_MODEL, GROUP, 2, 2)
MLP_DOWN = LinearCase("mlp_down_8192x49152x12288", 8192, D_MODEL, D_FF, GROUP, 2, 3)
# gate and up projections as one matrix of interleaved rows (gate 2j, up 2j+1),
# run with the fused SwiGLU epilogue: [8192, 12288] -> [8192, 49152]
MLP_SWIGLU = LinearCase("mlp_swiglu_8192x12288x2x49152", 8192, 2 * D_FF, D_MODEL, GROUP, 2, 4)
GEMV_MS = (1, 8, 16, 32)


def gemv_case(M: int) -> LinearCase:
    return LinearCase(f"gemv_m{M}_12288x49152", M, D_FF, D_MODEL, GROUP, 3, 3)


STACK_PAIRS = 64
STACK_TOKENS_PER_PAIR = 1024
STACK_M = STACK_PAIRS * STACK_TOKENS_PER_PAIR


def stack_case(layer: int, j: int, M: int = STACK_M) -> LinearCase:
    name, K, N = LAYER_LINEARS[j]
    return LinearCase(f"stack_l{layer}_{name}", M, N, K, GROUP,
                      1000 + 4 * layer + j, 2000 + 4 * layer + j)


def _gen(seed: int, device) -> torch.Generator:
    dev = torch.device(device)
    g = torch.Generator(device=dev.type if dev.type == "cuda" else "cpu")
    g.manual_seed(int(seed))
    return g


def make_x(M: int, K: int, seed: int, device="cpu") -> torch.Tensor:
    """bf16 [M, K] activations, N(0, 1) drawn in fp32 and cast to bf16."""
    g = _gen(seed + 7919, device)
    x = torch.randn((M, K), generator=g, device=device, dtype=torch.float32)
    return x.to(torch.bfloat16)


def make_w_master(N: int, K: int, seed: int, device="cpu") -> torch.Tensor:
    """fp32 [N, K] master weights, N(0, 0.02)."""
    g = _gen(seed, device)
    w = torch.randn((N, K), generator=g, device=device, dtype=torch.float32)
    return w.mul_(0.02)


def bf16_bits(t: torch.Tensor):
    """bf16 tensor -> numpy uint16 bit patterns (host copy)."""
    import numpy as np
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)
