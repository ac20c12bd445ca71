"""GPU parity: the CUDA library (through its C ABI) against the CPU oracle on
the same seeded inputs.  Integer work (unpack, dequant, quantise) must be
bit-exact; linear outputs must satisfy max|gpu-ref| <= 2e-2 * rms(ref) and
||gpu-ref||_F / ||ref||_F <= 5e-3 per output matrix."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2608_30877_gb300 import synthetic as S
from tests.gpu_helpers import (assert_close, assert_close_chain, bf16_to_f64, host_case,
                               oracle_chain, to_device)

pytestmark = pytest.mark.gpu


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


# ---------------------------------------------------------------- dequant

@pytest.mark.parametrize("N,K,g", [(1024, 512, 128), (3, 64, 64), (257, 768, 256), (130, 1024, 128)])
def test_dequant_bit_exact(N, K, g):
    W = _W()
    _, _, packed, scales = host_case(1, N, K, g, 100 + N, 0)
    want = O.dequant(packed, scales, N, K, g)
    _, wd, sd = to_device(torch.zeros(1, K, dtype=torch.bfloat16), packed, scales)
    got = W.dequant(wd, sd, g)
    torch.cuda.synchronize()
    got = got.cpu().view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(got, want)


def test_dequant_every_code_and_rounding_case():
    W = _W()
    scales_f = [1.0, 1.0 + 2 ** -7, 0.0078125, 0.10009765625, 3.0, -0.5, 0.0,
                0.0014982223510742188, 0.02099609375, 1.5, 6.5e-3, 250.0, -7.25e-3, 1e-30]
    N, K, g = len(scales_f), 64, 64
    q = np.tile(np.arange(16, dtype=np.uint8), 4)[None, :].repeat(N, 0)
    packed = O.pack(q)
    scales = np.array([[O.bf16_rne(s)] for s in scales_f], np.uint16)
    want = O.dequant(packed, scales, N, K, g)
    _, wd, sd = to_device(torch.zeros(1, K, dtype=torch.bfloat16), packed, scales)
    got = W.dequant(wd, sd, g).cpu().view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(got, want)


# ---------------------------------------------------------------- quantise

def test_quantize_bit_exact_tiny_and_adversarial():
    W = _W()
    N, K, g = 1024, 512, 128
    w = S.make_w_master(N, K, 0, "cpu").numpy()
    # adversarial groups: all zero, exact ties, +-amax, tiny values
    w[0, :128] = 0.0
    w[1, :5] = [7.0, 2.5, -2.5, 3.5, -0.5]
    w[1, 5:128] = 0.0
    w[2, :128] = np.linspace(-1, 1, 128, dtype=np.float32)
    w[3, :128] = 1e-30
    want_p, want_s = O.quantize(w, g)
    got_p, got_s = W.quantize(torch.from_numpy(w).cuda(), g)
    assert np.array_equal(got_p.cpu().numpy(), want_p)
    assert np.array_equal(got_s.cpu().view(torch.int16).numpy().view(np.uint16), want_s)


# ---------------------------------------------------------------- linear

def _run_linear(M, N, K, g, seed=0):
    W = _W()
    x, xb, packed, scales = host_case(M, N, K, g, seed, seed + 1)
    xd, wd, sd = to_device(x, packed, scales)
    out = W.linear(xd, wd, sd, g)
    torch.cuda.synchronize()
    ref = O.linear_rows(xb, packed, scales, N, K, g, nthreads=O.max_threads())
    return bf16_to_f64(out), ref


def test_linear_tiny_config_full():
    gpu, ref = _run_linear(64, 1024, 512, 128, seed=0)
    assert_close(gpu, ref, "tiny 64x512x1024")


@pytest.mark.parametrize("M,N,K,g", [
    (1, 128, 128, 128), (5, 200, 256, 128), (32, 384, 512, 128), (33, 300, 384, 128),
    (257, 130, 640, 128), (300, 1000, 1024, 128), (512, 256, 2048, 128),
    (40, 256, 256, 64), (100, 512, 1024, 256), (7, 129, 192, 64), (600, 2, 128, 128),
    (256, 1, 256, 128), (31, 77, 320, 64),
])
def test_linear_ragged_shapes(M, N, K, g):
    gpu, ref = _run_linear(M, N, K, g, seed=M * 7 + N)
    assert_close(gpu, ref, f"{M}x{K}x{N} g{g}")


def test_linear_m_sweep_around_dispatch_threshold():
    W = _W()
    N, K, g = 256, 512, 128
    x, xb, packed, scales = host_case(134, N, K, g, 77, 78)
    xd, wd, sd = to_device(x, packed, scales)
    ref = O.linear_rows(xb, packed, scales, N, K, g, nthreads=O.max_threads())
    for M in range(1, 135):
        out = W.linear(xd[:M].contiguous(), wd, sd, g)
        assert_close(bf16_to_f64(out), ref[:M], f"M={M}")


def test_linear_guard_bands_untouched():
    W = _W()
    M, N, K, g = 67, 258, 256, 128
    x, xb, packed, scales = host_case(M, N, K, g, 5, 6)
    xd, wd, sd = to_device(x, packed, scales)
    guard = 4096
    buf = torch.full((guard + M * N + guard,), -12345.0, dtype=torch.bfloat16, device="cuda")
    out = buf[guard:guard + M * N].view(M, N)
    W.linear(xd, wd, sd, g, out=out)
    torch.cuda.synchronize()
    assert (buf[:guard] == -12345.0).all() and (buf[guard + M * N:] == -12345.0).all()
    ref = O.linear_rows(xb, packed, scales, N, K, g, nthreads=O.max_threads())
    assert_close(bf16_to_f64(out), ref, "guarded")


def test_linear_deterministic():
    W = _W()
    x, xb, packed, scales = host_case(300, 512, 1024, 128, 9, 10)
    xd, wd, sd = to_device(x, packed, scales)
    a = W.linear(xd, wd, sd)
    b = W.linear(xd, wd, sd)
    assert torch.equal(a.view(torch.int16), b.view(torch.int16))


def test_linear_stack_chained_and_fresh():
    W = _W()
    g, M = 128, 96
    dims = [(256, 512), (512, 384), (384, 256)]   # (K, N) per layer; layer i+1 reads layer i's out
    refs, layers = [], []
    x0, x0b, _, _ = host_case(M, 1, dims[0][0], g, 0, 500)
    xin = x0.cuda()
    for i, (K, N) in enumerate(dims):
        w = S.make_w_master(N, K, 600 + i, "cpu").numpy()
        packed, scales = O.quantize(w, g)
        _, wd, sd = to_device(torch.zeros(1, K, dtype=torch.bfloat16), packed, scales)
        out = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
        layers.append((xin, wd, sd, out))
        refs.append((packed, scales, N, K))
        xin = out
    W.linear_stack(layers, M, g)
    torch.cuda.synchronize()
    # each layer against the oracle's own chain (layer i reads the oracle's
    # bf16 rounding of its layer i - 1), with the chain's depth-aware bound
    chain = oracle_chain(x0b, refs, g)
    for i, (_, _, _, out) in enumerate(layers):
        assert_close_chain(bf16_to_f64(out), chain[i], i, f"stack layer {i}")


def test_error_codes_launch_nothing():
    W = _W()
    L = W.lib()
    x = torch.zeros((4, 256), dtype=torch.bfloat16, device="cuda")
    w = torch.zeros((8, 128), dtype=torch.uint8, device="cuda")
    s = torch.zeros((8, 2), dtype=torch.bfloat16, device="cuda")
    o = torch.full((4, 8), 7.0, dtype=torch.bfloat16, device="cuda")
    st = torch.cuda.current_stream().cuda_stream
    args = [x.data_ptr(), w.data_ptr(), s.data_ptr(), o.data_ptr()]
    assert L.w4a16_linear(*args, 0, 8, 256, 128, st) == W.ERR_INVALID_ARG
    assert L.w4a16_linear(*args, 4, 8, 256, 96, st) == W.ERR_INVALID_ARG       # K % g
    assert L.w4a16_linear(*args, 4, 8, 256, 32, st) == W.ERR_UNSUPPORTED      # g % 64
    assert L.w4a16_linear(x.data_ptr() + 2, *args[1:], 4, 8, 256, 128, st) == W.ERR_ALIGNMENT
    assert L.w4a16_linear(*args[:3], x.data_ptr(), 4, 8, 256, 128, st) == W.ERR_INVALID_ARG  # overlap
    torch.cuda.synchronize()
    assert (o == 7.0).all()


@pytest.mark.parametrize("M,N,K,g", [
    (1, 1, 128, 128), (3, 100, 256, 128), (8, 1000, 1024, 128), (16, 4096, 512, 128),
    (17, 1234, 384, 128), (32, 8192, 256, 64), (32, 50000, 128, 128), (9, 77, 2048, 256),
    (8, 60000, 640, 128), (24, 60000, 1152, 128), (2, 53600, 2176, 128),
    (20, 1, 128, 128), (29, 130, 128, 128), (33, 130, 384, 128), (48, 60010, 256, 128),
    (64, 1, 128, 128), (64, 4100, 1152, 128), (100, 60010, 256, 128), (128, 1, 128, 128),
    (72, 4100, 1152, 128),
])
def test_small_m_streaming_kernel_shapes(M, N, K, g):
    """M <= 128 with g = 128 runs a row-range streaming kernel: ragged row
    ranges, 8 to 128 token columns, group counts that leave padding stages
    in the last round of stage slots, and N large enough that a CTA takes a
    second row range (more row ranges than SMs)."""
    gpu, ref = _run_linear(M, N, K, g, seed=3 * M + N)
    assert_close(gpu, ref, f"{M}x{K}x{N} g{g}")


_FORCED_KERNEL_CHECK = r"""
import sys
import numpy as np, torch
sys.path.insert(0, {root!r})
from oracle import oracle as O
from tests.gpu_helpers import assert_close, bf16_to_f64, host_case, to_device
from paper_2608_30877_gb300 import w4a16 as W
for (M, N, K) in {cases!r}:
    x, xb, packed, scales = host_case(M, N, K, 128, 300 + M, 301 + M)
    xd, wd, sd = to_device(x, packed, scales)
    out = W.linear(xd, wd, sd, 128)
    torch.cuda.synchronize()
    ref = O.linear_rows(xb, packed, scales, N, K, 128, nthreads=O.max_threads())
    assert_close(bf16_to_f64(out), ref, f"M={{M}} N={{N}} K={{K}}")
assert W.get_device_error() == W.OK
print("ok")
"""


@pytest.mark.parametrize("kernel", ["tc", "mma"])
def test_small_m_kernels_every_m(kernel):
    """Both small-M streaming kernels at every M they can be forced to
    (W4A16_SMALL_M), on ragged shapes: the dispatch picks one by M, and
    each must be correct everywhere."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    Ms = (1, 2, 5, 8, 13, 16, 17, 24, 31, 32) + ((33, 40, 57, 64, 65, 99, 128) if kernel == "tc"
                                                 else ())
    cases = [(M, 1000 + 2 * M, 384 if M % 2 else 1280) for M in Ms]
    env = dict(os.environ, W4A16_SMALL_M=kernel)
    r = subprocess.run([sys.executable, "-c", _FORCED_KERNEL_CHECK.format(root=root, cases=cases)],
                       env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0 and "ok" in r.stdout, r.stdout + r.stderr


@pytest.mark.parametrize("kernel", ["tc", "mma"])
def test_small_m_kernels_several_chunks_per_cta(kernel):
    """More weight rows than one row range per SM can hold (RB is capped at
    384 rows for the tensor-core kernel, 352 for the warp-level one), so some
    CTAs walk a second chunk: the tensor-core kernel's accumulator hand-off
    between chunks and both kernels' stage rings across chunks, on every
    output against the oracle."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    cases = [(M, 60010, 256) for M in (3, 16, 24, 32) + ((40, 64, 96, 128) if kernel == "tc" else ())]
    env = dict(os.environ, W4A16_SMALL_M=kernel)
    r = subprocess.run([sys.executable, "-c", _FORCED_KERNEL_CHECK.format(root=root, cases=cases)],
                       env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0 and "ok" in r.stdout, r.stdout + r.stderr


_FORCED_GEMM_CHECK = r"""
import sys
import numpy as np, torch
sys.path.insert(0, {root!r})
from oracle import oracle as O
from paper_2608_30877_gb300 import synthetic as S
from tests.gpu_helpers import assert_close, bf16_to_f64, host_case, to_device
from paper_2608_30877_gb300 import w4a16 as W
for (M, N, K) in {cases!r}:
    x, xb, packed, scales = host_case(M, N, K, 128, 500 + M, 501 + N)
    xd, wd, sd = to_device(x, packed, scales)
    out = W.linear(xd, wd, sd, 128)
    torch.cuda.synchronize()
    ref = O.linear_rows(xb, packed, scales, N, K, 128, nthreads=O.max_threads())
    assert_close(bf16_to_f64(out), ref, f"M={{M}} N={{N}} K={{K}}")
assert W.get_device_error() == W.OK
# the abort path under a lowered wait limit, then a correct call again
W.set_wait_limit(1)
W.linear(S.make_x(900, 2048, 3, "cuda"), torch.zeros((128 * 300, 1024), dtype=torch.uint8,
         device="cuda"), torch.zeros((128 * 300, 16), dtype=torch.bfloat16, device="cuda"), 128)
assert W.get_device_error() == W.ERR_TIMEOUT
W.set_wait_limit(0)
x, xb, packed, scales = host_case(500, 384, 512, 128, 7, 8)
xd, wd, sd = to_device(x, packed, scales)
out = W.linear(xd, wd, sd, 128)
torch.cuda.synchronize()
assert_close(bf16_to_f64(out), O.linear_rows(xb, packed, scales, 384, 512, 128), "after abort")
assert W.get_device_error() == W.OK
print("ok")
"""


@pytest.mark.parametrize("env", [{"W4A16_GEMM_WIDE": "1"}, {"W4A16_GEMM_WIDE": "0"},
                                 {"W4A16_GEMM_PAIR": "0"}])
def test_large_m_gemm_variants_ragged(env):
    """Every large-M GEMM variant forced on ragged shapes (ragged token tiles,
    an odd number of 128-row weight tiles, K not a multiple of the 384-token
    tile's stage count), then its abort path: the 384-token CTA pairs (the
    default from 16384 tokens), the 256-token CTA pairs and one CTA per tile."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    cases = [(33, 128, 128), (300, 384, 256), (385, 1000, 640), (769, 640, 1152), (1200, 2048, 512)]
    r = subprocess.run([sys.executable, "-c", _FORCED_GEMM_CHECK.format(root=root, cases=cases)],
                       env=dict(os.environ, **env), capture_output=True, text=True, timeout=600)
    assert r.returncode == 0 and "ok" in r.stdout, r.stdout + r.stderr
