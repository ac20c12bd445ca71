"""The W4A16_DEBUG build on the GPU: every kernel runs its index checks (TMA
coordinates and destinations, tensor-memory columns, store rows) on ragged
shapes of every dispatch path, no check fails, and the results still match
the oracle.  Runs in a child process that loads libw4a16_debug.so."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

_CHILD = r"""
import sys
import numpy as np, torch
sys.path.insert(0, {root!r})
from oracle import oracle as O
from paper_2608_30877_gb300 import synthetic as S
from paper_2608_30877_gb300 import w4a16 as W
from tests.gpu_helpers import assert_close, bf16_to_f64, host_case, to_device
assert W.LIB_PATH.endswith("libw4a16_debug.so"), W.LIB_PATH
# (M, N, K, g): CTA-pair GEMM with a ragged last pair, warp-level and
# tensor-core small-M kernels (32, 64 and 128 token columns), 32-token tiles
# (g = 64)
for (M, N, K, g) in [(300, 1000, 1024, 128), (520, 384, 512, 128), (8, 2000, 1280, 128),
                     (24, 1234, 640, 128), (48, 1234, 640, 128), (100, 1234, 640, 128),
                     (5, 200, 256, 64)]:
    x, xb, packed, scales = host_case(M, N, K, g, M + 1, N + 2)
    xd, wd, sd = to_device(x, packed, scales)
    out = W.linear(xd, wd, sd, g)
    torch.cuda.synchronize()
    ref = O.linear_rows(xb, packed, scales, N, K, g, nthreads=O.max_threads())
    assert_close(bf16_to_f64(out), ref, f"debug build {{M}}x{{N}}x{{K}} g{{g}}")
    assert W.get_device_error() == W.OK, (M, N, K, g)
# attention over ragged sequences
H = 2
st = torch.tensor([0, 100, 300, 301, 700], dtype=torch.int32)
qkv = S.make_x(700, 3 * H * 128, 4, "cpu")
out = W.attention_prefill(qkv.cuda(), st.cuda(), H, 160)
torch.cuda.synchronize()
assert W.get_device_error() == W.OK
bits = S.bf16_bits(qkv)
ref = O.attention_rows(bits, H, 128, st.numpy().astype(np.int64), 160)
v = O.bf16_bits_to_f32(bits[:, 2 * H * 128:]).astype(np.float64)
v_rms = float(np.sqrt(np.mean(v * v)))
err = np.abs(bf16_to_f64(out) - ref)
# the attention tests' bound: P rounded to bf16 for PV, one bf16 store
assert float(np.max(err / (2.0 ** -8 * np.abs(ref) + 2.0 ** -7 * v_rms))) <= 1.0
print("ok")
"""


def test_debug_build_checks_pass_and_results_match():
    from paper_2608_30877_gb300 import build as B
    B.build(debug=True)
    env = dict(os.environ, W4A16_DEBUG="1")
    r = subprocess.run([sys.executable, "-c", _CHILD.format(root=ROOT)], env=env,
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0 and "ok" in r.stdout, r.stdout[-3000:] + r.stderr[-3000:]
