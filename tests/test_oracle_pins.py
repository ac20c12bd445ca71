"""Pins for the CPU oracle: checked against values fixed by the format's
definition and by arithmetic, never against the oracle's own code.

The paper prints no worked example for the int4 path (Sec. 3.1 and Sec. 4.1
say only "4-bit pre-quantized"), so the pins are: hand-computed cases,
an independent exact-rational rounding, closed forms, textbook matmul on
inputs where every step is exact, and invariants.  Each is chosen so that a
plausible slip (swapped nibbles, a dropped zero point, a wrong group index,
a transposed operand, round-half-away instead of half-even) fails one.
"""
import math
import struct
from fractions import Fraction

import numpy as np
import pytest

from oracle import oracle as O

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


# ---- independent bf16 rounding, written in exact rationals ----------------

def _f32_bits(v: float) -> int:
    return struct.unpack("<I", struct.pack("<f", v))[0]


def _f32_from_bits(b: int) -> float:
    return struct.unpack("<f", struct.pack("<I", b & 0xFFFFFFFF))[0]


def _bf16_value(bits: int) -> Fraction:
    """Exact value of a finite bf16 bit pattern."""
    sign = -1 if bits & 0x8000 else 1
    e = (bits >> 7) & 0xFF
    m = bits & 0x7F
    if e == 0:
        return sign * Fraction(m, 1 << 7) * Fraction(1, 1 << 126)
    return sign * (1 + Fraction(m, 1 << 7)) * (Fraction(2) ** (e - 127))


def ref_bf16_rne(v: Fraction) -> int:
    """Nearest bf16 to the exact rational v, ties to the even significand.
    Found by searching the ordered bf16 magnitudes, independent of any bit trick."""
    sign = 0x8000 if v < 0 else 0
    a = -v if v < 0 else v
    if a == 0:
        return sign
    # exponent window: quantum of bf16 in [2^e, 2^(e+1)) is 2^(e-7); subnormal quantum 2^-133
    e = math.floor(math.log2(a)) if a > 0 else -200
    # correct floating error of log2 on huge/small rationals
    while Fraction(2) ** e > a:
        e -= 1
    while Fraction(2) ** (e + 1) <= a:
        e += 1
    e = max(e, -126)
    quantum = Fraction(2) ** (e - 7)
    n = a / quantum
    lo = math.floor(n)
    rem = n - lo
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and lo % 2 == 1):
        lo += 1
    mag = lo * quantum
    if mag >= Fraction(2) ** 128 - Fraction(2) ** 120:  # at or past the rounding boundary of the max
        return sign | 0x7F80
    # encode mag as bf16 bits
    if mag < Fraction(2) ** -126:
        return sign | int(mag / Fraction(2) ** -133)
    ee = e if mag < Fraction(2) ** (e + 1) else e + 1
    mant = int((mag / Fraction(2) ** ee - 1) * 128)
    return sign | ((ee + 127) << 7) | mant


def test_bf16_rne_hand_values():
    assert O.bf16_rne(1.0) == 0x3F80
    assert O.bf16_rne(1.0 + 2 ** -8) == 0x3F80            # exact tie, even side is 1.0
    assert O.bf16_rne(1.0 + 3 * 2 ** -8) == 0x3F82        # exact tie, even side is 1+2^-6
    assert O.bf16_rne(1.0 + 2 ** -8 + 2 ** -20) == 0x3F81  # just above the tie
    assert O.bf16_rne(-(1.0 + 2 ** -8)) == 0xBF80
    assert O.bf16_rne(0.1) == 0x3DCD                      # 0.10009765625
    assert O.bf16_rne(-0.0) == 0x8000
    assert O.bf16_rne(_f32_from_bits(0x7F7FFFFF)) == 0x7F80  # fp32 max rounds to +inf
    assert O.bf16_rne(_f32_from_bits(0x7F7F7FFF)) == 0x7F7F  # just below the midpoint


def test_bf16_rne_matches_exact_rational_rounding():
    rng = np.random.default_rng(1234)
    bits = rng.integers(0, 2 ** 32, size=6000, dtype=np.uint64).astype(np.uint32)
    # add every tie pattern shape: low 16 bits exactly 0x8000, with odd and even kept parts
    ties = (rng.integers(0, 2 ** 16, size=2000, dtype=np.uint64).astype(np.uint32) << 16) | 0x8000
    for b in np.concatenate([bits, ties]):
        b = int(b)
        if (b & 0x7F800000) == 0x7F800000:
            continue  # inf / NaN handled by the hand values
        v = _f32_from_bits(b)
        exact = Fraction(v)
        assert O.bf16_rne(v) == ref_bf16_rne(exact), hex(b)


# ---- packing ------------------------------------------------------------

def test_unpack_every_byte():
    packed = np.arange(256, dtype=np.uint8).reshape(1, 256)
    q = O.unpack(packed, 1, 512)
    for b in range(256):
        assert q[0, 2 * b] == (b & 0xF)        # even k -> bits 0..3
        assert q[0, 2 * b + 1] == (b >> 4)     # odd k  -> bits 4..7
    assert tuple(O.unpack(np.array([[0xA3]], np.uint8), 1, 2)[0]) == (3, 10)


def test_pack_unpack_round_trip():
    rng = np.random.default_rng(7)
    q = rng.integers(0, 16, size=(5, 96), dtype=np.uint8)
    assert np.array_equal(O.unpack(O.pack(q), 5, 96), q)
    packed = rng.integers(0, 256, size=(3, 40), dtype=np.uint8)
    assert np.array_equal(O.pack(O.unpack(packed, 3, 80)), packed)


# ---- dequantisation -----------------------------------------------------

SCALES = [1.0, 1.0 + 2 ** -7, 0.0078125, 0.10009765625, 3.0, -0.5, 0.0,
          0.0014982223510742188, 0.02099609375, 1.5, 6.5e-3, 250.0]


def test_dequant_table_all_codes_against_exact_product():
    s_bits = np.array([O.bf16_rne(s) for s in SCALES], dtype=np.uint16)
    N, K, g = len(SCALES), 16 * 2, 32            # each row: every code twice, one group
    q = np.tile(np.arange(16, dtype=np.uint8), 2)[None, :].repeat(N, 0)
    packed = O.pack(q)
    wd = O.dequant(packed, s_bits[:, None], N, K, g)
    for n in range(N):
        s = _bf16_value(int(s_bits[n]))
        for k in range(K):
            exact = Fraction(int(q[n, k]) - 8) * s
            want = ref_bf16_rne(exact)
            if exact == 0:
                # IEEE product sign: (q-8) is +0 when q == 8, so the sign is
                # negative exactly when one factor is negative
                neg = (int(q[n, k]) - 8 < 0) != bool(s_bits[n] & 0x8000)
                want = 0x8000 if neg else 0x0000
            assert wd[n, k] == want, (n, k)


def test_dequant_rounding_cases_by_hand():
    s = O.bf16_rne(1.0 + 2 ** -7)
    assert s == 0x3F81
    packed = O.pack(np.array([[15, 11, 0, 8]], dtype=np.uint8))
    wd = O.bf16_bits_to_f32(O.dequant(packed, np.array([[s]], np.uint16), 1, 4, 4))[0]
    assert wd[0] == 7.0625       # 7 * 1.0078125 = 7.0546875 rounds up (ulp 1/32)
    assert wd[1] == 3.03125      # 3 * 1.0078125 = 3.0234375 is a tie -> even significand
    assert wd[2] == -8.0625      # exact
    assert wd[3] == 0.0


def test_dequant_group_index():
    # K=256, g=64: 4 groups per row with scales 1, 2, 4, 8; all codes 9 (q-8 = 1)
    q = np.full((2, 256), 9, np.uint8)
    scales = np.array([[O.bf16_rne(v) for v in (1.0, 2.0, 4.0, 8.0)]] * 2, np.uint16)
    wd = O.bf16_bits_to_f32(O.dequant(O.pack(q), scales, 2, 256, 64))
    assert np.array_equal(wd[0], np.repeat([1.0, 2.0, 4.0, 8.0], 64).astype(np.float32))


# ---- linear -------------------------------------------------------------

def _bits(a):
    return np.array([O.bf16_rne(float(v)) for v in np.ravel(a)], np.uint16).reshape(np.shape(a))


def test_linear_hand_computed_2x3x256():
    K, g = 256, 128
    x = np.zeros((2, K), np.float32)
    x[0, :] = 1.0
    x[1, 0::2] = 1.0                                   # even k only
    q = np.zeros((3, K), np.uint8)
    q[0, :] = 9                                        # q-8 = 1
    q[1, 0::2], q[1, 1::2] = 15, 0                     # +7 on even k, -8 on odd k
    q[2, :] = np.arange(K) % 16
    s = np.array([[1.0, 2.0], [0.5, 0.25], [1 / 16, 1 / 8]])
    out = O.linear_rows(_bits(x), O.pack(q), _bits(s), 3, K, g)
    # row 0 of x (all ones): sum of the dequantised weights
    #   n=0: 128*1 + 128*2 = 384
    #   n=1: 64*(3.5-4) + 64*(1.75-2) = -48
    #   n=2: 8 * sum_{c=0..15}(c-8) * (1/16 + 1/8) = 8*(-8)*(3/16) = -12
    # row 1 (ones on even k): n=0: 64*1 + 64*2 = 192; n=1: 64*3.5 + 64*1.75 = 336;
    #   n=2: even codes 0,2,..,14 -> sum(c-8) = -8 per 16 k -> 8*(-8)*(3/16) = -12
    assert out.tolist() == [[384.0, -48.0, -12.0], [192.0, 336.0, -12.0]]


def test_linear_power_of_two_scales_equals_textbook_matmul():
    rng = np.random.default_rng(42)
    M, N, K, g = 7, 11, 512, 128
    x = rng.integers(-4, 5, size=(M, K)).astype(np.float32)       # exact in bf16
    q = rng.integers(0, 16, size=(N, K), dtype=np.uint8)
    e = rng.integers(-8, 3, size=(N, K // g))
    s = np.ldexp(1.0, e)
    out = O.linear_rows(_bits(x), O.pack(q), _bits(s), N, K, g)
    wd = (q.astype(np.float64) - 8.0) * np.repeat(s, g, axis=1)  # exact
    assert np.array_equal(out, x.astype(np.float64) @ wd.T)
    # and as integers: scale everything by 2^8
    wi = (q.astype(np.int64) - 8) * np.repeat(np.ldexp(1, e + 8).astype(np.int64), g, axis=1)
    xi = x.astype(np.int64)
    assert np.array_equal((out * 256).astype(np.int64), xi @ wi.T)


def test_linear_invariants():
    rng = np.random.default_rng(3)
    M, N, K, g = 4, 6, 256, 128
    q = rng.integers(0, 16, size=(N, K), dtype=np.uint8)
    s = _bits(rng.uniform(0.001, 0.02, size=(N, K // g)))
    x = _bits(rng.normal(size=(M, K)))
    ref = O.linear_rows(x, O.pack(q), s, N, K, g)
    # zero activations -> zero output
    assert not O.linear_rows(np.zeros_like(x), O.pack(q), s, N, K, g).any()
    # all codes 8 -> zero output
    assert not O.linear_rows(x, O.pack(np.full_like(q, 8)), s, N, K, g).any()
    # doubling x (exact in bf16) doubles the output exactly
    x2 = _bits(2.0 * O.bf16_bits_to_f32(x))
    assert np.array_equal(O.linear_rows(x2, O.pack(q), s, N, K, g), 2.0 * ref)
    # a zero-scale group contributes nothing: same as zeroing x over that group
    s0 = s.copy(); s0[:, 1] = 0
    xz = x.copy(); xz[:, g:2 * g] = 0
    a = O.linear_rows(x, O.pack(q), s0, N, K, g)
    b = O.linear_rows(xz, O.pack(q), s, N, K, g)
    assert np.array_equal(a, b)
    # points agree with rows
    mi = np.array([0, 3, 2]); ni = np.array([5, 0, 4])
    assert np.array_equal(O.linear_points(x, O.pack(q), s, N, K, g, mi, ni), ref[mi, ni])


def test_linear_brute_force_small():
    rng = np.random.default_rng(11)
    M, N, K, g = 2, 3, 128, 128
    q = rng.integers(0, 16, size=(N, K), dtype=np.uint8)
    s = _bits(rng.uniform(0.001, 0.05, size=(N, 1)))
    x = _bits(rng.normal(size=(M, K)))
    out = O.linear_rows(x, O.pack(q), s, N, K, g)
    xs = [[_bf16_value(int(b)) for b in row] for row in x]
    for m in range(M):
        for n in range(N):
            sv = _bf16_value(int(s[n, 0]))
            acc = Fraction(0)
            for k in range(K):
                wd = _bf16_value(ref_bf16_rne(Fraction(int(q[n, k]) - 8) * sv)) if q[n, k] != 8 else Fraction(0)
                acc += xs[m][k] * wd
            # fp64 accumulation of 128 products: within 128 ulps of the exact sum
            assert abs(Fraction(out[m, n]) - acc) <= abs(acc) * Fraction(128, 2 ** 52) + Fraction(1, 2 ** 60)


# ---- quantiser ----------------------------------------------------------

def test_quantize_hand_example():
    g = 128
    w = np.zeros((1, g), np.float32)
    w[0, :3] = [0.7, -0.35, 0.1]
    packed, scales = O.quantize(w, g)
    # amax/7 = 0.1 in fp32 -> bf16 0x3DCD = 0.10009765625
    assert scales[0, 0] == 0x3DCD
    q = O.unpack(packed, 1, g)[0]
    # 0.7/0.10009765625 = 6.993 -> 7; -0.35/.. = -3.497 -> -3; 0.1/.. = 0.999 -> 1; zeros -> 0
    assert q[:4].tolist() == [15, 5, 9, 8]
    assert (q[3:] == 8).all()


def test_quantize_rounds_half_to_even_and_zero_group():
    g = 64
    w = np.zeros((2, g), np.float32)
    w[0, :5] = [7.0, 2.5, -2.5, 3.5, -0.5]     # amax 7 -> s = 1 exactly
    packed, scales = O.quantize(w, g)
    assert scales[0, 0] == 0x3F80
    q = O.unpack(packed, 2, g)
    assert q[0, :5].tolist() == [15, 10, 6, 12, 8]   # 7, 2, -2, 4, -0 (half-even)
    assert scales[1, 0] == 0 and (q[1] == 8).all()  # all-zero group


def test_quantize_error_bound_and_code_range():
    rng = np.random.default_rng(5)
    N, K, g = 16, 1024, 128
    w = (rng.normal(size=(N, K)) * 0.02).astype(np.float32)
    packed, scales = O.quantize(w, g)
    q = O.unpack(packed, N, K)
    assert q.min() >= 1 and q.max() <= 15            # amax maps to +-7, never to -8
    s = np.repeat(O.bf16_bits_to_f32(scales).astype(np.float64), g, axis=1)
    wq = (q.astype(np.float64) - 8) * s
    assert (np.abs(w - wq) <= s / 2 * (1 + 1e-6)).all()
    # the largest |w| of every group maps to code 1 or 15
    for n in range(N):
        for j in range(K // g):
            grp = w[n, j * g:(j + 1) * g]
            i = int(np.argmax(np.abs(grp)))
            assert q[n, j * g + i] in (1, 15)


def test_error_metrics():
    ref = np.array([3.0, -4.0])
    m = O.error_metrics(ref + np.array([0.1, 0.0]), ref)
    assert abs(m["rms_ref"] - math.sqrt(12.5)) < 1e-12
    assert abs(m["max_abs_err"] - 0.1) < 1e-12
    assert abs(m["rel_fro"] - 0.1 / 5.0) < 1e-12


# ---- fused epilogue (operator fusion, Sec. 5; activations are the library's
# reading: SwiGLU over interleaved (gate, up) rows, exact GELU) -------------

def test_epilogue_silu_closed_form():
    # with up = 1, SwiGLU output j is silu(gate); sigma(ln 3) = 3/4, sigma(-ln 3) = 1/4
    ln3 = math.log(3.0)
    y = np.array([[0.0, 1.0, ln3, 1.0, -ln3, 1.0]])
    h = O.epilogue_rows(y, O.ACT_SWIGLU)
    assert h.shape == (1, 3)
    assert h[0, 0] == 0.0
    assert abs(h[0, 1] - 0.75 * ln3) < 1e-15
    assert abs(h[0, 2] + 0.25 * ln3) < 1e-15


def test_epilogue_swiglu_hand_example_and_gate_up_order():
    # gate = z[2j], up = z[2j+1]: silu(ln 3) * 2 and silu(-ln 3) * 4
    ln3 = math.log(3.0)
    h = O.epilogue_rows(np.array([[ln3, 2.0, -ln3, 4.0]]), O.ACT_SWIGLU)
    assert abs(h[0, 0] - 1.5 * ln3) < 1e-14
    assert abs(h[0, 1] + 1.0 * ln3) < 1e-14


def test_epilogue_gelu_normal_cdf_values():
    # GELU(t) = t * Phi(t); Phi(1) = 0.841344746068542948..., Phi(-1) = 1 - Phi(1)
    phi1 = 0.8413447460685429
    h = O.epilogue_rows(np.array([[0.0, 1.0, -1.0, 10.0, -10.0]]), O.ACT_GELU)[0]
    assert h[0] == 0.0
    assert abs(h[1] - phi1) < 1e-15
    assert abs(h[2] + (1.0 - phi1)) < 1e-15
    assert abs(h[3] - 10.0) < 1e-12
    assert abs(h[4]) < 1e-20


def test_epilogue_bias_residual_by_hand():
    # bf16 bits: 0.25 = 0x3E80, 0.5 = 0x3F00, 1.0 = 0x3F80, -1.0 = 0xBF80, 2.0 = 0x4000
    y = np.array([[1.5, -2.0]])
    bias = np.array([0x3E80, 0x3F00], dtype=np.uint16)
    residual = np.array([[0x4000, 0x4000], [0x4000, 0x4000], [0x3F80, 0xBF80]], dtype=np.uint16)
    h = O.epilogue_rows(y, O.ACT_NONE, bias=bias, residual=residual, rows=[2])
    assert h.tolist() == [[2.75, -2.5]]            # 1.5 + 0.25 + 1, -2 + 0.5 - 1
    assert O.epilogue_rows(y, O.ACT_NONE).tolist() == y.tolist()


def test_epilogue_bias_enters_before_the_activation():
    # gate 0 + bias 1 -> silu(1) = e / (1 + e); up 3 + bias 0 -> 3
    bias = np.array([0x3F80, 0x0000], dtype=np.uint16)
    h = O.epilogue_rows(np.array([[0.0, 3.0]]), O.ACT_SWIGLU, bias=bias)
    assert abs(h[0, 0] - 3.0 * math.e / (1.0 + math.e)) < 1e-15
    hg = O.epilogue_rows(np.array([[0.0]]), O.ACT_GELU, bias=np.array([0x3F80], dtype=np.uint16))
    assert abs(hg[0, 0] - 0.8413447460685429) < 1e-15


# ---- scoring readout: gather and top-k (Sec. 3.3: affinity prediction, then
# result sorting; the best binders have the smallest free energy) -----------

def test_gather_rows_by_hand():
    src = np.arange(12, dtype=np.uint16).reshape(4, 3)
    dst, ok = O.gather_rows(src, [3, 0, 3])
    assert ok and dst.tolist() == [[9, 10, 11], [0, 1, 2], [9, 10, 11]]
    dst, ok = O.gather_rows(src, [1, 4, -1])
    assert not ok and dst.tolist() == [[3, 4, 5], [0, 0, 0], [0, 0, 0]]


def test_topk_hand_example_ties_zeros_nan():
    s = np.array([3.0, -1.0, np.nan, -1.0, 0.0, -0.0, 2.5], dtype=np.float32)
    idx, val = O.topk_smallest(s, 7)
    assert idx.tolist() == [1, 3, 5, 4, 6, 0, 2]       # -1 (idx 1, 3), -0, +0, 2.5, 3, NaN
    assert np.signbit(val[2]) and not np.signbit(val[3])
    idx, _ = O.topk_smallest(s, 2)
    assert idx.tolist() == [1, 3]
    idx, _ = O.topk_smallest(np.array([np.nan, np.nan, 5.0], dtype=np.float32), 3)
    assert idx.tolist() == [2, 0, 1]                    # NaNs last, by index


def test_topk_matches_a_textbook_sort():
    # totalOrder on non-NaN floats with ties by index = a stable sort of the
    # (value, -0 before +0) keys; check against Python's sorted on random data
    rng = np.random.default_rng(11)
    s = rng.normal(size=500).astype(np.float32)
    s[rng.integers(0, 500, 40)] = 0.25                  # many ties
    s[rng.integers(0, 500, 5)] = -0.0
    s[rng.integers(0, 500, 5)] = 0.0
    order = sorted(range(500), key=lambda i: (float(s[i]), 0 if np.signbit(s[i]) else 1, i))
    for k in (1, 17, 500):
        idx, val = O.topk_smallest(s, k)
        assert idx.tolist() == order[:k]
        assert val.tobytes() == s[order[:k]].tobytes()


# ---- attention prefill over packed sequences (causal per sequence, sliding
# window; Sec. 2.1's 32K window) ---------------------------------------------

def _qkv(M, H, d, seed, q_zero=False):
    rng = np.random.default_rng(seed)
    a = rng.normal(size=(M, 3 * H * d)).astype(np.float32)
    if q_zero:
        a[:, :H * d] = 0.0
    return O.bf16_rne_array(a)


def test_attention_single_key_and_window_one_return_v():
    H, d = 2, 8
    qkv = _qkv(10, H, d, 1)
    v = O.bf16_bits_to_f32(qkv[:, 2 * H * d:]).astype(np.float64)
    out = O.attention_rows(qkv, H, d, [0, 4, 10], window=1 << 15)
    assert np.array_equal(out[0], v[0]) and np.array_equal(out[4], v[4])   # first of each sequence
    out1 = O.attention_rows(qkv, H, d, [0, 4, 10], window=1)               # only itself
    assert np.array_equal(out1, v)


def test_attention_equal_scores_give_the_mean():
    H, d = 1, 16
    qkv = _qkv(9, H, d, 2, q_zero=True)          # q = 0: every score is 0
    v = O.bf16_bits_to_f32(qkv[:, 2 * d:]).astype(np.float64)
    out = O.attention_rows(qkv, H, d, [0, 9], window=4)
    for i in range(9):
        lo = max(0, i - 3)
        assert np.allclose(out[i], v[lo:i + 1].mean(axis=0), rtol=0, atol=1e-14)


def test_attention_two_keys_closed_form():
    # d = 4 (scale 1/2): q1 = e0, k0 = 0, k1 = 2 e0 -> scores 0 and 1, weights 1:e
    H, d = 1, 4
    qkv = np.zeros((2, 12), dtype=np.uint16)
    qkv[1, 0] = 0x3F80                           # q1[0] = 1
    qkv[1, 4] = 0x4000                           # k1[0] = 2
    qkv[0, 8:12] = [0x3F80, 0x4000, 0xBF80, 0]   # v0 = (1, 2, -1, 0)
    qkv[1, 8:12] = [0x4040, 0, 0x3F00, 0x4080]   # v1 = (3, 0, 0.5, 4)
    out = O.attention_rows(qkv, H, d, [0, 2], window=8)
    e = math.e
    want = (np.array([1, 2, -1, 0]) + e * np.array([3, 0, 0.5, 4])) / (1 + e)
    assert np.allclose(out[1], want, rtol=0, atol=1e-15)


def test_attention_is_causal_and_sequences_are_independent():
    H, d = 2, 8
    qkv = _qkv(12, H, d, 3)
    st = [0, 5, 12]
    base = O.attention_rows(qkv, H, d, st, window=64)
    later = qkv.copy()
    later[8:, H * d:] = O.bf16_rne_array(np.full((4, 2 * H * d), 7.0, dtype=np.float32))
    moved = O.attention_rows(later, H, d, st, window=64)
    assert np.array_equal(moved[:8], base[:8])     # keys/values after a query do not matter
    other = qkv.copy()
    other[:5] = O.bf16_rne_array(np.full((5, 3 * H * d), -3.0, dtype=np.float32))
    iso = O.attention_rows(other, H, d, st, window=64)
    assert np.array_equal(iso[5:], base[5:])       # another sequence does not matter


def test_attention_heads_use_their_own_q_k_v_columns():
    """Two heads of d = 4 (scale 1/2) whose scores differ by head: query 1 of
    head 0 favours key 0 (scores 1, 0), query 1 of head 1 favours key 1
    (scores 0, 2); every (token, head) has its own value vector.  Reading q,
    k or v from another head's columns changes the weights or the values."""
    H, d = 2, 4
    one, two, four = 0x3F80, 0x4000, 0x4080
    qkv = np.zeros((2, 3 * H * d), dtype=np.uint16)
    q = lambda t, h, c, b: qkv.__setitem__((t, h * d + c), b)
    k = lambda t, h, c, b: qkv.__setitem__((t, H * d + h * d + c), b)
    v = lambda t, h, c, b: qkv.__setitem__((t, 2 * H * d + h * d + c), b)
    q(1, 0, 0, two)           # head 0: q1 = 2 e0
    q(1, 1, 1, four)          # head 1: q1 = 4 e1
    k(0, 0, 0, one)           # head 0: k0 = e0, k1 = 0    -> scores (1, 0)
    k(1, 1, 1, one)           # head 1: k0 = 0,  k1 = e1   -> scores (0, 2)
    v(0, 0, 0, one)           # v of (token, head): four different unit vectors
    v(1, 0, 1, one)
    v(0, 1, 2, one)
    v(1, 1, 3, one)
    out = O.attention_rows(qkv, H, d, [0, 2], window=8)
    e = math.e
    want1 = np.array([e / (1 + e), 1 / (1 + e), 0, 0,
                      0, 0, 1 / (1 + e * e), e * e / (1 + e * e)])
    want0 = np.array([1, 0, 0, 0, 0, 0, 1, 0])   # query 0 sees only key 0
    assert np.allclose(out[1], want1, rtol=0, atol=1e-15)
    assert np.array_equal(out[0], want0)
