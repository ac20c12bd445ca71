"""The pins must catch plausible mistakes in the oracle.

Each case compiles a copy of oracle/w4a16_oracle.c with one planted mistake
(swapped nibbles, dropped zero point, wrong group index, round-half-away,
truncating bf16 rounding, fp32 accumulation, wrong activation row, and in
the fused epilogue swapped gate/up, a wrong SiLU sign, the tanh GELU
approximation, a wrong residual row, bias after the activation; in the
readout top-k ties by the last index, unordered zeros, NaN first, and a gather
that does not zero the rows of bad indices; in attention a dropped 1/sqrt(d),
a window one token too wide, values read from the keys, keys of other
sequences, and q, k, v or the output of head 0 used for every head), points
the oracle module at it and runs the pins: at least one must fail.  The
mistakes live only in temporary copies on the CPU."""
import ctypes
import os
import subprocess
import tempfile

import pytest

from oracle import oracle as O
from tests import test_oracle_pins as P

SRC = os.path.join(os.path.dirname(O.__file__), "w4a16_oracle.c")

MUTANTS = {
    "swapped_nibbles": [("(k % 2 == 0) ? (b & 0x0F) : (b >> 4)", "(k % 2 == 0) ? (b >> 4) : (b & 0x0F)")],
    "no_zero_point": [("(float)(q - 8) * s", "(float)(q) * s")],
    "group_index_mod": [("scales[n * KG + k / g]", "scales[n * KG + (k % KG)]")],
    "round_half_away": [("nearbyintf(grp[t] / s)", "roundf(grp[t] / s)")],
    "bf16_truncates": [("u += 0x7FFFu + kept_lsb;", "u += 0u * kept_lsb;")],
    "fp32_accumulate": [("double acc = 0.0;", "float acc = 0.0f;")],
    "wrong_x_row": [("const uint16_t* xrow = x + rows[r] * K;", "const uint16_t* xrow = x;")],
    "swiglu_gate_up_swapped": [("h = silu_d(gate) * up;", "h = silu_d(up) * gate;")],
    "silu_wrong_sign": [("return t / (1.0 + exp(-t));", "return t / (1.0 + exp(t));")],
    "gelu_tanh_approximation": [("return 0.5 * t * (1.0 + erf(t / sqrt(2.0)));",
                                 "return 0.5 * t * (1.0 + tanh(0.7978845608028654 * (t + 0.044715 * t * t * t)));")],
    "residual_wrong_row": [("residual[rows[r] * n_out + j]", "residual[r * n_out + j]")],
    "bias_after_activation": [("h = act == 2 ? gelu_d(z) : z;",
                               "h = act == 2 ? gelu_d(yr[j]) + (z - yr[j]) : z;")],
    "topk_ties_by_last_index": [("return ia < ib ? -1 : (ia > ib ? 1 : 0);",
                                 "return ia > ib ? -1 : (ia < ib ? 1 : 0);")],
    "topk_zeros_unordered": [("if (sa != sb) return sa ? -1 : 1;", "(void)sa; (void)sb;")],
    "topk_nan_first": [("if (na != nb) return na ? 1 : -1;", "if (na != nb) return na ? -1 : 1;")],
    "attention_no_scale": [("scratch[j - lo] = dot * scale;", "scratch[j - lo] = dot;")],
    "attention_window_off_by_one": [("i - window + 1 > lo0 ? i - window + 1 : lo0",
                                     "i - window > lo0 ? i - window : lo0")],
    "attention_v_from_k": [("qkv[j * ld + 2 * H * d + h * d + t]", "qkv[j * ld + H * d + h * d + t]")],
    "attention_ignores_sequences": [("const int64_t lo0 = seq_start[s];", "const int64_t lo0 = 0;")],
    "attention_k_of_head_0": [("const uint16_t* k = qkv + j * ld + H * d + h * d;",
                               "const uint16_t* k = qkv + j * ld + H * d;")],
    "attention_q_of_head_0": [("const uint16_t* q = qkv + i * ld + h * d;",
                               "const uint16_t* q = qkv + i * ld;")],
    "attention_v_of_head_0": [("qkv[j * ld + 2 * H * d + h * d + t]", "qkv[j * ld + 2 * H * d + t]")],
    "attention_out_of_head_0": [("out[r * H * d + h * d + t] = acc / den;",
                                 "out[r * H * d + t] = acc / den;")],
    "gather_bad_rows_not_zeroed": [("for (int64_t d = 0; d < D; ++d) dst[p * D + d] = 0;",
                                    "for (int64_t d = 0; d < D; ++d) dst[p * D + d] = 1;")],
}

PINS = [
    P.test_bf16_rne_hand_values,
    P.test_unpack_every_byte,
    P.test_dequant_table_all_codes_against_exact_product,
    P.test_dequant_rounding_cases_by_hand,
    P.test_dequant_group_index,
    P.test_linear_hand_computed_2x3x256,
    P.test_linear_power_of_two_scales_equals_textbook_matmul,
    P.test_linear_invariants,
    P.test_linear_brute_force_small,
    P.test_quantize_hand_example,
    P.test_quantize_rounds_half_to_even_and_zero_group,
    P.test_quantize_error_bound_and_code_range,
    P.test_epilogue_silu_closed_form,
    P.test_epilogue_swiglu_hand_example_and_gate_up_order,
    P.test_epilogue_gelu_normal_cdf_values,
    P.test_epilogue_bias_residual_by_hand,
    P.test_epilogue_bias_enters_before_the_activation,
    P.test_gather_rows_by_hand,
    P.test_topk_hand_example_ties_zeros_nan,
    P.test_topk_matches_a_textbook_sort,
    P.test_attention_single_key_and_window_one_return_v,
    P.test_attention_equal_scores_give_the_mean,
    P.test_attention_two_keys_closed_form,
    P.test_attention_is_causal_and_sequences_are_independent,
    P.test_attention_heads_use_their_own_q_k_v_columns,
]


def _build_mutant(name, edits, outdir):
    src = open(SRC).read()
    for old, new in edits:
        assert old in src, (name, old)
        src = src.replace(old, new)
    c = os.path.join(outdir, f"{name}.c")
    so = os.path.join(outdir, f"{name}.so")
    open(c, "w").write(src)
    subprocess.run(["gcc", "-O2", "-fPIC", "-shared", "-fopenmp", "-fno-fast-math",
                    "-ffp-contract=off", "-o", so, c, "-lm"], check=True)
    return so


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_planted_mistake(name, monkeypatch):
    good = O.lib()
    with tempfile.TemporaryDirectory() as d:
        so = _build_mutant(name, MUTANTS[name], d)
        mut = ctypes.CDLL(so)
        for fn in ("oracle_bf16_rne", "oracle_bf16_to_f32", "oracle_unpack", "oracle_pack",
                   "oracle_quantize", "oracle_dequant", "oracle_linear_rows",
                   "oracle_linear_points", "oracle_epilogue_rows", "oracle_gather_rows",
                   "oracle_topk_smallest", "oracle_attention_rows", "oracle_max_threads"):
            getattr(mut, fn).argtypes = getattr(good, fn).argtypes
            getattr(mut, fn).restype = getattr(good, fn).restype
        monkeypatch.setattr(O, "_lib", mut)
        failed = []
        for pin in PINS:
            try:
                pin()
            except AssertionError:
                failed.append(pin.__name__)
        assert failed, f"no pin caught the planted mistake {name}"
