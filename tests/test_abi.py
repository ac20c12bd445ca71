"""Host-side checks of the C ABI (no GPU needed): the library loads, exports
every function include/w4a16.h declares, and rejects bad arguments before
touching the device."""
import ctypes

import pytest

from paper_2608_30877_gb300 import w4a16 as W


@pytest.fixture(scope="module")
def L():
    from paper_2608_30877_gb300 import build as B
    B.build()
    return W.lib()


def test_header_declares_the_boundary():
    names = W.header_functions()
    for f in ("w4a16_linear", "w4a16_linear_stack", "w4a16_dequant", "w4a16_quantize",
              "w4a16_get_device_error", "w4a16_status_string", "w4a16_version"):
        assert f in names


def test_every_declared_symbol_is_exported(L):
    for name in W.header_functions():
        assert hasattr(L, name), name


def test_status_strings(L):
    assert W.status_string(0) == "ok"
    assert "aligned" in W.status_string(W.ERR_ALIGNMENT)
    assert W.status_string(99) == "unknown status"
    assert W.version() >= 100


A = 1 << 20  # fake, 16-byte aligned, non-overlapping "device" addresses (never dereferenced)


@pytest.mark.parametrize("args,want", [
    ((0, A, 2 * A, 3 * A, 4, 8, 256, 128), W.ERR_INVALID_ARG),        # null x
    ((A, 2 * A, 3 * A, 4 * A, 0, 8, 256, 128), W.ERR_INVALID_ARG),     # M = 0
    ((A, 2 * A, 3 * A, 4 * A, 4, -1, 256, 128), W.ERR_INVALID_ARG),    # N < 0
    ((A, 2 * A, 3 * A, 4 * A, 4, 8, 200, 128), W.ERR_INVALID_ARG),     # K % g
    ((A, 2 * A, 3 * A, 4 * A, 4, 8, 256, 32), W.ERR_UNSUPPORTED),      # g % 64
    ((A + 8, 2 * A, 3 * A, 4 * A, 4, 8, 256, 128), W.ERR_ALIGNMENT),   # misaligned x
    ((A, 2 * A, 3 * A, 4 * A + 2, 4, 8, 256, 128), W.ERR_ALIGNMENT),   # misaligned out
    ((A, 2 * A, 3 * A, A + 64, 4, 8, 256, 128), W.ERR_INVALID_ARG),    # out overlaps x
    ((A, 2 * A, 3 * A, 4 * A, 1 << 31, 8, 256, 128), W.ERR_UNSUPPORTED),
])
def test_linear_rejects_before_launch(L, args, want):
    assert L.w4a16_linear(*args, None) == want


def test_stack_validates_every_layer_first(L):
    good = W.Layer(A, 2 * A, 3 * A, 4 * A, 8, 256)
    bad = W.Layer(A, 2 * A, 3 * A, 4 * A, 8, 200)
    arr = (W.Layer * 2)(good, bad)
    assert L.w4a16_linear_stack(arr, 2, 4, 128, None) == W.ERR_INVALID_ARG
    assert L.w4a16_linear_stack(arr, 0, 4, 128, None) == W.ERR_INVALID_ARG
    assert L.w4a16_linear_stack(None, 1, 4, 128, None) == W.ERR_INVALID_ARG


def test_dequant_and_quantize_reject_bad_args(L):
    assert L.w4a16_dequant(A, 2 * A, 0, 8, 256, 128, None) == W.ERR_INVALID_ARG
    assert L.w4a16_dequant(A, 2 * A, 3 * A + 4, 8, 256, 128, None) == W.ERR_ALIGNMENT
    assert L.w4a16_quantize(0, 2 * A, 3 * A, 8, 256, 128, None) == W.ERR_INVALID_ARG
    assert L.w4a16_quantize(A, 2 * A, 3 * A, 8, 256, 48, None) == W.ERR_INVALID_ARG


@pytest.mark.parametrize("bias,res,out,N,act,want", [
    (0, 0, 4 * A, 8, 3, W.ERR_INVALID_ARG),             # unknown activation
    (0, 0, 4 * A, 7, W.ACT_SWIGLU, W.ERR_INVALID_ARG),  # SwiGLU needs even N
    (5 * A + 2, 0, 4 * A, 8, W.ACT_GELU, W.ERR_ALIGNMENT),   # misaligned bias
    (0, 6 * A + 8, 4 * A, 8, W.ACT_NONE, W.ERR_ALIGNMENT),   # misaligned residual
    (4 * A + 16, 0, 4 * A, 8, W.ACT_NONE, W.ERR_INVALID_ARG),  # bias overlaps out
    (0, 4 * A + 16, 4 * A, 8, W.ACT_NONE, W.ERR_INVALID_ARG),  # residual partly overlaps out
    (0, 0, A + 64, 8, W.ACT_SWIGLU, W.ERR_INVALID_ARG),        # out overlaps x
])
def test_fused_rejects_before_launch(L, bias, res, out, N, act, want):
    assert L.w4a16_linear_fused(A, 2 * A, 3 * A, bias or None, res or None, out, 4, N, 256, 128,
                                act, None) == want


def test_readout_rejects_before_launch(L):
    # gather: null, zero sizes, misaligned, dst overlapping src
    assert L.w4a16_gather_rows(0, 4, 8, 2 * A, 2, 3 * A, None) == W.ERR_INVALID_ARG
    assert L.w4a16_gather_rows(A, 0, 8, 2 * A, 2, 3 * A, None) == W.ERR_INVALID_ARG
    assert L.w4a16_gather_rows(A, 4, 8, 2 * A + 4, 2, 3 * A, None) == W.ERR_ALIGNMENT
    assert L.w4a16_gather_rows(A, 4, 8, 2 * A, 2, A + 16, None) == W.ERR_INVALID_ARG
    # top-k: bad score width, k out of range, k above the supported limit, overlap
    assert L.w4a16_topk_smallest(A, 8, 100, 10, 2 * A, 3 * A, None) == W.ERR_INVALID_ARG
    assert L.w4a16_topk_smallest(A, 32, 100, 0, 2 * A, 3 * A, None) == W.ERR_INVALID_ARG
    assert L.w4a16_topk_smallest(A, 32, 100, 101, 2 * A, 3 * A, None) == W.ERR_INVALID_ARG
    assert L.w4a16_topk_smallest(A, 32, 5000, 1025, 2 * A, 3 * A, None) == W.ERR_UNSUPPORTED
    assert L.w4a16_topk_smallest(A, 16, 100, 10, A + 16, 3 * A, None) == W.ERR_INVALID_ARG
    assert L.w4a16_topk_smallest(A, 32, 100, 10, 2 * A, 2 * A + 16, None) == W.ERR_INVALID_ARG


def test_attention_rejects_before_launch(L):
    assert L.w4a16_attention_prefill(0, 2 * A, 1, 64, 2, 128, 100, 3 * A, None) == W.ERR_INVALID_ARG
    assert L.w4a16_attention_prefill(A, 2 * A, 1, 64, 2, 64, 100, 3 * A, None) == W.ERR_UNSUPPORTED
    assert L.w4a16_attention_prefill(A, 2 * A, 1, 64, 2, 128, 0, 3 * A, None) == W.ERR_INVALID_ARG
    assert L.w4a16_attention_prefill(A, 2 * A + 4, 1, 64, 2, 128, 9, 3 * A, None) == W.ERR_ALIGNMENT
    assert L.w4a16_attention_prefill(A, 2 * A, 1, 64, 2, 128, 9, A + 64, None) == W.ERR_INVALID_ARG


def test_stack_graph_rejects_bad_handles(L):
    import ctypes
    h = ctypes.c_void_p()
    good = W.Layer(A, 2 * A, 3 * A, 4 * A, 8, 256)
    arr = (W.Layer * 1)(good)
    assert L.w4a16_stack_graph_create(arr, 1, 4, 128, None) == W.ERR_INVALID_ARG
    assert L.w4a16_stack_graph_create(None, 1, 4, 128, ctypes.byref(h)) == W.ERR_INVALID_ARG
    bad = (W.Layer * 1)(W.Layer(A, 2 * A, 3 * A, 4 * A, 8, 200))
    assert L.w4a16_stack_graph_create(bad, 1, 4, 128, ctypes.byref(h)) == W.ERR_INVALID_ARG
    assert not h.value
    assert L.w4a16_stack_graph_launch(None, None) == W.ERR_INVALID_ARG
    assert L.w4a16_stack_graph_destroy(None) == W.ERR_INVALID_ARG


def test_debug_build_exports_the_same_symbols():
    """The W4A16_DEBUG build (the kernels' index checks) compiles and exports
    every declared function; its status string for the check is defined."""
    import ctypes as C
    from paper_2608_30877_gb300 import build as B
    D = C.CDLL(B.build(debug=True))
    for name in W.header_functions():
        assert hasattr(D, name), name
    D.w4a16_status_string.restype = C.c_char_p
    assert b"debug" in D.w4a16_status_string(W.ERR_INDEX)
