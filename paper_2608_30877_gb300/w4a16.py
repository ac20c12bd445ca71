"""Thin Python binding of libw4a16.so (include/w4a16.h).

Argument marshalling only: torch tensors supply device memory and the
current CUDA stream; every step of the computation runs in the library's
kernels.  There is no fallback -- if the library is not built or the GPU is
missing, the call raises.
"""
from __future__ import annotations

import ctypes
import os
import re

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
# W4A16_DEBUG=1 loads the build with the kernels' index checks
LIB_PATH = os.path.join(_PKG, "libw4a16_debug.so" if os.environ.get("W4A16_DEBUG") == "1"
                        else "libw4a16.so")
HEADER = os.path.join(os.path.dirname(_PKG), "include", "w4a16.h")

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_ALIGNMENT, ERR_CUDA, ERR_TIMEOUT, ERR_INDEX = range(7)
ACT_NONE, ACT_SWIGLU, ACT_GELU = range(3)

_lib = None


class W4A16Error(RuntimeError):
    def __init__(self, fn: str, status: int):
        self.status = status
        super().__init__(f"{fn} failed: {status_string(status)} (status {status})")


class Layer(ctypes.Structure):
    _fields_ = [("x", ctypes.c_void_p), ("w_packed", ctypes.c_void_p),
                ("scales", ctypes.c_void_p), ("out", ctypes.c_void_p),
                ("N", ctypes.c_int64), ("K", ctypes.c_int64)]


def header_functions() -> list[str]:
    """Names of the functions include/w4a16.h declares."""
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w[\w\s\*]*?\b(w4a16_\w+)\s*\(", text, re.M)))


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built; run `python -c 'import __graft_entry__ as g; "
                               "g.build()'` first (needs nvcc)")
        L = ctypes.CDLL(LIB_PATH)
        i64, p = ctypes.c_int64, ctypes.c_void_p
        L.w4a16_linear.argtypes = [p, p, p, p, i64, i64, i64, i64, p]
        L.w4a16_linear_fused.argtypes = [p, p, p, p, p, p, i64, i64, i64, i64, ctypes.c_int, p]
        L.w4a16_linear_stack.argtypes = [ctypes.POINTER(Layer), i64, i64, i64, p]
        L.w4a16_dequant.argtypes = [p, p, p, i64, i64, i64, p]
        L.w4a16_stack_graph_create.argtypes = [ctypes.POINTER(Layer), i64, i64, i64,
                                               ctypes.POINTER(ctypes.c_void_p)]
        L.w4a16_stack_graph_launch.argtypes = [p, p]
        L.w4a16_stack_graph_destroy.argtypes = [p]
        L.w4a16_gather_rows.argtypes = [p, i64, i64, p, i64, p, p]
        L.w4a16_attention_prefill.argtypes = [p, p, i64, i64, i64, i64, i64, p, p]
        L.w4a16_topk_smallest.argtypes = [p, ctypes.c_int, i64, i64, p, p, p]
        L.w4a16_quantize.argtypes = [p, p, p, i64, i64, i64, p]
        L.w4a16_get_device_error.argtypes = [p]
        L.w4a16_selftest_wait_timeout.argtypes = [i64, p]
        L.w4a16_selftest_set_wait_limit.argtypes = [i64]
        L.w4a16_status_string.argtypes = [ctypes.c_int]
        L.w4a16_status_string.restype = ctypes.c_char_p
        L.w4a16_version.restype = ctypes.c_int
        for f in ("w4a16_linear", "w4a16_linear_fused", "w4a16_linear_stack",
                  "w4a16_gather_rows", "w4a16_topk_smallest", "w4a16_attention_prefill",
                  "w4a16_stack_graph_create", "w4a16_stack_graph_launch",
                  "w4a16_stack_graph_destroy", "w4a16_dequant", "w4a16_quantize",
                  "w4a16_get_device_error", "w4a16_selftest_wait_timeout",
                  "w4a16_selftest_set_wait_limit"):
            getattr(L, f).restype = ctypes.c_int
        _lib = L
    return _lib


def status_string(status: int) -> str:
    return lib().w4a16_status_string(int(status)).decode()


def version() -> int:
    return int(lib().w4a16_version())


def _stream(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream) if hasattr(stream, "cuda_stream") else int(stream)


def _check(fn: str, rc: int):
    if rc != OK:
        raise W4A16Error(fn, rc)


def _need_cuda(*ts):
    for t in ts:
        if not (isinstance(t, torch.Tensor) and t.is_cuda and t.is_contiguous()):
            raise ValueError("expected contiguous CUDA tensors")


def linear(x: torch.Tensor, w_packed: torch.Tensor, scales: torch.Tensor, g: int = 128,
           out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """out[M, N] = x[M, K] @ dequant(w_packed[N, K/2], scales[N, K/g])^T, bf16."""
    M, K = x.shape
    N = w_packed.shape[0]
    if out is None:
        out = torch.empty((M, N), dtype=torch.bfloat16, device=x.device)
    _need_cuda(x, w_packed, scales, out)
    assert x.dtype == torch.bfloat16 and w_packed.dtype == torch.uint8
    assert scales.dtype == torch.bfloat16 and out.dtype == torch.bfloat16
    assert w_packed.shape[1] * 2 == K and scales.shape == (N, K // g) and out.shape == (M, N)
    _check("w4a16_linear", lib().w4a16_linear(x.data_ptr(), w_packed.data_ptr(), scales.data_ptr(),
                                              out.data_ptr(), M, N, K, g, _stream(stream)))
    return out


def linear_fused(x: torch.Tensor, w_packed: torch.Tensor, scales: torch.Tensor, g: int = 128,
                 act: int = ACT_NONE, bias: torch.Tensor | None = None,
                 residual: torch.Tensor | None = None, out: torch.Tensor | None = None,
                 stream=None) -> torch.Tensor:
    """out = act(x @ dequant(w)^T + bias) + residual (include/w4a16.h); for
    ACT_SWIGLU rows (2j, 2j+1) of w are (gate, up) and out has N/2 columns."""
    M, K = x.shape
    N = w_packed.shape[0]
    n_out = N // 2 if act == ACT_SWIGLU else N
    if out is None:
        out = torch.empty((M, n_out), dtype=torch.bfloat16, device=x.device)
    _need_cuda(x, w_packed, scales, out, *(t for t in (bias, residual) if t is not None))
    _check("w4a16_linear_fused", lib().w4a16_linear_fused(
        x.data_ptr(), w_packed.data_ptr(), scales.data_ptr(),
        None if bias is None else bias.data_ptr(),
        None if residual is None else residual.data_ptr(),
        out.data_ptr(), M, N, K, g, int(act), _stream(stream)))
    return out


def linear_raw(x_ptr: int, w_ptr: int, s_ptr: int, out_ptr: int, M: int, N: int, K: int, g: int,
               stream: int) -> int:
    """Direct call with raw pointers; returns the status code."""
    return lib().w4a16_linear(x_ptr, w_ptr, s_ptr, out_ptr, M, N, K, g, stream)


def linear_stack(layers, M: int, g: int = 128, stream=None) -> None:
    """layers: sequence of (x, w_packed, scales, out) tensors, run in order."""
    arr = (Layer * len(layers))()
    for i, (x, w, s, o) in enumerate(layers):
        _need_cuda(x, w, s, o)
        arr[i] = Layer(x.data_ptr(), w.data_ptr(), s.data_ptr(), o.data_ptr(), w.shape[0],
                       w.shape[1] * 2)
    _check("w4a16_linear_stack", lib().w4a16_linear_stack(arr, len(layers), M, g, _stream(stream)))


def make_layer_array(layers) -> ctypes.Array:
    """Pre-built Layer array for repeated w4a16_linear_stack calls."""
    arr = (Layer * len(layers))()
    for i, (x, w, s, o) in enumerate(layers):
        arr[i] = Layer(x.data_ptr(), w.data_ptr(), s.data_ptr(), o.data_ptr(), w.shape[0],
                       w.shape[1] * 2)
    return arr


class StackGraph:
    """A layer stack captured as a CUDA graph (include/w4a16.h); replay with
    launch(), release with close() (or as a context manager)."""

    def __init__(self, layers, M: int, g: int = 128):
        self._arr = make_layer_array(layers)
        self._h = ctypes.c_void_p()
        _check("w4a16_stack_graph_create", lib().w4a16_stack_graph_create(
            self._arr, len(self._arr), M, g, ctypes.byref(self._h)))

    def launch(self, stream=None):
        _check("w4a16_stack_graph_launch", lib().w4a16_stack_graph_launch(self._h, _stream(stream)))

    def close(self):
        if self._h:
            _check("w4a16_stack_graph_destroy", lib().w4a16_stack_graph_destroy(self._h))
            self._h = ctypes.c_void_p()

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()


def linear_stack_array(arr: ctypes.Array, M: int, g: int = 128, stream=None) -> None:
    _check("w4a16_linear_stack", lib().w4a16_linear_stack(arr, len(arr), M, g, _stream(stream)))


def attention_prefill(qkv: torch.Tensor, seq_start: torch.Tensor, H: int, window: int = 32768,
                      out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Causal sliding-window attention over packed sequences (include/w4a16.h):
    qkv bf16 [M, 3 H 128], seq_start int32 [nseq + 1] -> out bf16 [M, H 128]."""
    M = qkv.shape[0]
    d = qkv.shape[1] // (3 * H)
    if out is None:
        out = torch.zeros((M, H * d), dtype=torch.bfloat16, device=qkv.device)
    _need_cuda(qkv, seq_start, out)
    assert qkv.dtype == torch.bfloat16 and seq_start.dtype == torch.int32
    _check("w4a16_attention_prefill", lib().w4a16_attention_prefill(
        qkv.data_ptr(), seq_start.data_ptr(), seq_start.shape[0] - 1, M, H, d, int(window),
        out.data_ptr(), _stream(stream)))
    return out


def gather_rows(src: torch.Tensor, index: torch.Tensor, out=None, stream=None) -> torch.Tensor:
    """dst[p] = src[index[p]] for bf16 rows; index int32 (include/w4a16.h)."""
    rows, D = src.shape
    P = index.shape[0]
    if out is None:
        out = torch.empty((P, D), dtype=torch.bfloat16, device=src.device)
    _need_cuda(src, index, out)
    assert src.dtype == torch.bfloat16 and index.dtype == torch.int32
    _check("w4a16_gather_rows", lib().w4a16_gather_rows(src.data_ptr(), rows, D, index.data_ptr(),
                                                        P, out.data_ptr(), _stream(stream)))
    return out


def topk_smallest(scores: torch.Tensor, k: int, stream=None):
    """(int32 indices [k], fp32 scores [k]) of the k smallest scores (fp32 or
    bf16), ascending by totalOrder, NaN last, ties by index."""
    n = scores.shape[0]
    _need_cuda(scores)
    bits = {torch.float32: 32, torch.bfloat16: 16}[scores.dtype]
    idx = torch.empty(k, dtype=torch.int32, device=scores.device)
    val = torch.empty(k, dtype=torch.float32, device=scores.device)
    _check("w4a16_topk_smallest", lib().w4a16_topk_smallest(
        scores.data_ptr(), bits, n, k, idx.data_ptr(), val.data_ptr(), _stream(stream)))
    return idx, val


def dequant(w_packed: torch.Tensor, scales: torch.Tensor, g: int = 128, out=None,
            stream=None) -> torch.Tensor:
    N, K2 = w_packed.shape
    K = 2 * K2
    if out is None:
        out = torch.empty((N, K), dtype=torch.bfloat16, device=w_packed.device)
    _need_cuda(w_packed, scales, out)
    _check("w4a16_dequant", lib().w4a16_dequant(w_packed.data_ptr(), scales.data_ptr(),
                                                out.data_ptr(), N, K, g, _stream(stream)))
    return out


def quantize(w: torch.Tensor, g: int = 128, stream=None):
    """fp32 [N, K] (CUDA) -> (packed uint8 [N, K/2], scales bf16 [N, K/g])."""
    N, K = w.shape
    _need_cuda(w)
    assert w.dtype == torch.float32
    packed = torch.empty((N, K // 2), dtype=torch.uint8, device=w.device)
    scales = torch.empty((N, K // g), dtype=torch.bfloat16, device=w.device)
    _check("w4a16_quantize", lib().w4a16_quantize(w.data_ptr(), packed.data_ptr(),
                                                  scales.data_ptr(), N, K, g, _stream(stream)))
    return packed, scales


def selftest_wait_timeout(limit_ns: int, stream=None) -> None:
    """Launch the bounded-wait self test (see include/w4a16.h)."""
    _check("w4a16_selftest_wait_timeout",
           lib().w4a16_selftest_wait_timeout(int(limit_ns), _stream(stream)))


def set_wait_limit(limit_ns: int) -> None:
    """Wait limit of the kernels launched from now on (0: the default);
    test hook, see include/w4a16.h."""
    _check("w4a16_selftest_set_wait_limit", lib().w4a16_selftest_set_wait_limit(int(limit_ns)))


def get_device_error(stream=None) -> int:
    return int(lib().w4a16_get_device_error(_stream(stream)))
