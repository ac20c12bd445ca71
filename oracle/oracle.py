"""Python face of the CPU oracle (oracle/w4a16_oracle.c).

TEST INFRASTRUCTURE ONLY: imported by tests/, by __graft_entry__.smoke() and
by bench.py's cpu_baseline and --impl reference legs.  The product path never
imports it; it shares no code with the CUDA library.

The oracle states the method's definition (Sec. 3.1 / Sec. 4.1 give only
"4-bit pre-quantized"; the format is the library's): int4 codes with zero
point 8, low nibble = even k, one bf16 scale per g consecutive k, dequant
wd = RNE_bf16((q - 8) * s), out = x @ wd^T accumulated in fp64.  Arrays are
numpy; bf16 values travel as their uint16 bit patterns.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "w4a16_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "liboracle.so")

_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain C, OpenMP for the row loop)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        # -O2 without -ffast-math: IEEE fp32 division and nearest-even rounding.
        cmd = ["gcc", "-O2", "-fPIC", "-shared", "-fopenmp", "-fno-fast-math",
               "-ffp-contract=off", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(_LIB)
        i64, p = ctypes.c_int64, ctypes.c_void_p
        L.oracle_bf16_rne.argtypes = [ctypes.c_float]
        L.oracle_bf16_rne.restype = ctypes.c_uint16
        L.oracle_bf16_to_f32.argtypes = [ctypes.c_uint16]
        L.oracle_bf16_to_f32.restype = ctypes.c_float
        L.oracle_unpack.argtypes = [p, i64, i64, p]
        L.oracle_pack.argtypes = [p, i64, i64, p]
        L.oracle_quantize.argtypes = [p, i64, i64, i64, p, p]
        L.oracle_quantize.restype = ctypes.c_int
        L.oracle_dequant.argtypes = [p, p, i64, i64, i64, p]
        L.oracle_linear_rows.argtypes = [p, p, p, i64, i64, i64, i64, p, i64, p, ctypes.c_int]
        L.oracle_linear_points.argtypes = [p, p, p, i64, i64, i64, i64, p, p, i64, p, ctypes.c_int]
        L.oracle_epilogue_rows.argtypes = [p, i64, i64, p, p, p, ctypes.c_int, p]
        L.oracle_gather_rows.argtypes = [p, i64, i64, p, i64, p]
        L.oracle_gather_rows.restype = ctypes.c_int
        L.oracle_topk_smallest.argtypes = [p, i64, i64, p, p, p]
        L.oracle_attention_rows.argtypes = [p, i64, i64, i64, p, i64, i64, p, i64, p, p]
        L.oracle_max_threads.restype = ctypes.c_int
        _lib = L
    return _lib


def _ptr(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


def bf16_rne(f32: float) -> int:
    return int(lib().oracle_bf16_rne(ctypes.c_float(f32)))


def bf16_rne_array(a: np.ndarray) -> np.ndarray:
    """Element-wise oracle rounding of an fp32 array (slow, for pins)."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    L = lib()
    return np.array([L.oracle_bf16_rne(ctypes.c_float(float(v))) for v in a.ravel()],
                    dtype=np.uint16).reshape(a.shape)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to fp32 (a bit shift)."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def unpack(packed: np.ndarray, N: int, K: int) -> np.ndarray:
    packed = np.ascontiguousarray(packed, dtype=np.uint8)
    q = np.empty((N, K), dtype=np.uint8)
    lib().oracle_unpack(_ptr(packed), N, K, _ptr(q))
    return q


def pack(q: np.ndarray) -> np.ndarray:
    q = np.ascontiguousarray(q, dtype=np.uint8)
    N, K = q.shape
    packed = np.empty((N, K // 2), dtype=np.uint8)
    lib().oracle_pack(_ptr(q), N, K, _ptr(packed))
    return packed


def quantize(w: np.ndarray, g: int):
    """fp32 master weights [N, K] -> (packed uint8 [N, K/2], scales bf16-bits [N, K/g])."""
    w = np.ascontiguousarray(w, dtype=np.float32)
    N, K = w.shape
    packed = np.zeros((N, K // 2), dtype=np.uint8)
    scales = np.zeros((N, K // g), dtype=np.uint16)
    rc = lib().oracle_quantize(_ptr(w), N, K, g, _ptr(packed), _ptr(scales))
    if rc != 0:
        raise ValueError(f"oracle_quantize rejected shape N={N} K={K} g={g}")
    return packed, scales


def dequant(packed: np.ndarray, scales: np.ndarray, N: int, K: int, g: int) -> np.ndarray:
    """-> bf16 bit patterns [N, K]."""
    packed = np.ascontiguousarray(packed, dtype=np.uint8)
    scales = np.ascontiguousarray(scales, dtype=np.uint16)
    wd = np.empty((N, K), dtype=np.uint16)
    lib().oracle_dequant(_ptr(packed), _ptr(scales), N, K, g, _ptr(wd))
    return wd


def linear_rows(x_bits: np.ndarray, packed: np.ndarray, scales: np.ndarray,
                N: int, K: int, g: int, rows=None, nthreads: int = 1) -> np.ndarray:
    """fp64 reference rows: out[r, n] = sum_k x[rows[r], k] * wd[n, k]."""
    x_bits = np.ascontiguousarray(x_bits, dtype=np.uint16)
    M = x_bits.shape[0]
    rows = np.arange(M, dtype=np.int64) if rows is None else np.ascontiguousarray(rows, dtype=np.int64)
    packed = np.ascontiguousarray(packed, dtype=np.uint8)
    scales = np.ascontiguousarray(scales, dtype=np.uint16)
    out = np.empty((rows.shape[0], N), dtype=np.float64)
    lib().oracle_linear_rows(_ptr(x_bits), _ptr(packed), _ptr(scales), M, N, K, g,
                             _ptr(rows), rows.shape[0], _ptr(out), int(nthreads))
    return out


def linear_points(x_bits: np.ndarray, packed: np.ndarray, scales: np.ndarray,
                  N: int, K: int, g: int, mi, ni, nthreads: int = 1) -> np.ndarray:
    """fp64 reference values at the points (mi[i], ni[i])."""
    x_bits = np.ascontiguousarray(x_bits, dtype=np.uint16)
    M = x_bits.shape[0]
    mi = np.ascontiguousarray(mi, dtype=np.int64)
    ni = np.ascontiguousarray(ni, dtype=np.int64)
    packed = np.ascontiguousarray(packed, dtype=np.uint8)
    scales = np.ascontiguousarray(scales, dtype=np.uint16)
    out = np.empty(mi.shape[0], dtype=np.float64)
    lib().oracle_linear_points(_ptr(x_bits), _ptr(packed), _ptr(scales), M, N, K, g,
                               _ptr(mi), _ptr(ni), mi.shape[0], _ptr(out), int(nthreads))
    return out


ACT_NONE, ACT_SWIGLU, ACT_GELU = 0, 1, 2


def epilogue_rows(y: np.ndarray, act: int = ACT_NONE, bias=None, residual=None,
                  rows=None) -> np.ndarray:
    """Fused epilogue on fp64 linear outputs y [nrows, N] (rows `rows` of the
    batch): act(y + bias) + residual, fp64 [nrows, N_out]; SwiGLU takes rows
    (2j, 2j+1) of the weights as (gate, up) of output j."""
    y = np.ascontiguousarray(y, dtype=np.float64)
    nrows, N = y.shape
    rows = np.arange(nrows, dtype=np.int64) if rows is None else np.ascontiguousarray(rows, dtype=np.int64)
    n_out = N // 2 if act == ACT_SWIGLU else N
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.uint16)
    res = None if residual is None else np.ascontiguousarray(residual, dtype=np.uint16)
    out = np.empty((nrows, n_out), dtype=np.float64)
    lib().oracle_epilogue_rows(_ptr(y), nrows, N, None if b is None else _ptr(b),
                               None if res is None else _ptr(res), _ptr(rows), int(act), _ptr(out))
    return out


def gather_rows(src_bits: np.ndarray, idx) -> tuple[np.ndarray, bool]:
    """dst[p] = src[idx[p]] (bf16 bits); out-of-range indices give zero rows
    and ok = False."""
    src_bits = np.ascontiguousarray(src_bits, dtype=np.uint16)
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    rows, D = src_bits.shape
    dst = np.empty((idx.shape[0], D), dtype=np.uint16)
    bad = lib().oracle_gather_rows(_ptr(src_bits), rows, D, _ptr(idx), idx.shape[0], _ptr(dst))
    return dst, bad == 0


def topk_smallest(scores: np.ndarray, k: int):
    """(indices int32 [k], scores fp32 [k]) of the k smallest scores, ascending
    by IEEE totalOrder (NaN last), ties by index."""
    scores = np.ascontiguousarray(scores, dtype=np.float32)
    n = scores.shape[0]
    idx = np.empty(k, dtype=np.int32)
    val = np.empty(k, dtype=np.float32)
    taken = np.empty(max(n, 1), dtype=np.uint8)
    lib().oracle_topk_smallest(_ptr(scores), n, k, _ptr(idx), _ptr(val), _ptr(taken))
    return idx, val


def attention_rows(qkv_bits: np.ndarray, H: int, d: int, seq_start, window: int,
                   rows=None) -> np.ndarray:
    """fp64 attention outputs [len(rows), H d] for query tokens `rows` of the
    packed batch: causal within each sequence [seq_start[s], seq_start[s+1])
    and within a window of `window` tokens; qkv bf16 bits [M, 3 H d]."""
    qkv_bits = np.ascontiguousarray(qkv_bits, dtype=np.uint16)
    M = qkv_bits.shape[0]
    st = np.ascontiguousarray(seq_start, dtype=np.int64)
    rows = np.arange(M, dtype=np.int64) if rows is None else np.ascontiguousarray(rows, dtype=np.int64)
    out = np.empty((rows.shape[0], H * d), dtype=np.float64)
    scratch = np.empty(max(1, min(M, window)), dtype=np.float64)
    lib().oracle_attention_rows(_ptr(qkv_bits), M, H, d, _ptr(st), st.shape[0] - 1, window,
                                _ptr(rows), rows.shape[0], _ptr(out), _ptr(scratch))
    return out


def max_threads() -> int:
    return int(lib().oracle_max_threads())


def error_metrics(gpu: np.ndarray, ref: np.ndarray) -> dict:
    """The two tolerance statistics for one output matrix (or a sample of one)."""
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    diff = gpu - ref
    rms = float(np.sqrt(np.mean(ref * ref))) if ref.size else 0.0
    fro_ref = float(np.linalg.norm(ref.ravel()))
    return {
        "max_abs_err": float(np.max(np.abs(diff))) if diff.size else 0.0,
        "rms_ref": rms,
        "max_err_over_rms": (float(np.max(np.abs(diff))) / rms) if rms > 0 else 0.0,
        "rel_fro": (float(np.linalg.norm(diff.ravel())) / fro_ref) if fro_ref > 0 else 0.0,
    }
