"""CPU oracle for the quantized linear layer -- TEST INFRASTRUCTURE ONLY.

A plain C restatement (``qlin_oracle.c``) of the FP8 / NVFP4 quantizers and of
the linear layer's exact fp64 result, written from the format definitions the
paper's quantization recipe relies on (Sec. 4, "Quantization").  This module
compiles it with gcc and exposes numpy-facing wrappers.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  It shares no code with the CUDA library
in ``paper_2609_21849_gb300`` and never imports it.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "qlin_oracle.c")
_LIB_DIR = os.path.join(_HERE, "_lib")
_LIB = os.path.join(_LIB_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

_i64 = ctypes.c_int64
_p = ctypes.c_void_p


def build(force: bool = False) -> str:
    """Compile the oracle into ``oracle/_lib/liboracle.so`` (gcc, -O2,
    -ffp-contract=off, OpenMP when available)."""
    os.makedirs(_LIB_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    base = ["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-std=c11",
            "-shared", "-fPIC", _SRC, "-o", _LIB + ".tmp", "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True,
                       capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(_LIB + ".tmp", _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        sig = {
            "oracle_num_threads": (ctypes.c_int, []),
            "oracle_set_num_threads": (None, [ctypes.c_int]),
            "oracle_bf16_to_f32": (ctypes.c_float, [ctypes.c_uint16]),
            "oracle_e2m1_decode": (ctypes.c_double, [ctypes.c_int]),
            "oracle_e2m1_encode": (ctypes.c_int, [ctypes.c_double]),
            "oracle_e4m3_decode": (ctypes.c_double, [ctypes.c_int]),
            "oracle_e4m3_encode": (ctypes.c_int, [ctypes.c_double]),
            "oracle_amax_bf16": (ctypes.c_float, [_p, _i64]),
            "oracle_nvfp4_tensor_scale": (ctypes.c_float, [ctypes.c_float]),
            "oracle_fp8_tensor_scale": (ctypes.c_float, [ctypes.c_float]),
            "oracle_encode_scale": (ctypes.c_float, [ctypes.c_float]),
            "oracle_quant_nvfp4": (None, [_p, _i64, _i64, ctypes.c_float, _p, _p]),
            "oracle_quant_fp8": (None, [_p, _i64, _i64, ctypes.c_float, _p]),
            "oracle_quant_fp8_rows": (None, [_p, _i64, _i64, _p, _p]),
            "oracle_swizzled_scale_bytes": (_i64, [_i64, _i64]),
            "oracle_swizzle_offset": (_i64, [_i64, _i64, _i64]),
            "oracle_swizzle_scales": (None, [_p, _i64, _i64, _p]),
            "oracle_unswizzle_scales": (None, [_p, _i64, _i64, _p]),
            "oracle_dequant_nvfp4": (None, [_p, _p, ctypes.c_float, _i64, _i64,
                                            _p, _i64, _p]),
            "oracle_dequant_fp8": (None, [_p, _p, ctypes.c_int, _i64, _i64, _p,
                                          _i64, _p]),
            "oracle_gemm_f64": (None, [_p, _p, _i64, _i64, _i64, _p, _p, _p]),
            "oracle_round_bf16": (ctypes.c_uint16, [ctypes.c_double]),
            "oracle_round_bf16_array": (None, [_p, _i64, _p]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def _ptr(a: np.ndarray | None):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


def _bits(x) -> np.ndarray:
    """bf16 bit patterns as a C-contiguous uint16 array."""
    x = np.ascontiguousarray(x)
    assert x.dtype == np.uint16, "bf16 inputs are passed as uint16 bit arrays"
    return x


# ---------------------------------------------------------------- formats --

def num_threads() -> int:
    return _load().oracle_num_threads()


def set_num_threads(n: int) -> None:
    _load().oracle_set_num_threads(int(n))


def e2m1_decode(code: int) -> float:
    return _load().oracle_e2m1_decode(int(code))


def e2m1_encode(v: float) -> int:
    return _load().oracle_e2m1_encode(float(v))


def e4m3_decode(code: int) -> float:
    return _load().oracle_e4m3_decode(int(code))


def e4m3_encode(v: float) -> int:
    return _load().oracle_e4m3_encode(float(v))


def bf16_to_f32(bits: int) -> float:
    return _load().oracle_bf16_to_f32(int(bits))


def round_bf16(v: float) -> int:
    """bf16 bits of the nearest bf16 to an fp64 value (ties to even)."""
    return _load().oracle_round_bf16(float(v))


def round_bf16_array(v: np.ndarray) -> np.ndarray:
    v = np.ascontiguousarray(v, np.float64)
    out = np.empty(v.shape, np.uint16)
    _load().oracle_round_bf16_array(_ptr(v), v.size, _ptr(out))
    return out


# ---------------------------------------------------------------- scales ---

def amax_bf16(x) -> float:
    x = _bits(x)
    return _load().oracle_amax_bf16(_ptr(x), x.size)


def nvfp4_tensor_scale(amax: float) -> float:
    return _load().oracle_nvfp4_tensor_scale(amax)


def fp8_tensor_scale(amax: float) -> float:
    return _load().oracle_fp8_tensor_scale(amax)


def encode_scale(s_dec: float) -> float:
    return _load().oracle_encode_scale(s_dec)


# ---------------------------------------------------------------- quantizers

def quant_nvfp4(x, s_dec: float | None = None):
    """NVFP4-quantize bf16 bits [rows, K].  ``s_dec=None`` takes the dynamic
    tensor scale amax/2688.  Returns (codes [rows, K/2] u8, canonical scales
    [rows, K/16] u8, s_dec as np.float32)."""
    x = _bits(x)
    rows, K = x.shape
    assert K % 16 == 0
    lib = _load()
    if s_dec is None:
        s_dec = lib.oracle_nvfp4_tensor_scale(lib.oracle_amax_bf16(_ptr(x), x.size))
    s_dec = float(np.float32(s_dec))
    codes = np.empty((rows, K // 2), np.uint8)
    scales = np.empty((rows, K // 16), np.uint8)
    lib.oracle_quant_nvfp4(_ptr(x), rows, K, s_dec, _ptr(codes), _ptr(scales))
    return codes, scales, np.float32(s_dec)


def quant_fp8(x, s_dec: float | None = None):
    """FP8-quantize bf16 bits [rows, K] with one tensor scale (dynamic
    amax/448 when ``s_dec`` is None).  Returns (codes u8 [rows, K], s_dec)."""
    x = _bits(x)
    rows, K = x.shape
    lib = _load()
    if s_dec is None:
        s_dec = lib.oracle_fp8_tensor_scale(lib.oracle_amax_bf16(_ptr(x), x.size))
    s_dec = float(np.float32(s_dec))
    codes = np.empty((rows, K), np.uint8)
    lib.oracle_quant_fp8(_ptr(x), rows, K, s_dec, _ptr(codes))
    return codes, np.float32(s_dec)


def quant_fp8_rows(w):
    """FP8-quantize bf16 bits [rows, K] with one scale per row (output
    channel).  Returns (codes u8 [rows, K], s_dec f32 [rows])."""
    w = _bits(w)
    rows, K = w.shape
    codes = np.empty((rows, K), np.uint8)
    s = np.empty(rows, np.float32)
    _load().oracle_quant_fp8_rows(_ptr(w), rows, K, _ptr(codes), _ptr(s))
    return codes, s


# ---------------------------------------------------------------- layout ---

def swizzled_scale_bytes(rows: int, K: int) -> int:
    return _load().oracle_swizzled_scale_bytes(rows, K)


def swizzle_offset(r: int, c: int, K: int) -> int:
    return _load().oracle_swizzle_offset(r, c, K)


def swizzle_scales(canon: np.ndarray, K: int) -> np.ndarray:
    canon = np.ascontiguousarray(canon, np.uint8)
    rows = canon.shape[0]
    out = np.empty(swizzled_scale_bytes(rows, K), np.uint8)
    _load().oracle_swizzle_scales(_ptr(canon), rows, K, _ptr(out))
    return out


def unswizzle_scales(swz: np.ndarray, rows: int, K: int) -> np.ndarray:
    swz = np.ascontiguousarray(swz, np.uint8)
    assert swz.size >= swizzled_scale_bytes(rows, K)
    out = np.empty((rows, K // 16), np.uint8)
    _load().oracle_unswizzle_scales(_ptr(swz), rows, K, _ptr(out))
    return out


# ---------------------------------------------------------------- GEMM -----

def _sel(rows_sel, rows):
    if rows_sel is None:
        return None, rows
    s = np.ascontiguousarray(rows_sel, np.int64)
    assert s.size == 0 or (s.min() >= 0 and s.max() < rows)
    return s, s.size


def dequant_nvfp4(codes, scales_canon, s_dec, rows_sel=None) -> np.ndarray:
    codes = np.ascontiguousarray(codes, np.uint8)
    scales_canon = np.ascontiguousarray(scales_canon, np.uint8)
    rows, K = codes.shape[0], codes.shape[1] * 2
    sel, n = _sel(rows_sel, rows)
    out = np.empty((n, K), np.float64)
    _load().oracle_dequant_nvfp4(_ptr(codes), _ptr(scales_canon),
                                 float(np.float32(s_dec)), rows, K, _ptr(sel),
                                 n, _ptr(out))
    return out


def dequant_fp8(codes, s_dec, rows_sel=None) -> np.ndarray:
    codes = np.ascontiguousarray(codes, np.uint8)
    rows, K = codes.shape
    s = np.ascontiguousarray(np.atleast_1d(s_dec), np.float32)
    assert s.size in (1, rows)
    per_row = 1 if s.size > 1 else 0
    sel, n = _sel(rows_sel, rows)
    out = np.empty((n, K), np.float64)
    _load().oracle_dequant_fp8(_ptr(codes), _ptr(s), per_row, rows, K,
                               _ptr(sel), n, _ptr(out))
    return out


def gemm_f64(a: np.ndarray, w: np.ndarray):
    """y = a @ w.T in fp64 plus the row norms ||a_m|| and ||w_n||."""
    a = np.ascontiguousarray(a, np.float64)
    w = np.ascontiguousarray(w, np.float64)
    M, K = a.shape
    N = w.shape[0]
    assert w.shape[1] == K
    y = np.empty((M, N), np.float64)
    na = np.empty(M, np.float64)
    nw = np.empty(N, np.float64)
    _load().oracle_gemm_f64(_ptr(a), _ptr(w), M, N, K, _ptr(y), _ptr(na), _ptr(nw))
    return y, na, nw


def gemm_nvfp4(a_q, w_q, rows_sel=None):
    """Exact fp64 result of the NVFP4 linear on quantized operands.
    a_q, w_q = (codes, canonical scales, s_dec).  Returns (y, ||a||, ||w||)
    for the selected rows of A."""
    a = dequant_nvfp4(*a_q, rows_sel=rows_sel)
    w = dequant_nvfp4(*w_q)
    return gemm_f64(a, w)


def gemm_fp8(a_q, w_q, rows_sel=None):
    """Exact fp64 result of the FP8 linear.  a_q = (codes, s_dec scalar),
    w_q = (codes, s_dec per row)."""
    a = dequant_fp8(a_q[0], np.float32(a_q[1]), rows_sel=rows_sel)
    w = dequant_fp8(w_q[0], np.asarray(w_q[1], np.float32))
    return gemm_f64(a, w)
