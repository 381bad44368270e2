"""Thin ctypes binding of libqlin (include/qlin.h): same names, argument
marshalling only.  Every step runs in the library's CUDA kernels; PyTorch
supplies device memory and the current stream.  There is no CPU fallback: if
the library is missing or fails to load, every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading
from dataclasses import dataclass

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libqlin.so")

QLIN_FMT_NVFP4 = 1
QLIN_FMT_FP8 = 2
STATUS = {0: "QLIN_OK", 1: "QLIN_ERR_INVALID_ARG", 2: "QLIN_ERR_UNSUPPORTED",
          3: "QLIN_ERR_MISALIGNED", 4: "QLIN_ERR_CUDA", 5: "QLIN_ERR_TIMEOUT",
          6: "QLIN_ERR_WORKSPACE"}

# Every function declared in include/qlin.h.
EXPORTS = ("qlin_nvfp4_scale_bytes", "qlin_workspace_size", "qlin_quantize_act_nvfp4",
           "qlin_quantize_act_fp8", "qlin_quantize_weight", "qlin_gemm_nvfp4", "qlin_gemm_fp8",
           "qlin_linear_fused", "qlin_linear_fused_fp8", "qlin_linear_dynamic", "qlin_gemm_bf16",
           "qlin_gemm_fp16", "qlin_quantize_act_nvfp4_noalloc",
           "qlin_sync_status", "qlin_selftest_bounded_wait",
           "qlin_set_wait_timeout_ns", "qlin_status_str", "qlin_last_error")


class QlinError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str = ""):
        self.status = status
        super().__init__(f"{where}: {STATUS.get(status, status)}" + (f" ({detail})" if detail else ""))


class NVFP4Desc(ctypes.Structure):
    _fields_ = [("codes", ctypes.c_void_p), ("scales", ctypes.c_void_p),
                ("tensor_scale", ctypes.c_void_p), ("rows", ctypes.c_int64),
                ("K", ctypes.c_int64)]


class FP8Desc(ctypes.Structure):
    _fields_ = [("codes", ctypes.c_void_p), ("scale", ctypes.c_void_p),
                ("rows", ctypes.c_int64), ("K", ctypes.c_int64),
                ("per_channel", ctypes.c_int32)]


_lock = threading.Lock()
_lib = None


def load_library(path: str = LIB_PATH):
    """Load libqlin.so (built by ``paper_2609_21849_gb300.build``)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(path):
            raise RuntimeError(f"libqlin is not built ({path} missing); run "
                               "python -m paper_2609_21849_gb300.build")
        lib = ctypes.CDLL(path)
        i64, p, sz = ctypes.c_int64, ctypes.c_void_p, ctypes.c_size_t
        sig = {
            "qlin_nvfp4_scale_bytes": (sz, [i64, i64]),
            "qlin_workspace_size": (sz, [i64, i64]),
            "qlin_quantize_act_nvfp4": (ctypes.c_int, [p, i64, i64, p, ctypes.POINTER(NVFP4Desc), p, sz, p]),
            "qlin_quantize_act_fp8": (ctypes.c_int, [p, i64, i64, p, ctypes.POINTER(FP8Desc), p, sz, p]),
            "qlin_quantize_weight": (ctypes.c_int, [p, i64, i64, ctypes.c_int, p, p, sz, p]),
            "qlin_gemm_nvfp4": (ctypes.c_int, [ctypes.POINTER(NVFP4Desc), ctypes.POINTER(NVFP4Desc), p, p]),
            "qlin_gemm_fp8": (ctypes.c_int, [ctypes.POINTER(FP8Desc), ctypes.POINTER(FP8Desc), p, p]),
            "qlin_linear_fused": (ctypes.c_int, [ctypes.POINTER(NVFP4Desc), ctypes.POINTER(NVFP4Desc), p, p,
                                                 ctypes.POINTER(NVFP4Desc), i64, p]),
            "qlin_gemm_bf16": (ctypes.c_int, [p, i64, p, i64, i64, i64, p, p]),
            "qlin_gemm_fp16": (ctypes.c_int, [p, i64, p, i64, i64, i64, p, p]),
            "qlin_linear_fused_fp8": (ctypes.c_int, [ctypes.POINTER(FP8Desc), ctypes.POINTER(FP8Desc), p, p,
                                                     ctypes.POINTER(FP8Desc), i64, p]),
            "qlin_linear_dynamic": (ctypes.c_int, [ctypes.POINTER(NVFP4Desc), ctypes.POINTER(NVFP4Desc), p,
                                                   ctypes.POINTER(NVFP4Desc), p, sz, p]),
            "qlin_quantize_act_nvfp4_noalloc": (ctypes.c_int, [p, i64, i64, ctypes.POINTER(NVFP4Desc), p]),
            "qlin_sync_status": (ctypes.c_int, [p]),
            "qlin_selftest_bounded_wait": (ctypes.c_int, [ctypes.c_uint64, p]),
            "qlin_set_wait_timeout_ns": (None, [ctypes.c_uint64]),
            "qlin_status_str": (ctypes.c_char_p, [ctypes.c_int]),
            "qlin_last_error": (ctypes.c_char_p, []),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def _check(status: int, where: str):
    if status != 0:
        lib = load_library()
        detail = lib.qlin_last_error().decode() if status == 4 else ""
        raise QlinError(status, where, detail)


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _bf16_2d(x: torch.Tensor):
    if x.dtype != torch.bfloat16 or x.dim() != 2 or not x.is_contiguous() or not x.is_cuda:
        raise ValueError("expected a contiguous 2-D bf16 CUDA tensor")
    return x.shape[0], x.shape[1]


# ----------------------------------------------------------- containers ---

@dataclass
class NVFP4Tensor:
    """NVFP4 operand [rows, K] in device memory: packed e2m1 codes, E4M3 block
    scales in the tensor-core layout, fp32 tensor scale."""
    codes: torch.Tensor          # uint8 [rows, K/2]
    scales: torch.Tensor         # uint8 [qlin_nvfp4_scale_bytes(rows, K)]
    tensor_scale: torch.Tensor   # float32 [1]
    rows: int
    K: int

    def desc(self) -> NVFP4Desc:
        return NVFP4Desc(self.codes.data_ptr(), self.scales.data_ptr(),
                         self.tensor_scale.data_ptr(), self.rows, self.K)


@dataclass
class FP8Tensor:
    """FP8 operand [rows, K]: E4M3 codes plus one fp32 scale (per_channel=0)
    or one per row (per_channel=1)."""
    codes: torch.Tensor          # uint8 [rows, K]
    scale: torch.Tensor          # float32 [1] or [rows]
    rows: int
    K: int
    per_channel: int

    def desc(self) -> FP8Desc:
        return FP8Desc(self.codes.data_ptr(), self.scale.data_ptr(), self.rows, self.K,
                       self.per_channel)


def qlin_nvfp4_scale_bytes(rows: int, K: int) -> int:
    return load_library().qlin_nvfp4_scale_bytes(rows, K)


def qlin_workspace_size(M: int = 0, K: int = 0) -> int:
    return load_library().qlin_workspace_size(M, K)


def alloc_nvfp4(rows: int, K: int, device="cuda") -> NVFP4Tensor:
    nb = qlin_nvfp4_scale_bytes(rows, K)
    if nb == 0:
        raise ValueError(f"invalid NVFP4 shape [{rows}, {K}]")
    return NVFP4Tensor(torch.empty((rows, K // 2), dtype=torch.uint8, device=device),
                       torch.zeros(nb, dtype=torch.uint8, device=device),
                       torch.zeros(1, dtype=torch.float32, device=device), rows, K)


def alloc_fp8(rows: int, K: int, per_channel: bool, device="cuda") -> FP8Tensor:
    return FP8Tensor(torch.empty((rows, K), dtype=torch.uint8, device=device),
                     torch.zeros(rows if per_channel else 1, dtype=torch.float32, device=device),
                     rows, K, 1 if per_channel else 0)


def alloc_workspace(device="cuda") -> torch.Tensor:
    return torch.zeros(qlin_workspace_size(), dtype=torch.uint8, device=device)


# ------------------------------------------------------------ the calls ---

def qlin_quantize_act_nvfp4(x: torch.Tensor, static_scale: torch.Tensor | None = None,
                            out: NVFP4Tensor | None = None, workspace: torch.Tensor | None = None,
                            stream=None) -> NVFP4Tensor:
    M, K = _bf16_2d(x)
    out = out if out is not None else alloc_nvfp4(M, K, x.device)
    if static_scale is None and workspace is None:
        workspace = alloc_workspace(x.device)
    d = out.desc()
    _check(load_library().qlin_quantize_act_nvfp4(
        _ptr(x), M, K, _ptr(static_scale), ctypes.byref(d), _ptr(workspace),
        0 if workspace is None else workspace.numel(), _stream(stream)), "qlin_quantize_act_nvfp4")
    return out


def qlin_quantize_act_nvfp4_noalloc(x: torch.Tensor, out: NVFP4Tensor, stream=None) -> NVFP4Tensor:
    """Dynamic-scale NVFP4 quantization for callers that cannot allocate device
    memory: no workspace argument; the library keeps the amax scratch in its
    own static device array.  ``out`` must be supplied by the caller.  Calls
    that overlap on the GPU share that scratch and race; the first call on a
    device should come before any stream capture."""
    M, K = _bf16_2d(x)
    d = out.desc()
    _check(load_library().qlin_quantize_act_nvfp4_noalloc(_ptr(x), M, K, ctypes.byref(d),
                                                          _stream(stream)),
           "qlin_quantize_act_nvfp4_noalloc")
    return out


def qlin_quantize_act_fp8(x: torch.Tensor, static_scale: torch.Tensor | None = None,
                          out: FP8Tensor | None = None, workspace: torch.Tensor | None = None,
                          stream=None) -> FP8Tensor:
    M, K = _bf16_2d(x)
    out = out if out is not None else alloc_fp8(M, K, False, x.device)
    if static_scale is None and workspace is None:
        workspace = alloc_workspace(x.device)
    d = out.desc()
    _check(load_library().qlin_quantize_act_fp8(
        _ptr(x), M, K, _ptr(static_scale), ctypes.byref(d), _ptr(workspace),
        0 if workspace is None else workspace.numel(), _stream(stream)), "qlin_quantize_act_fp8")
    return out


def qlin_quantize_weight(w: torch.Tensor, fmt: int, out=None, workspace: torch.Tensor | None = None,
                         stream=None):
    N, K = _bf16_2d(w)
    if fmt == QLIN_FMT_NVFP4:
        out = out if out is not None else alloc_nvfp4(N, K, w.device)
        workspace = workspace if workspace is not None else alloc_workspace(w.device)
    elif fmt == QLIN_FMT_FP8:
        out = out if out is not None else alloc_fp8(N, K, True, w.device)
    else:
        raise ValueError("fmt must be QLIN_FMT_NVFP4 or QLIN_FMT_FP8")
    d = out.desc()
    _check(load_library().qlin_quantize_weight(
        _ptr(w), N, K, fmt, ctypes.cast(ctypes.byref(d), ctypes.c_void_p), _ptr(workspace),
        0 if workspace is None else workspace.numel(), _stream(stream)), "qlin_quantize_weight")
    return out


def _y_out(y, M, N, device):
    if y is None:
        return torch.empty((M, N), dtype=torch.bfloat16, device=device)
    if y.dtype != torch.bfloat16 or tuple(y.shape) != (M, N) or not y.is_contiguous():
        raise ValueError("y must be a contiguous bf16 [M, N] tensor")
    return y


def qlin_gemm_nvfp4(A: NVFP4Tensor, W: NVFP4Tensor, y: torch.Tensor | None = None,
                    stream=None) -> torch.Tensor:
    y = _y_out(y, A.rows, W.rows, A.codes.device)
    da, dw = A.desc(), W.desc()
    _check(load_library().qlin_gemm_nvfp4(ctypes.byref(da), ctypes.byref(dw), _ptr(y),
                                          _stream(stream)), "qlin_gemm_nvfp4")
    return y


def qlin_gemm_fp8(A: FP8Tensor, W: FP8Tensor, y: torch.Tensor | None = None,
                  stream=None) -> torch.Tensor:
    y = _y_out(y, A.rows, W.rows, A.codes.device)
    da, dw = A.desc(), W.desc()
    _check(load_library().qlin_gemm_fp8(ctypes.byref(da), ctypes.byref(dw), _ptr(y),
                                        _stream(stream)), "qlin_gemm_fp8")
    return y


def qlin_linear_fused(A: NVFP4Tensor, W: NVFP4Tensor, y: torch.Tensor | None,
                      next_scale: torch.Tensor | None, y_q: NVFP4Tensor | None,
                      rq_col0: int = 0, stream=None):
    da, dw = A.desc(), W.desc()
    dq = y_q.desc() if y_q is not None else None
    _check(load_library().qlin_linear_fused(
        ctypes.byref(da), ctypes.byref(dw), _ptr(y), _ptr(next_scale),
        ctypes.byref(dq) if dq is not None else None, rq_col0, _stream(stream)),
        "qlin_linear_fused")
    return y, y_q


def qlin_linear_fused_fp8(A: FP8Tensor, W: FP8Tensor, y: torch.Tensor | None,
                          next_scale: torch.Tensor, y_q: FP8Tensor, rq_col0: int = 0, stream=None):
    """FP8 linear whose epilogue also writes the next layer's FP8 input
    (columns [rq_col0, rq_col0 + y_q.K) of bf16(y), static scale)."""
    da, dw, dq = A.desc(), W.desc(), y_q.desc()
    _check(load_library().qlin_linear_fused_fp8(
        ctypes.byref(da), ctypes.byref(dw), _ptr(y), _ptr(next_scale), ctypes.byref(dq), rq_col0,
        _stream(stream)), "qlin_linear_fused_fp8")
    return y, y_q


def _gemm16(name: str, dtype, a: torch.Tensor, w: torch.Tensor, y, stream):
    if a.dtype != dtype or w.dtype != dtype or a.dim() != 2 or a.stride(1) != 1:
        raise ValueError(f"a, w: {dtype} matrices with unit column stride")
    w = w.contiguous()
    M, K = a.shape
    N = w.shape[0]
    if y is None:
        y = torch.empty((M, N), dtype=dtype, device=a.device)
    elif y.dtype != dtype or not y.is_contiguous() or tuple(y.shape) != (M, N):
        raise ValueError(f"y: contiguous {dtype} [{M}, {N}]")
    _check(getattr(load_library(), name)(_ptr(a), a.stride(0), _ptr(w), M, N, K, _ptr(y),
                                         _stream(stream)), name)
    return y


def qlin_gemm_bf16(a: torch.Tensor, w: torch.Tensor, y: torch.Tensor | None = None, stream=None):
    """y = a w^T for bf16 a [M, K] (rows may be strided: any view with unit
    column stride) and w [N, K]; bf16 y [M, N]."""
    return _gemm16("qlin_gemm_bf16", torch.bfloat16, a, w, y, stream)


def qlin_gemm_fp16(a: torch.Tensor, w: torch.Tensor, y: torch.Tensor | None = None, stream=None):
    """As qlin_gemm_bf16 with fp16 operands and an fp16 y."""
    return _gemm16("qlin_gemm_fp16", torch.float16, a, w, y, stream)


def qlin_linear_dynamic(A: NVFP4Tensor, W: NVFP4Tensor, y: torch.Tensor | None = None,
                        y_q: NVFP4Tensor | None = None, workspace: torch.Tensor | None = None,
                        stream=None):
    """y = A W^T (bf16) and y_q = NVFP4(y) with y's own dynamic tensor scale,
    the amax taken in the GEMM epilogue.  Returns (y, y_q)."""
    M, N = A.rows, W.rows
    if y is None:
        y = torch.empty((M, N), dtype=torch.bfloat16, device=A.codes.device)
    if y_q is None:
        y_q = alloc_nvfp4(M, N, A.codes.device)
    if workspace is None:
        workspace = alloc_workspace(A.codes.device)
    da, dw, dq = A.desc(), W.desc(), y_q.desc()
    _check(load_library().qlin_linear_dynamic(
        ctypes.byref(da), ctypes.byref(dw), _ptr(y), ctypes.byref(dq), _ptr(workspace),
        workspace.numel(), _stream(stream)), "qlin_linear_dynamic")
    return y, y_q


def qlin_sync_status(stream=None) -> int:
    """Synchronise `stream`; return (and clear) the device status code."""
    return load_library().qlin_sync_status(_stream(stream))


def qlin_selftest_bounded_wait(timeout_ns: int, stream=None) -> None:
    _check(load_library().qlin_selftest_bounded_wait(timeout_ns, _stream(stream)),
           "qlin_selftest_bounded_wait")


def qlin_set_wait_timeout_ns(ns: int) -> None:
    load_library().qlin_set_wait_timeout_ns(ns)


def qlin_status_str(status: int) -> str:
    return load_library().qlin_status_str(status).decode()


def qlin_last_error() -> str:
    return load_library().qlin_last_error().decode()
