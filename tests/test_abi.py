"""The C-ABI library loads, exports every function include/qlin.h declares,
and rejects bad arguments on the host before any CUDA call (no GPU needed)."""
import ctypes
import os
import re

import pytest

from conftest import ROOT


@pytest.fixture(scope="module")
def lib():
    from paper_2609_21849_gb300 import build, qlin
    build.build()
    return qlin.load_library()


def _declared(header="qlin.h"):
    src = open(os.path.join(ROOT, "include", header)).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(qlin_\w+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("qlin_quantize_weight", "qlin_quantize_act_nvfp4", "qlin_quantize_act_fp8",
              "qlin_gemm_nvfp4", "qlin_gemm_fp8", "qlin_linear_fused"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    from paper_2609_21849_gb300 import qlin
    for name in _declared():
        assert hasattr(lib, name), name
    assert sorted(qlin.EXPORTS) == _declared()


def test_probe_library_exports_its_header(lib):
    # the tensor-core rate probe of the measurement harness: its own library
    from paper_2609_21849_gb300 import build
    probe = ctypes.CDLL(build.PROBE_LIB)
    names = _declared("qlin_probe.h")
    assert names == ["qlin_probe_fill", "qlin_probe_mma", "qlin_probe_scale_copy"]
    for name in names:
        assert hasattr(probe, name), name
    f = probe.qlin_probe_mma
    f.restype = ctypes.c_int
    f.argtypes = [ctypes.c_int] * 5 + [ctypes.c_void_p] * 3
    one = ctypes.c_ulonglong(0)
    p1 = ctypes.addressof(one)
    # argument errors are returned before any launch
    assert f(4, 1, 256, 3, 16, p1, p1, None) == 1  # odd pair grid
    assert f(4, 0, 64, 2, 16, p1, p1, None) == 1   # no such case
    assert f(4, 0, 256, 2, 16, None, None, None) == 1
    g = probe.qlin_probe_scale_copy
    g.restype = ctypes.c_int
    g.argtypes = [ctypes.c_int] * 5 + [ctypes.c_void_p] * 3
    assert g(4, 12, 4, 3, 16, p1, p1, None) == 1   # odd pair grid
    assert g(5, 12, 4, 2, 16, p1, p1, None) == 1   # copies not a multiple of the warps
    assert g(9, 18, 4, 2, 16, p1, p1, None) == 1   # more than 8 copy warps
    assert g(4, 12, 4, 2, 16, None, None, None) == 1
    h = probe.qlin_probe_fill
    h.restype = ctypes.c_int
    h.argtypes = [ctypes.c_int] * 5 + [ctypes.c_void_p, ctypes.c_ulonglong] + [ctypes.c_void_p] * 3
    big = 1 << 30   # never dereferenced: the checks fail first
    assert h(2, 4, 2, 1, 16, 256, big, p1, p1, None) == 1          # no such mode
    assert h(0, 8, 8, 1, 16, 256, big, p1, p1, None) == 1          # 1 MB of rings
    assert h(0, 4, 2, 1, 16, 256, 1536 * 64, p1, p1, None) == 1    # fewer than 128 rows
    assert h(0, 4, 2, 1, 16, 256 + 64, big, p1, p1, None) == 1     # source not 128-byte aligned


def test_scale_bytes_and_workspace(lib):
    from paper_2609_21849_gb300 import qlin
    assert qlin.qlin_nvfp4_scale_bytes(128, 256) == 2048
    assert qlin.qlin_nvfp4_scale_bytes(129, 256) == 4096
    assert qlin.qlin_nvfp4_scale_bytes(4608, 3072) == 36 * 48 * 512
    assert qlin.qlin_nvfp4_scale_bytes(128, 100) == 0
    assert qlin.qlin_workspace_size(1, 64) >= 4


def test_argument_errors_return_before_launch(lib):
    from paper_2609_21849_gb300 import qlin
    d = qlin.NVFP4Desc(16, 16, 16, 128, 256)  # fake, never dereferenced
    # null input
    assert lib.qlin_quantize_act_nvfp4(None, 128, 256, None, ctypes.byref(d), 16, 256, None) == 1
    # K not a multiple of 64
    d2 = qlin.NVFP4Desc(16, 16, 16, 128, 96)
    assert lib.qlin_quantize_act_nvfp4(16, 128, 96, None, ctypes.byref(d2), 16, 256, None) == 1
    # rows mismatch between the descriptor and the call
    assert lib.qlin_quantize_act_nvfp4(16, 64, 256, None, ctypes.byref(d), 16, 256, None) == 1
    # misaligned input pointer
    assert lib.qlin_quantize_act_nvfp4(24, 128, 256, None, ctypes.byref(d), 16, 256, None) == 3
    # dynamic scale without workspace, with one smaller than qlin_workspace_size(), and with
    # one only 4-byte aligned (its first two words are read as one 64-bit load)
    assert lib.qlin_quantize_act_nvfp4(16, 128, 256, None, ctypes.byref(d), None, 0, None) == 6
    assert lib.qlin_quantize_act_nvfp4(16, 128, 256, None, ctypes.byref(d), 16, 28, None) == 6
    assert lib.qlin_quantize_act_nvfp4(16, 128, 256, None, ctypes.byref(d), 20, 256, None) == 3
    f8 = qlin.FP8Desc(16, 16, 128, 256, 0)
    assert lib.qlin_quantize_act_fp8(16, 128, 256, None, ctypes.byref(f8), 20, 256, None) == 3
    # GEMM: K mismatch, N not a multiple of 64, nothing to write
    a = qlin.NVFP4Desc(16, 16, 16, 128, 256)
    w = qlin.NVFP4Desc(16, 16, 16, 256, 512)
    assert lib.qlin_gemm_nvfp4(ctypes.byref(a), ctypes.byref(w), 16, None) == 1
    w = qlin.NVFP4Desc(16, 16, 16, 96, 256)
    assert lib.qlin_gemm_nvfp4(ctypes.byref(a), ctypes.byref(w), 16, None) == 1
    w = qlin.NVFP4Desc(16, 16, 16, 256, 256)
    assert lib.qlin_linear_fused(ctypes.byref(a), ctypes.byref(w), None, None, None, 0, None) == 1
    # re-quantization window outside the output
    q = qlin.NVFP4Desc(16, 16, 16, 128, 128)
    assert lib.qlin_linear_fused(ctypes.byref(a), ctypes.byref(w), 16, 16, ctypes.byref(q), 192,
                                 None) == 1
    # dynamic chain: output descriptor of the wrong shape, missing workspace
    q = qlin.NVFP4Desc(16, 16, 16, 128, 128)
    assert lib.qlin_linear_dynamic(ctypes.byref(a), ctypes.byref(w), 16, ctypes.byref(q), 16, 256,
                                   None) == 1
    q = qlin.NVFP4Desc(16, 16, 16, 128, 256)
    assert lib.qlin_linear_dynamic(ctypes.byref(a), ctypes.byref(w), 16, ctypes.byref(q), None, 0,
                                   None) == 6
    assert lib.qlin_linear_dynamic(ctypes.byref(a), ctypes.byref(w), None, ctypes.byref(q), 16, 256,
                                   None) == 1
    # FP8 fused re-quantization without its static scale
    f8 = qlin.FP8Desc(16, 16, 128, 256, 0)
    f8w = qlin.FP8Desc(16, 16, 256, 256, 1)
    f8q = qlin.FP8Desc(16, 16, 128, 256, 0)
    assert lib.qlin_linear_fused_fp8(ctypes.byref(f8), ctypes.byref(f8w), 16, None, ctypes.byref(f8q),
                                     0, None) == 1
    # bf16 GEMM: K not a multiple of 64, row stride below K, misaligned row stride
    assert lib.qlin_gemm_bf16(16, 96, 16, 128, 128, 96, 16, None) == 1
    assert lib.qlin_gemm_bf16(16, 64, 16, 128, 128, 128, 16, None) == 1
    assert lib.qlin_gemm_bf16(16, 132, 16, 128, 128, 128, 16, None) == 3
    # the fp16 linear shares the checks
    assert lib.qlin_gemm_fp16(None, 128, 16, 128, 128, 128, 16, None) == 1
    assert lib.qlin_gemm_fp16(16, 96, 16, 128, 128, 96, 16, None) == 1
    assert lib.qlin_gemm_fp16(16, 132, 16, 128, 128, 128, 16, None) == 3
    # FP8: per-channel activation descriptor is rejected; unknown weight format
    f = qlin.FP8Desc(16, 16, 128, 256, 1)
    assert lib.qlin_quantize_act_fp8(16, 128, 256, 16, ctypes.byref(f), None, 0, None) == 1
    assert lib.qlin_quantize_weight(16, 128, 256, 7, ctypes.byref(f), None, 0, None) == 2
    assert lib.qlin_status_str(5) == b"device wait timed out"


def test_python_binding_fails_loudly_without_library(tmp_path):
    from paper_2609_21849_gb300 import qlin
    saved = qlin._lib
    try:
        qlin._lib = None
        with pytest.raises(RuntimeError, match="not built"):
            qlin.load_library(str(tmp_path / "missing.so"))
    finally:
        qlin._lib = saved


def test_empty_dimensions_are_rejected_before_launch(lib):
    # an empty matrix (M, N or K of 0) has nothing to compute; every entry
    # point reports it as an argument error instead of launching
    from paper_2609_21849_gb300 import qlin
    d0 = qlin.NVFP4Desc(16, 16, 16, 0, 256)
    assert lib.qlin_quantize_act_nvfp4(16, 0, 256, 16, ctypes.byref(d0), 16, 256, None) == 1
    dk = qlin.NVFP4Desc(16, 16, 16, 128, 0)
    assert lib.qlin_quantize_act_nvfp4(16, 128, 0, 16, ctypes.byref(dk), 16, 256, None) == 1
    assert lib.qlin_quantize_act_nvfp4_noalloc(16, 0, 256, ctypes.byref(d0), None) == 1
    f0 = qlin.FP8Desc(16, 16, 0, 256, 0)
    assert lib.qlin_quantize_act_fp8(16, 0, 256, 16, ctypes.byref(f0), 16, 256, None) == 1
    assert lib.qlin_quantize_weight(16, 0, 256, 1, ctypes.byref(d0), 16, 256, None) == 1
    w = qlin.NVFP4Desc(16, 16, 16, 256, 256)
    assert lib.qlin_gemm_nvfp4(ctypes.byref(d0), ctypes.byref(w), 16, None) == 1
    a = qlin.NVFP4Desc(16, 16, 16, 128, 256)
    assert lib.qlin_gemm_nvfp4(ctypes.byref(a), ctypes.byref(d0), 16, None) == 1
    fw = qlin.FP8Desc(16, 16, 256, 256, 1)
    assert lib.qlin_gemm_fp8(ctypes.byref(f0), ctypes.byref(fw), 16, None) == 1
    assert lib.qlin_gemm_bf16(16, 128, 16, 0, 128, 128, 16, None) == 1
    assert lib.qlin_gemm_fp16(16, 128, 16, 128, 0, 128, 16, None) == 1
