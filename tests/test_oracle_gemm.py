"""Pins of the oracle's linear-layer result y = x W^T over quantized operands.

The quantized linear of Sec. 4 computes the GEMM over dequantized FP8 / NVFP4
operands; its exact value is the fp64 dot product of the decoded, scaled
operands.  These tests check the oracle against brute force with an
independent decoder (ml_dtypes), closed forms and dyadic exact cases.
"""
import numpy as np
import pytest

from paper_2609_21849_gb300 import synthetic

ml_dtypes = pytest.importorskip("ml_dtypes")


def _decode_nvfp4_independent(codes, scales, s_dec):
    lo = (codes & 0xF).view(ml_dtypes.float4_e2m1fn).astype(np.float64)
    hi = (codes >> 4).view(ml_dtypes.float4_e2m1fn).astype(np.float64)
    v = np.empty((codes.shape[0], codes.shape[1] * 2))
    v[:, 0::2], v[:, 1::2] = lo, hi
    sc = scales.view(ml_dtypes.float8_e4m3fn).astype(np.float64)
    return v * np.repeat(sc, 16, axis=1) * float(s_dec)


@pytest.mark.parametrize("M,N,K", [(1, 1, 16), (3, 5, 32), (8, 8, 64), (7, 2, 48)])
def test_nvfp4_gemm_brute_force(oracle, M, N, K):
    rng = np.random.default_rng(M * 100 + N * 10 + K)
    ca = rng.integers(0, 256, (M, K // 2), dtype=np.uint8)
    cw = rng.integers(0, 256, (N, K // 2), dtype=np.uint8)
    sa = rng.integers(0, 0x7F, (M, K // 16), dtype=np.uint8)   # finite scales
    sw = rng.integers(0, 0x7F, (N, K // 16), dtype=np.uint8)
    da, dw = np.float32(0.37), np.float32(1.9)
    y, na, nw = oracle.gemm_nvfp4((ca, sa, da), (cw, sw, dw))
    a = _decode_nvfp4_independent(ca, sa, da)
    w = _decode_nvfp4_independent(cw, sw, dw)
    # brute force, one dot product at a time
    for m in range(M):
        for n in range(N):
            ref = sum(a[m, k] * w[n, k] for k in range(K))
            assert abs(y[m, n] - ref) <= 1e-12 * (np.abs(a[m]) @ np.abs(w[n]) + 1e-300)
        assert abs(na[m] - np.sqrt((a[m] ** 2).sum())) <= 1e-12 * na[m] + 1e-300
    for n in range(N):
        assert abs(nw[n] - np.sqrt((w[n] ** 2).sum())) <= 1e-12 * nw[n] + 1e-300


def test_nvfp4_gemm_dyadic_exact(oracle):
    # power-of-two scales and S_dec = 1: every product is dyadic and the sum
    # is exact in fp64, so the oracle must equal numpy's matmul exactly.
    M, N, K = 16, 24, 128
    rng = np.random.default_rng(0)
    ca = rng.integers(0, 256, (M, K // 2), dtype=np.uint8)
    cw = rng.integers(0, 256, (N, K // 2), dtype=np.uint8)
    pow2 = np.array([0x30, 0x38, 0x40, 0x48, 0x28], np.uint8)    # 0.5, 1, 2, 4, 0.25
    sa = rng.choice(pow2, (M, K // 16))
    sw = rng.choice(pow2, (N, K // 16))
    y, _, _ = oracle.gemm_nvfp4((ca, sa, 1.0), (cw, sw, 1.0))
    a = _decode_nvfp4_independent(ca, sa, 1.0)
    w = _decode_nvfp4_independent(cw, sw, 1.0)
    assert np.array_equal(y, a @ w.T)


def test_nvfp4_gemm_selects_transposed_weight(oracle):
    # A = "identity": row m is 1.0 at k = m and 0 elsewhere, so y[m, n] = W[n, m]:
    # catches a transposed operand or a swapped index.
    M, N, K = 16, 8, 64
    ca = np.zeros((M, K // 2), np.uint8)
    for m in range(M):
        ca[m, m // 2] = 0x2 << (4 * (m % 2))        # e2m1 code 2 = 1.0
    sa = np.full((M, K // 16), 0x38, np.uint8)        # scale 1.0
    rng = np.random.default_rng(4)
    cw = rng.integers(0, 256, (N, K // 2), dtype=np.uint8)
    sw = rng.integers(0x20, 0x50, (N, K // 16), dtype=np.uint8)
    y, _, _ = oracle.gemm_nvfp4((ca, sa, 1.0), (cw, sw, 1.0))
    w = _decode_nvfp4_independent(cw, sw, 1.0)
    assert np.array_equal(y, w[:, :M].T)


def test_nvfp4_gemm_row_selection(oracle):
    x, w = synthetic.tiny_nvfp4(M=32, K=64, N=16)
    aq = oracle.quant_nvfp4(x)
    wq = oracle.quant_nvfp4(w)
    y_all, na_all, _ = oracle.gemm_nvfp4(aq, wq)
    sel = np.array([31, 0, 7])
    y_sel, na_sel, _ = oracle.gemm_nvfp4(aq, wq, rows_sel=sel)
    assert np.array_equal(y_sel, y_all[sel]) and np.array_equal(na_sel, na_all[sel])


def test_fp8_gemm_brute_force(oracle):
    M, N, K = 5, 6, 40
    rng = np.random.default_rng(2)
    ca = rng.integers(0, 256, (M, K), dtype=np.uint8)
    ca[(ca & 0x7F) == 0x7F] = 0x11                    # no NaN codes
    cw = rng.integers(0, 256, (N, K), dtype=np.uint8)
    cw[(cw & 0x7F) == 0x7F] = 0x22
    sa = np.float32(0.03)
    sw = rng.uniform(0.001, 0.01, N).astype(np.float32)
    y, _, _ = oracle.gemm_fp8((ca, sa), (cw, sw))
    a = ca.view(ml_dtypes.float8_e4m3fn).astype(np.float64) * float(sa)
    w = cw.view(ml_dtypes.float8_e4m3fn).astype(np.float64) * sw.astype(np.float64)[:, None]
    for m in range(M):
        for n in range(N):
            ref = sum(a[m, k] * w[n, k] for k in range(K))
            assert abs(y[m, n] - ref) <= 1e-12 * (np.abs(a[m]) @ np.abs(w[n]))


def test_quantized_linear_tracks_bf16_linear(oracle):
    # End-to-end sanity on the tiny workload: the NVFP4 linear stays close to
    # the unquantized product (4-bit error, not an exact pin).
    x, w = synthetic.tiny_nvfp4()
    y, na, nw = oracle.gemm_nvfp4(oracle.quant_nvfp4(x), oracle.quant_nvfp4(w))
    ref = synthetic.bf16_to_f32(x).astype(np.float64) @ synthetic.bf16_to_f32(w).astype(np.float64).T
    rel = np.linalg.norm(y - ref) / np.linalg.norm(ref)
    assert rel < 0.2
