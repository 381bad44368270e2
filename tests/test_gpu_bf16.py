"""GPU parity of the unquantized bf16 and fp16 linears (the BF16 and FP16
rows of Table 2's precision ladder) on the tensor-core skeleton: y = a w^T
against the exact fp64 product of the same 16-bit inputs."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2609_21849_gb300 import qlin, synthetic

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from gpu_util import bf16_bits, gemm_errors, sample_rows, to_dev

# fp32 accumulation, bf16 output: the error against the exact result is the
# output rounding (2^-9 of |y| <= |a||w|) plus accumulation rounding
BF16_TOL = 4e-3


def _f64(bits):
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _check(a_bits, w_bits, y, rows, label):
    a, w = _f64(a_bits[rows]), _f64(w_bits)
    yref, na, nw = oracle.gemm_f64(a, w)
    err, exact = gemm_errors(bf16_bits(y)[rows], yref, na, nw)
    assert err.max() <= BF16_TOL, (label, err.max())
    assert exact >= 0.95, (label, exact)


@pytest.mark.parametrize("M,N,K", [(1, 64, 64), (130, 320, 192), (333, 512, 1088), (4608, 3072, 3072)])
def test_bf16_linear(M, N, K):
    a = synthetic.act_entry_outliers(M + 2 * N + K, M, K)
    (w,) = synthetic.weights(N + K, [(N, K)], 0.02)
    y = qlin.qlin_gemm_bf16(to_dev(a), to_dev(w))
    assert qlin.qlin_sync_status() == 0
    _check(a, w, y, sample_rows(M, 48), f"{M}x{N}x{K}")


def test_bf16_linear_strided_input():
    # the value columns of a QKV output feed the out-projection: a column
    # window of a wider matrix, rows 3 K apart
    M, K, N = 256, 1024, 512
    wide = synthetic.act_normal(5, M, 3 * K)
    (w,) = synthetic.weights(6, [(N, K)], 0.02)
    wide_dev = to_dev(wide)
    y = qlin.qlin_gemm_bf16(wide_dev[:, 2 * K:], to_dev(w))
    assert qlin.qlin_sync_status() == 0
    _check(np.ascontiguousarray(wide[:, 2 * K:]), w, y, sample_rows(M, 32), "strided")


# fp16 output: rounding 2^-11 of |y| <= |a||w| plus accumulation rounding
FP16_TOL = 1e-3


def _to_f16(bits):
    """The seeded bf16 values rounded to fp16 (both sides take these)."""
    return _f64(bits).astype(np.float16)


def _check16(a16, w16, y, rows, label):
    yref, na, nw = oracle.gemm_f64(a16[rows].astype(np.float64), w16.astype(np.float64))
    yg = y.cpu().numpy()[rows]
    denom = np.outer(na, nw)
    denom[denom == 0] = 1.0
    err = np.abs(yg.astype(np.float64) - yref) / denom
    assert err.max() <= FP16_TOL, (label, err.max())
    exact = np.mean(yg == yref.astype(np.float16))
    assert exact >= 0.95, (label, exact)


@pytest.mark.parametrize("M,N,K", [(1, 64, 64), (130, 320, 192), (333, 512, 1088), (4608, 3072, 3072)])
def test_fp16_linear(M, N, K):
    a16 = _to_f16(synthetic.act_entry_outliers(M + 2 * N + K, M, K))
    (w,) = synthetic.weights(N + K, [(N, K)], 0.02)
    w16 = _to_f16(w)
    y = qlin.qlin_gemm_fp16(torch.from_numpy(a16).cuda(), torch.from_numpy(w16).cuda())
    assert qlin.qlin_sync_status() == 0
    assert y.dtype == torch.float16
    _check16(a16, w16, y, sample_rows(M, 48), f"fp16 {M}x{N}x{K}")


def test_fp16_linear_strided_input_and_same_as_bf16_on_exact_values():
    # strided rows as for bf16; and on inputs exact in both formats with an
    # exactly representable product (small integers), both linears agree
    M, K, N = 256, 1024, 512
    wide16 = _to_f16(synthetic.act_normal(5, M, 3 * K))
    (w,) = synthetic.weights(6, [(N, K)], 0.02)
    w16 = _to_f16(w)
    y = qlin.qlin_gemm_fp16(torch.from_numpy(wide16).cuda()[:, 2 * K:], torch.from_numpy(w16).cuda())
    assert qlin.qlin_sync_status() == 0
    _check16(np.ascontiguousarray(wide16[:, 2 * K:]), w16, y, sample_rows(M, 32), "fp16 strided")

    rng = np.random.default_rng(8)
    ai = rng.integers(-1, 2, size=(192, 64)).astype(np.float32)
    wi = rng.integers(-2, 3, size=(128, 64)).astype(np.float32)
    y16 = qlin.qlin_gemm_fp16(torch.from_numpy(ai).half().cuda(), torch.from_numpy(wi).half().cuda())
    yb = qlin.qlin_gemm_bf16(torch.from_numpy(ai).bfloat16().cuda(), torch.from_numpy(wi).bfloat16().cuda())
    assert qlin.qlin_sync_status() == 0
    exact = ai.astype(np.float64) @ wi.astype(np.float64).T        # |y| <= 128: exact in both
    assert np.array_equal(y16.float().cpu().numpy(), exact)
    assert np.array_equal(yb.float().cpu().numpy(), exact)
