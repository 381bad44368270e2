"""GPU parity of the unquantized bf16 linear (the BF16 row of Table 2's
precision ladder) on the tensor-core skeleton: y = a w^T against the exact
fp64 product of the same bf16 inputs."""
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
