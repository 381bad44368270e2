"""GPU parity of the dynamic-scale chain qlin_linear_dynamic (Sec. 4,
"Quantization": run-time activation quantization, here with the next layer's
input scale taken from the layer's own output): the GEMM epilogue reduces
amax(|y|), and the NVFP4 quantization of y with that scale must equal the
oracle's dynamic quantization of the same bf16 y, bit for bit."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2609_21849_gb300 import qlin, synthetic

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from gpu_util import GEMM_TOL, assert_nvfp4_equal, bf16_bits, gemm_errors, sample_rows, to_dev


def _chain(x, w, label, rows=None):
    M, N = x.shape[0], w.shape[0]
    A = qlin.qlin_quantize_act_nvfp4(to_dev(x))
    W = qlin.qlin_quantize_weight(to_dev(w), qlin.QLIN_FMT_NVFP4)
    y, yq = qlin.qlin_linear_dynamic(A, W)
    assert qlin.qlin_sync_status() == 0
    # y is the plain GEMM's output, bit for bit
    y0 = torch.empty_like(y)
    qlin.qlin_gemm_nvfp4(A, W, y0)
    assert torch.equal(y.view(torch.int16), y0.view(torch.int16)), label
    yb = bf16_bits(y)
    # ... and within the GEMM tolerance of the oracle on sampled rows
    rows = sample_rows(M, 64) if rows is None else rows
    yref, na, nw = oracle.gemm_nvfp4(oracle.quant_nvfp4(x), oracle.quant_nvfp4(w), rows_sel=rows)
    err, _ = gemm_errors(yb[rows], yref, na, nw)
    assert err.max() <= GEMM_TOL, (label, err.max())
    # the quantized output: the oracle's dynamic quantization of this bf16 y
    assert_nvfp4_equal(yq, oracle.quant_nvfp4(yb), label + " y_q")
    return yq


@pytest.mark.parametrize("M,N,K", [(128, 256, 256), (130, 320, 192), (333, 512, 1088)])
def test_dynamic_chain_ragged(M, N, K):
    x = synthetic.act_entry_outliers(M + N + K, M, K)
    (w,) = synthetic.weights(N + 1, [(N, K)], 0.02)
    _chain(x, w, f"{M}x{N}x{K}")


def test_dynamic_chain_mlp_up_full_size():
    xb, wb = synthetic.nvfp4_mlp_up()
    _chain(xb, wb, "4608x12288x3072")


def test_dynamic_chain_zero_output_takes_unit_scale():
    M, N, K = 128, 256, 128
    x = np.zeros((M, K), np.uint16)
    (w,) = synthetic.weights(3, [(N, K)], 0.02)
    yq = _chain(x, w, "zero x", rows=np.arange(8))
    assert float(yq.tensor_scale.cpu()[0]) == 1.0


def test_dynamic_chain_repeated_calls_reset_the_amax():
    # a smaller output after a larger one must not inherit the larger amax
    M, N, K = 256, 512, 256
    (w,) = synthetic.weights(4, [(N, K)], 0.02)
    W = qlin.qlin_quantize_weight(to_dev(w), qlin.QLIN_FMT_NVFP4)
    ws = qlin.alloc_workspace()
    for seed, gain in ((8, 16.0), (9, 1.0)):
        x = synthetic.act_normal(seed, M, K)
        xf = (x.astype(np.uint32) << 16).view(np.float32) * np.float32(gain)
        A = qlin.qlin_quantize_act_nvfp4(to_dev(synthetic.bf16_bits(xf)))
        y, yq = qlin.qlin_linear_dynamic(A, W, workspace=ws)
        assert qlin.qlin_sync_status() == 0
        assert_nvfp4_equal(yq, oracle.quant_nvfp4(bf16_bits(y)), f"gain {gain}")
