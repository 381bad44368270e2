"""GPU parity of the NVFP4 linear with the fused re-quantizing epilogue (the
bf16 output is also quantized to NVFP4 for the next layer, with a static,
calibrated next-layer scale as in post-training quantization, Sec. 4).

The bf16 output is checked against the oracle's exact product within the GEMM
tolerance; the re-quantized codes and scales are checked bit-exactly, on every
block of the compared rows, against the oracle's NVFP4 quantization of the
layer's own bf16 output with the same static scale."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2609_21849_gb300 import qlin, synthetic

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from gpu_util import (GEMM_TOL, assert_nvfp4_equal, assert_requant_exact, bf16_bits,
                          gemm_errors, nvfp4_to_host, requant_agreement, stratified_rows, to_dev,
                          u8)


def _run(x, w, rows, rq_col0=0, rq_cols=None, label=""):
    M, N = x.shape[0], w.shape[0]
    rq_cols = N - rq_col0 if rq_cols is None else rq_cols
    aq, wq = oracle.quant_nvfp4(x), oracle.quant_nvfp4(w)
    yref, na, nw = oracle.gemm_nvfp4(aq, wq, rows_sel=rows)
    y16_ref = oracle.round_bf16_array(yref)
    win = slice(rq_col0, rq_col0 + rq_cols)
    # static next-layer scale, calibrated by the oracle on the sampled rows
    s_next = oracle.nvfp4_tensor_scale(oracle.amax_bf16(np.ascontiguousarray(y16_ref[:, win])))

    A = qlin.qlin_quantize_act_nvfp4(to_dev(x))
    W = qlin.qlin_quantize_weight(to_dev(w), qlin.QLIN_FMT_NVFP4)
    nxt = torch.tensor([np.float32(s_next)], device="cuda")
    y = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    yq = qlin.alloc_nvfp4(M, rq_cols)
    qlin.qlin_linear_fused(A, W, y, nxt, yq, rq_col0)
    assert qlin.qlin_sync_status() == 0
    assert_nvfp4_equal(A, aq, label + " A")
    assert_nvfp4_equal(W, wq, label + " W")

    yb = bf16_bits(y)
    err, exact = gemm_errors(yb[rows], yref, na, nw)
    assert err.max() <= GEMM_TOL, (label, err.max())
    assert exact >= 0.99, (label, exact)

    codes, canon, s = nvfp4_to_host(yq)
    assert s == np.float32(s_next)
    # bit-exact against the oracle's quantization of the GPU's own bf16 y
    assert_requant_exact(codes[rows], canon[rows], yb[rows][:, win], s_next, label)
    # and, as a statistic, against the oracle's quantization of its own bf16
    # rounding of the exact result (blocks with identical inputs must agree)
    agree = requant_agreement(codes[rows], canon[rows], yb[rows][:, win],
                              np.ascontiguousarray(y16_ref[:, win]), s_next)
    assert agree >= 0.99, (label, agree)

    # Re-quantization equals the standalone quantizer applied to the layer's
    # own bf16 output (both on the GPU), over every row.
    ystd = qlin.qlin_quantize_act_nvfp4(y[:, win].contiguous(), static_scale=nxt)
    assert np.array_equal(u8(ystd.codes), codes), label
    assert np.array_equal(u8(ystd.scales), u8(yq.scales)), label

    # Re-quantization only (no bf16 output) writes the same codes.
    yq2 = qlin.alloc_nvfp4(M, rq_cols)
    qlin.qlin_linear_fused(A, W, None, nxt, yq2, rq_col0)
    assert qlin.qlin_sync_status() == 0
    assert np.array_equal(u8(yq2.codes), codes) and np.array_equal(u8(yq2.scales), u8(yq.scales))
    return err.max(), exact, agree


def test_fused_tiny():
    x, w = synthetic.tiny_nvfp4()
    _run(x, w, np.arange(128), label="tiny")


def test_fused_mlp_up_full_size():
    # 4608 x 12288 x 3072 with the whole output re-quantized (the benchmark's
    # launch configuration), every row compared
    x, w = synthetic.nvfp4_mlp_up()
    e, ex, ag = _run(x, w, np.arange(x.shape[0]), label="mlp-up fused")
    print(f"mlp-up fused: err {e:.2e} exact {ex:.4f} requant agree {ag:.5f}")


def test_fused_qkv_value_window():
    # QKV projection (N = 9216) whose epilogue re-quantizes only the value
    # columns 6144..9215 for the out-projection
    x = synthetic.stack_input(1)
    (w,) = synthetic.weights(4, [(9216, 3072)], 0.02)
    _run(x, w, stratified_rows(x.shape[0], 64), rq_col0=6144, rq_cols=3072, label="qkv window")


@pytest.mark.parametrize("M,N,K,c0,cols", [(77, 320, 192, 64, 192), (1300, 3648, 320, 0, 3648),
                                           (513, 1024, 2560, 512, 512),
                                           # CTA pairs: partial last wave, row block and N block
                                           (4500, 12224, 1024, 0, 12224),
                                           # CTA pairs with a partial last K stage (one MMA step)
                                           (2048, 4096, 1088, 0, 4096)])
def test_fused_ragged(M, N, K, c0, cols):
    x = synthetic.act_entry_outliers(M * 3 + K, M, K)
    (w,) = synthetic.weights(M * 3 + K, [(N, K)], 0.02)
    _run(x, w, stratified_rows(M, 48, seed=1), rq_col0=c0, rq_cols=cols, label=f"{M}x{N}x{K}")
