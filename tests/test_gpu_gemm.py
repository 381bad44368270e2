"""GPU parity of the block-scaled GEMMs (Sec. 4: the quantized linears run on
the NVFP4 / FP8 tensor cores).  Operands are quantized on the GPU and checked
bit-exact against the oracle; the bf16 output is checked against the oracle's
exact fp64 result with |y - y_exact| / (||a_m|| ||w_n||) <= 2e-3, and at least
99% of the outputs must equal the correctly rounded bf16 of the exact result
(the kernels differ from it only by fp32 accumulation order)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2609_21849_gb300 import qlin, synthetic

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from gpu_util import (GEMM_TOL, assert_nvfp4_equal, bf16_bits, f32, gemm_errors,
                          sample_rows, stratified_rows, to_dev, u8)


def _check_nvfp4(x, w, rows=None, label=""):
    aq = oracle.quant_nvfp4(x)
    wq = oracle.quant_nvfp4(w)
    A = qlin.qlin_quantize_act_nvfp4(to_dev(x))
    W = qlin.qlin_quantize_weight(to_dev(w), qlin.QLIN_FMT_NVFP4)
    y = qlin.qlin_gemm_nvfp4(A, W)
    assert qlin.qlin_sync_status() == 0
    assert_nvfp4_equal(A, aq, label + " A")
    assert_nvfp4_equal(W, wq, label + " W")
    sel = np.arange(x.shape[0]) if rows is None else rows
    yref, na, nw = oracle.gemm_nvfp4(aq, wq, rows_sel=sel)
    yb = bf16_bits(y)[sel]
    err, exact = gemm_errors(yb, yref, na, nw)
    assert np.all(np.isfinite(err)), label
    assert err.max() <= GEMM_TOL, (label, err.max(), np.unravel_index(err.argmax(), err.shape))
    assert exact >= 0.99, (label, exact)
    return err.max(), exact


def _check_fp8(x, w, rows=None, label=""):
    ac, as_ = oracle.quant_fp8(x)
    wc, ws = oracle.quant_fp8_rows(w)
    A = qlin.qlin_quantize_act_fp8(to_dev(x))
    W = qlin.qlin_quantize_weight(to_dev(w), qlin.QLIN_FMT_FP8)
    y = qlin.qlin_gemm_fp8(A, W)
    assert qlin.qlin_sync_status() == 0
    assert np.array_equal(u8(A.codes), ac) and f32(A.scale)[0] == as_, label
    assert np.array_equal(u8(W.codes), wc) and np.array_equal(f32(W.scale), ws), label
    sel = np.arange(x.shape[0]) if rows is None else rows
    yref, na, nw = oracle.gemm_fp8((ac, as_), (wc, ws), rows_sel=sel)
    err, exact = gemm_errors(bf16_bits(y)[sel], yref, na, nw)
    assert np.all(np.isfinite(err)), label
    assert err.max() <= GEMM_TOL, (label, err.max())
    assert exact >= 0.99, (label, exact)
    return err.max(), exact


def test_nvfp4_tiny_all_outputs():
    x, w = synthetic.tiny_nvfp4()
    e, ex = _check_nvfp4(x, w, label="tiny")
    print(f"tiny nvfp4: max err {e:.3e}, exact {ex:.4f}")


# ragged shapes: partial M and N tiles, K not a multiple of a pipeline stage,
# both tile widths (128 x 128 when the 128 x 256 grid would not fill the GPU)
RAGGED = [(1, 64, 64), (77, 320, 192), (300, 128, 512), (129, 576, 1088),
          (1300, 3648, 320), (2048, 4096, 256),
          # CTA pairs (256 x 256 tiles fill the GPU) with a partial last K stage
          (2048, 4096, 1088)]


@pytest.mark.parametrize("M,N,K", RAGGED)
def test_nvfp4_ragged(M, N, K):
    x = synthetic.act_entry_outliers(M + N + K, M, K)
    (w,) = synthetic.weights(M + N + K, [(N, K)], 0.02)
    rows = stratified_rows(M, 48, seed=M) if M > 64 else None
    _check_nvfp4(x, w, rows, f"nvfp4 {M}x{N}x{K}")


@pytest.mark.parametrize("M,N,K", RAGGED)
def test_fp8_ragged(M, N, K):
    x = synthetic.act_channel_gain(M + N + K, M, K)
    (w,) = synthetic.weights(M + N + K, [(N, K)], 0.02)
    rows = stratified_rows(M, 48, seed=M) if M > 64 else None
    _check_fp8(x, w, rows, f"fp8 {M}x{N}x{K}")


def test_nvfp4_mlp_up_full_size():
    # 4608 x 12288 x 3072, in the launch configuration the benchmark times;
    # every output is compared with the oracle (every tile position and TMEM
    # lane quarter)
    x, w = synthetic.nvfp4_mlp_up()
    e, ex = _check_nvfp4(x, w, None, "mlp-up")
    print(f"mlp-up nvfp4: max err {e:.3e}, exact {ex:.4f}")


def test_fp8_linear_full_size():
    x, w = synthetic.fp8_linear()
    e, ex = _check_fp8(x, w, None, "fp8-linear")   # every output
    print(f"fp8 linear: max err {e:.3e}, exact {ex:.4f}")


@pytest.mark.parametrize("fmt", ["nvfp4", "fp8"])
def test_translator_small_m(fmt):
    x1, x2, w1, w2 = synthetic.translator()
    chk = _check_nvfp4 if fmt == "nvfp4" else _check_fp8
    chk(x1, w1, None, f"translator {fmt} 512x2560x1024")
    chk(x2, w2, None, f"translator {fmt} 512x1024x2560")


def test_nvfp4_dyadic_exact():
    # Values on the e2m1 grid, every block holding a 6, tensor scale 1: all
    # block scales are 1, the codes are the values themselves, every product
    # and partial sum is exact in fp32, so the bf16 output must equal the
    # correctly rounded exact result everywhere.
    rng = np.random.default_rng(0)
    M, N, K = 256, 512, 512
    vals = np.array([0, 0.5, 1, 1.5, 2, 3, 4, 6, -0.5, -1, -1.5, -2, -3, -4, -6], np.float32)
    x = rng.choice(vals, (M, K)).astype(np.float32)
    w = rng.choice(vals, (N, K)).astype(np.float32)
    x[:, ::16] = 6.0
    w[:, ::16] = -6.0
    xb, wb = synthetic.bf16_bits(x), synthetic.bf16_bits(w)
    one = torch.ones(1, device="cuda")
    aq = oracle.quant_nvfp4(xb, 1.0)
    wq = oracle.quant_nvfp4(wb, 1.0)
    assert np.all(aq[1] == 0x38) and np.all(wq[1] == 0x38)
    A = qlin.qlin_quantize_act_nvfp4(to_dev(xb), static_scale=one)
    W = qlin.qlin_quantize_act_nvfp4(to_dev(wb), static_scale=one)
    assert_nvfp4_equal(A, aq, "dyadic A")
    assert_nvfp4_equal(W, wq, "dyadic W")
    y = qlin.qlin_gemm_nvfp4(A, W)
    yref, na, nw = oracle.gemm_nvfp4(aq, wq)
    assert np.array_equal(yref, x.astype(np.float64) @ w.astype(np.float64).T)
    err, exact = gemm_errors(bf16_bits(y), yref, na, nw)
    assert exact == 1.0, exact


def test_fp8_output_alignment_16_and_32_bytes():
    # The pair-tile FP8 epilogue stores y straight from registers, with
    # 32-byte vectors when y is 32-byte aligned and 16-byte ones otherwise;
    # both must write the same bits (rows 1..M of a padded buffer check that
    # nothing lands outside y).
    x, w = synthetic.fp8_linear()
    A = qlin.qlin_quantize_act_fp8(to_dev(x))
    W = qlin.qlin_quantize_weight(to_dev(w), qlin.QLIN_FMT_FP8)
    M, N = A.rows, W.rows
    y32 = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    qlin.qlin_gemm_fp8(A, W, y32)
    pad = torch.full((M * N + 32,), -7.0, dtype=torch.bfloat16, device="cuda")
    y16 = pad[8:8 + M * N].view(M, N)              # 16 bytes past a 32-byte boundary
    assert y16.data_ptr() % 32 == 16
    qlin.qlin_gemm_fp8(A, W, y16)
    assert qlin.qlin_sync_status() == 0
    assert torch.equal(y16.view(torch.int16), y32.view(torch.int16))
    assert torch.all(pad[:8] == -7.0) and torch.all(pad[8 + M * N:] == -7.0)


def test_nvfp4_ragged_pair_tiles_partial_last_wave():
    # 4500 x 12224 on CTA pairs: 864 tiles of 256 x 256 over the persistent
    # clusters, a partial last wave, a partial last row block (20 rows) and a
    # last N block with 192 valid columns of 256.
    M, N, K = 4500, 12224, 1024
    x = synthetic.act_entry_outliers(77, M, K)
    (w,) = synthetic.weights(78, [(N, K)], 0.02)
    rows = np.unique(np.concatenate([stratified_rows(M, 64, seed=5), np.arange(M - 20, M)]))
    _check_nvfp4(x, w, rows, "pair tiles 4500x12224x1024")
