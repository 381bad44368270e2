"""GPU parity of the embedding translator's MLP forward (Sec. 3, Table 1: the
d3072 translator, a single 3072-wide MLP from the 0.6B encoder's 1024-wide
features to the 4B encoder's 2560-wide conditioning) on the small-M path: 512
tokens, x [512, 1024] -> hidden [512, 3072] -> y [512, 2560], NVFP4 (W4A4) and
FP8 (W8A8), the first linear's epilogue re-quantizing the hidden activations
with a static scale calibrated by the oracle.

Checked against the oracle on every token row:
- the input quantization and both weights, bit-exact;
- the hidden bf16 activations within the GEMM tolerance of the exact product;
- the re-quantized hidden activations, bit-exact against the oracle's
  quantization of the GPU's own hidden bf16 values;
- the output within the GEMM tolerance of the exact product of those
  re-quantized activations and W2."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2609_21849_gb300 import qlin, synthetic, translator

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from gpu_util import (GEMM_TOL, assert_nvfp4_equal, assert_requant_exact, bf16_bits, f32,
                          gemm_errors, nvfp4_to_host, to_dev, u8)


def _check_gemm(y_gpu_bits, yref, na, nw, label):
    err, exact = gemm_errors(y_gpu_bits, yref, na, nw)
    assert np.all(np.isfinite(err)), label
    assert err.max() <= GEMM_TOL, (label, err.max())
    assert exact >= 0.99, (label, exact)
    return err.max()


@pytest.mark.parametrize("fmt", ["nvfp4", "fp8"])
def test_translator_mlp_forward(fmt):
    x, w1, w2 = synthetic.translator_mlp()
    M = x.shape[0]
    if fmt == "nvfp4":
        xq, w1q, w2q = oracle.quant_nvfp4(x), oracle.quant_nvfp4(w1), oracle.quant_nvfp4(w2)
        h_ref, na, nw = oracle.gemm_nvfp4(xq, w1q)
        s_h = oracle.nvfp4_tensor_scale(oracle.amax_bf16(oracle.round_bf16_array(h_ref)))
    else:
        xq, w1q, w2q = oracle.quant_fp8(x), oracle.quant_fp8_rows(w1), oracle.quant_fp8_rows(w2)
        h_ref, na, nw = oracle.gemm_fp8(xq, w1q)
        s_h = oracle.fp8_tensor_scale(oracle.amax_bf16(oracle.round_bf16_array(h_ref)))

    t = translator.build_translator(fmt, w1, w2, M)
    t.set_hidden_scale(s_h)
    xd = to_dev(x)
    t.forward(xd, write_hidden=True)
    assert qlin.qlin_sync_status() == 0
    y1 = bf16_bits(t.y)

    if fmt == "nvfp4":
        assert_nvfp4_equal(t.x_q, xq, "x")
        assert_nvfp4_equal(t.W1, w1q, "W1")
        assert_nvfp4_equal(t.W2, w2q, "W2")
    else:
        assert np.array_equal(u8(t.x_q.codes), xq[0]) and f32(t.x_q.scale)[0] == xq[1]
        assert np.array_equal(u8(t.W1.codes), w1q[0]) and np.array_equal(f32(t.W1.scale), w1q[1])
        assert np.array_equal(u8(t.W2.codes), w2q[0]) and np.array_equal(f32(t.W2.scale), w2q[1])

    hb = bf16_bits(t.h)
    e1 = _check_gemm(hb, h_ref, na, nw, f"{fmt} hidden")
    if fmt == "nvfp4":
        codes, canon, s = nvfp4_to_host(t.h_q)
        assert s == np.float32(s_h)
        hq = assert_requant_exact(codes, canon, hb, s_h, "hidden re-quantization")
        yref, na2, nw2 = oracle.gemm_nvfp4(hq, w2q)
    else:
        hq = oracle.quant_fp8(hb, s_h)
        assert f32(t.h_q.scale)[0] == np.float32(s_h)
        assert np.array_equal(u8(t.h_q.codes), hq[0]), "hidden FP8 re-quantization"
        yref, na2, nw2 = oracle.gemm_fp8(hq, w2q)
    e2 = _check_gemm(y1, yref, na2, nw2, f"{fmt} output")

    # the forward without the hidden bf16 output, and as a CUDA graph replayed
    # twice, gives the same bits
    t.y.zero_()
    t.forward(xd)
    torch.cuda.synchronize()
    assert np.array_equal(bf16_bits(t.y), y1)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        t.forward(xd, s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        t.forward(xd, s)
    t.y.zero_()
    g.replay()
    g.replay()
    torch.cuda.synchronize()
    assert qlin.qlin_sync_status() == 0
    assert np.array_equal(bf16_bits(t.y), y1)
    print(f"translator {fmt}: hidden err {e1:.2e}, output err {e2:.2e}")
