"""GPU parity of the FP8 linear with the re-quantizing epilogue (the next
layer's FP8 input written by the GEMM, static post-training scale, Sec. 4):
the codes must equal the oracle's FP8 quantization of the same bf16 output,
bit for bit."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2609_21849_gb300 import qlin, synthetic

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from gpu_util import bf16_bits, to_dev, u8


@pytest.mark.parametrize("M,N,K,col0,cols", [(128, 256, 256, 0, 256), (333, 512, 1088, 128, 256),
                                             (4608, 3072, 3072, 0, 3072)])
def test_fp8_fused_requant(M, N, K, col0, cols):
    x = synthetic.act_channel_gain(M + N, M, K)
    (w,) = synthetic.weights(N + 7, [(N, K)], 0.02)
    A = qlin.qlin_quantize_act_fp8(to_dev(x))
    W = qlin.qlin_quantize_weight(to_dev(w), qlin.QLIN_FMT_FP8)
    y0 = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    qlin.qlin_gemm_fp8(A, W, y0)
    assert qlin.qlin_sync_status() == 0
    yb0 = bf16_bits(y0)
    # static next-layer scale: calibrated (by the oracle) on this output window
    s_next = oracle.fp8_tensor_scale(oracle.amax_bf16(np.ascontiguousarray(yb0[:, col0:col0 + cols])))
    nxt = torch.tensor([np.float32(s_next)], device="cuda")
    y = torch.empty_like(y0)
    yq = qlin.alloc_fp8(M, cols, False)
    qlin.qlin_linear_fused_fp8(A, W, y, nxt, yq, col0)
    assert qlin.qlin_sync_status() == 0
    assert torch.equal(y.view(torch.int16), y0.view(torch.int16))
    rc, rs = oracle.quant_fp8(np.ascontiguousarray(yb0[:, col0:col0 + cols]), s_next)
    assert np.float32(yq.scale.cpu()[0]) == np.float32(s_next)
    assert np.array_equal(u8(yq.codes), rc)
    # only the quantized output
    yq2 = qlin.alloc_fp8(M, cols, False)
    qlin.qlin_linear_fused_fp8(A, W, None, nxt, yq2, col0)
    assert qlin.qlin_sync_status() == 0
    assert np.array_equal(u8(yq2.codes), rc)
