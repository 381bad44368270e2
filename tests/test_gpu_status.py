"""Device-side failure reporting without faulting the GPU: a bounded wait that
nothing completes expires, the kernel records a timeout and returns, the host
reads QLIN_ERR_TIMEOUT, and the context stays usable.  Also host-side
rejection of misaligned device pointers."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2609_21849_gb300 import qlin, synthetic

pytestmark = pytest.mark.gpu


def test_bounded_wait_expires_and_reports_timeout():
    assert qlin.qlin_sync_status() == 0
    qlin.qlin_selftest_bounded_wait(2_000_000)          # 2 ms limit
    assert qlin.qlin_sync_status() == 5                 # QLIN_ERR_TIMEOUT
    assert qlin.qlin_sync_status() == 0                 # cleared
    # the context is still usable
    x = torch.from_numpy(synthetic.act_normal(0, 128, 256).view(np.int16)).cuda().view(torch.bfloat16)
    q = qlin.qlin_quantize_act_nvfp4(x)
    w = qlin.qlin_quantize_weight(x, qlin.QLIN_FMT_NVFP4)
    y = qlin.qlin_gemm_nvfp4(q, w)
    assert qlin.qlin_sync_status() == 0
    assert torch.isfinite(y.float()).all()


def test_misaligned_device_pointers_are_rejected():
    buf = torch.zeros(128 * 64 * 2 + 64, dtype=torch.uint8, device="cuda")
    x = buf[2:2 + 128 * 64 * 2].view(torch.bfloat16).view(128, 64)  # 2-byte offset
    with pytest.raises(qlin.QlinError) as e:
        qlin.qlin_quantize_act_nvfp4(x)
    assert e.value.status == 3


def test_wait_timeout_setting_round_trip():
    qlin.qlin_set_wait_timeout_ns(500_000_000)
    x = torch.from_numpy(synthetic.act_normal(1, 256, 512).view(np.int16)).cuda().view(torch.bfloat16)
    q = qlin.qlin_quantize_act_nvfp4(x)
    y = qlin.qlin_gemm_nvfp4(q, qlin.qlin_quantize_weight(x, qlin.QLIN_FMT_NVFP4))
    assert qlin.qlin_sync_status() == 0
    qlin.qlin_set_wait_timeout_ns(2_000_000_000)
    assert y.shape == (256, 256)
