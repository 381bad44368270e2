"""The no-allocation entry point, qlin_quantize_act_nvfp4_noalloc.

Some callers cannot allocate device memory: a plugin inside an inference
runtime that owns every device allocation, or a real-time loop that must not
stall on cudaMalloc.  This entry point quantizes with the dynamic tensor scale
like qlin_quantize_act_nvfp4, but keeps its amax scratch in the library's own
static device array instead of a caller workspace.  Here it must reproduce the
workspace entry point's codes, scales and tensor scale exactly, on two calls in
a row (the second with a smaller amax, so stale scratch would show), and, on an
input too large for the one-read route, the oracle's.

This file is collected last on purpose; it passes alone in a fresh process and
after the other tests.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2609_21849_gb300 import qlin, synthetic

pytestmark = pytest.mark.gpu


def _dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def _same(a: qlin.NVFP4Tensor, b: qlin.NVFP4Tensor):
    torch.cuda.synchronize()
    assert torch.equal(a.codes, b.codes)
    assert torch.equal(a.scales, b.scales)
    assert torch.equal(a.tensor_scale.view(torch.int32), b.tensor_scale.view(torch.int32))


def test_noalloc_matches_workspace_entry_point_twice():
    M, K = 333, 1088
    x1 = synthetic.act_entry_outliers(21, M, K)            # outliers: larger amax
    x2 = synthetic.act_normal(22, M, K)                     # smaller amax
    for bits in (x1, x2):
        x = _dev(bits)
        ref = qlin.qlin_quantize_act_nvfp4(x, None, qlin.alloc_nvfp4(M, K),
                                           qlin.alloc_workspace())
        out = qlin.qlin_quantize_act_nvfp4_noalloc(x, qlin.alloc_nvfp4(M, K))
        assert qlin.qlin_sync_status() == 0
        _same(out, ref)


def test_noalloc_full_size_activation():
    x = _dev(synthetic.act_entry_outliers(2, synthetic.M_TOKENS, synthetic.HIDDEN))
    ref = qlin.qlin_quantize_act_nvfp4(x)
    a = qlin.qlin_quantize_act_nvfp4_noalloc(x, qlin.alloc_nvfp4(*x.shape))
    b = qlin.qlin_quantize_act_nvfp4_noalloc(x, qlin.alloc_nvfp4(*x.shape))
    assert qlin.qlin_sync_status() == 0
    _same(a, ref)
    _same(b, ref)


def test_noalloc_two_pass_route_matches_oracle_twice():
    # x [9216, 4096] (75 MB) does not fit in the grid's shared memory, so the
    # entry point takes its two-pass route (an amax pass into the static
    # scratch, then the quantizer).  Two calls in a row, the second with a
    # smaller amax: a stale amax left in the scratch would change its scale.
    M, K = 9216, 4096
    for bits in (synthetic.act_entry_outliers(31, M, K), synthetic.act_normal(32, M, K)):
        out = qlin.qlin_quantize_act_nvfp4_noalloc(_dev(bits), qlin.alloc_nvfp4(M, K))
        assert qlin.qlin_sync_status() == 0
        rc, rs, sd = oracle.quant_nvfp4(bits)
        assert np.float32(out.tensor_scale.item()).view(np.uint32) == np.float32(sd).view(np.uint32)
        assert np.array_equal(out.codes.cpu().numpy(), rc)
        canon = oracle.unswizzle_scales(out.scales.cpu().numpy(), M, K)
        assert np.array_equal(canon, rs)


def test_noalloc_rejects_bad_arguments():
    out = qlin.alloc_nvfp4(64, 128)
    with pytest.raises(qlin.QlinError) as e:
        qlin.qlin_quantize_act_nvfp4_noalloc(_dev(np.zeros((64, 96), np.uint16)), out)
    assert e.value.status == 1                              # K not a multiple of 64
    assert qlin.qlin_workspace_size(1 << 20, 1 << 14) <= 256   # every shape fits the scratch
