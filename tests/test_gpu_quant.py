"""GPU parity of the quantizers (Sec. 4, "Quantization": run-time FP8 / NVFP4
activation quantization and offline weight quantization): codes, block scales
and tensor scales must equal the CPU oracle's bit for bit."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2609_21849_gb300 import qlin, synthetic

from conftest import read_golden

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from gpu_util import assert_nvfp4_equal, f32, nvfp4_to_host, to_dev, u8


RAGGED = [(1, 64), (3, 128), (130, 192), (257, 320), (128, 4096), (333, 1088)]


@pytest.mark.parametrize("M,K", RAGGED)
@pytest.mark.parametrize("dynamic", [True, False])
def test_nvfp4_act_ragged(M, K, dynamic):
    x = synthetic.act_entry_outliers(M * 7 + K, M, K)
    s_dec = None if dynamic else 0.0123
    ref = oracle.quant_nvfp4(x, s_dec)
    static = None if dynamic else torch.tensor([np.float32(s_dec)], device="cuda")
    q = qlin.qlin_quantize_act_nvfp4(to_dev(x), static_scale=static)
    assert qlin.qlin_sync_status() == 0
    assert_nvfp4_equal(q, ref, f"[{M},{K}] dynamic={dynamic}")


def test_nvfp4_tiny_workload():
    x, w = synthetic.tiny_nvfp4()
    q = qlin.qlin_quantize_act_nvfp4(to_dev(x))
    assert_nvfp4_equal(q, oracle.quant_nvfp4(x), "tiny x")
    qw = qlin.qlin_quantize_weight(to_dev(w), qlin.QLIN_FMT_NVFP4)
    assert_nvfp4_equal(qw, oracle.quant_nvfp4(w), "tiny W")


def test_nvfp4_act_full_size_mlp_up():
    # the 4608 x 3072 activation of the MLP up-projection, full tensor
    x = synthetic.act_entry_outliers(2, synthetic.M_TOKENS, synthetic.HIDDEN)
    ref = oracle.quant_nvfp4(x)
    q = qlin.qlin_quantize_act_nvfp4(to_dev(x))
    assert qlin.qlin_sync_status() == 0
    assert_nvfp4_equal(q, ref, "4608x3072 dynamic")
    # static mode with the calibrated scale gives the same result
    q2 = qlin.qlin_quantize_act_nvfp4(to_dev(x), static_scale=q.tensor_scale.clone())
    assert_nvfp4_equal(q2, ref, "4608x3072 static")


def test_nvfp4_weight_full_size():
    (w,) = synthetic.weights(2, [(synthetic.MLP, synthetic.HIDDEN)], 0.02)
    q = qlin.qlin_quantize_weight(to_dev(w), qlin.QLIN_FMT_NVFP4)
    assert_nvfp4_equal(q, oracle.quant_nvfp4(w), "W 12288x3072")


def test_nvfp4_hand_worked_blocks_on_gpu():
    # every golden block, placed in different rows / block positions
    lines = read_golden("nvfp4_blocks.txt")
    blocks = []
    for i in range(0, len(lines), 4):
        if float(lines[i].split()[3]) == 1.0:
            blocks.append([float(v) for v in lines[i + 1].split()[1:]])
    K = 64 * 2
    x = np.zeros((len(blocks) * 3, K), np.float32)
    for r in range(x.shape[0]):
        for b in range(K // 16):
            x[r, b * 16:(b + 1) * 16] = blocks[(r + b) % len(blocks)]
    bits = synthetic.bf16_bits(x)
    ref = oracle.quant_nvfp4(bits, 1.0)
    q = qlin.qlin_quantize_act_nvfp4(to_dev(bits), static_scale=torch.ones(1, device="cuda"))
    assert_nvfp4_equal(q, ref, "golden blocks")


def test_nvfp4_extreme_values():
    # zeros, signed zeros, subnormal bf16, huge values, and an all-zero tensor
    rng = np.random.default_rng(0)
    K = 256
    x = (rng.standard_normal((64, K)) * 10.0 ** rng.integers(-38, 38, (64, K))).astype(np.float32)
    x[0] = 0.0
    x[1] = -0.0
    x[2, ::3] = 1e-40
    x[3, :16] = 3e38
    bits = synthetic.bf16_bits(np.clip(np.nan_to_num(x, posinf=3e38, neginf=-3e38), -3e38, 3e38))
    for s in (None, 1.0, 1e-30, 1e30):
        ref = oracle.quant_nvfp4(bits, s)
        st = None if s is None else torch.tensor([np.float32(s)], device="cuda")
        q = qlin.qlin_quantize_act_nvfp4(to_dev(bits), static_scale=st)
        assert_nvfp4_equal(q, ref, f"extreme s={s}")
    z = np.zeros((5, 64), np.uint16)
    q = qlin.qlin_quantize_act_nvfp4(to_dev(z))
    assert_nvfp4_equal(q, oracle.quant_nvfp4(z), "all zero")


@pytest.mark.parametrize("M,K", RAGGED)
@pytest.mark.parametrize("dynamic", [True, False])
def test_fp8_act_ragged(M, K, dynamic):
    x = synthetic.act_channel_gain(M + K, M, K)
    s_dec = None if dynamic else 0.37
    rc, rs = oracle.quant_fp8(x, s_dec)
    static = None if dynamic else torch.tensor([np.float32(s_dec)], device="cuda")
    q = qlin.qlin_quantize_act_fp8(to_dev(x), static_scale=static)
    assert qlin.qlin_sync_status() == 0
    assert f32(q.scale)[0].view(np.uint32) == np.float32(rs).view(np.uint32)
    assert np.array_equal(u8(q.codes), rc)


def test_fp8_act_full_size():
    x = synthetic.act_channel_gain(1, synthetic.M_TOKENS, synthetic.HIDDEN)
    rc, rs = oracle.quant_fp8(x)
    q = qlin.qlin_quantize_act_fp8(to_dev(x))
    assert f32(q.scale)[0] == rs
    assert np.array_equal(u8(q.codes), rc)


@pytest.mark.parametrize("N,K", [(1, 64), (65, 192), (3072, 3072)])
def test_fp8_weight_per_channel(N, K):
    (w,) = synthetic.weights(N, [(N, K)], 0.02)
    w = w.copy()
    w[0] = 0  # an all-zero channel takes scale 1
    rc, rs = oracle.quant_fp8_rows(w)
    q = qlin.qlin_quantize_weight(to_dev(w), qlin.QLIN_FMT_FP8)
    assert np.array_equal(f32(q.scale).view(np.uint32), rs.view(np.uint32))
    assert np.array_equal(u8(q.codes), rc)


@pytest.mark.parametrize("fmt", ["nvfp4", "fp8"])
def test_dynamic_scale_x_larger_than_on_chip(fmt):
    # 9216 x 4096 bf16 (75.5 MB) exceeds what the grid can hold on chip, so
    # the dynamic scale takes the amax pass + quantizer route; the 4608 x 3072
    # cases above take the one-read route.  Both must equal the oracle.
    M, K = 9216, 4096
    x = synthetic.act_entry_outliers(77, M, K)
    if fmt == "nvfp4":
        q = qlin.qlin_quantize_act_nvfp4(to_dev(x))
        assert qlin.qlin_sync_status() == 0
        assert_nvfp4_equal(q, oracle.quant_nvfp4(x), "9216x4096 dynamic")
    else:
        rc, rs = oracle.quant_fp8(x)
        q = qlin.qlin_quantize_act_fp8(to_dev(x))
        assert qlin.qlin_sync_status() == 0
        assert f32(q.scale)[0].view(np.uint32) == np.float32(rs).view(np.uint32)
        assert np.array_equal(u8(q.codes), rc)


def test_dynamic_scale_two_pass_ragged_last_tile():
    # 9217 x 4096 takes the amax pass + quantizer route and ends in a partial
    # 16 KB tile (4 719 104 chunks of 16 bytes); the quantizer pass visits
    # its tiles last-first, so that partial tile is the first it copies.
    # Rows past the last 128-row atom are a ragged scale block as well.
    M, K = 9217, 4096
    assert (M * K // 8) % 1024 != 0
    x = synthetic.act_entry_outliers(78, M, K)
    q = qlin.qlin_quantize_act_nvfp4(to_dev(x))
    assert qlin.qlin_sync_status() == 0
    assert_nvfp4_equal(q, oracle.quant_nvfp4(x), "9217x4096 dynamic")


def test_dynamic_scale_one_read_repeated():
    # the one-read route keeps its grid-wide amax in two scratch words that
    # each launch clears: back-to-back calls on tensors of decreasing amax
    # must not see a stale maximum
    M, K = 4608, 3072
    ws = qlin.alloc_workspace()
    for seed, gain in ((5, 8.0), (6, 1.0), (7, 0.125)):
        x = (synthetic.act_normal(seed, M, K).view(np.uint16))
        xf = (x.astype(np.uint32) << 16).view(np.float32) * np.float32(gain)
        xb = synthetic.bf16_bits(xf)
        q = qlin.qlin_quantize_act_nvfp4(to_dev(xb), None, qlin.alloc_nvfp4(M, K), ws)
        assert qlin.qlin_sync_status() == 0
        assert_nvfp4_equal(q, oracle.quant_nvfp4(xb), f"gain {gain}")


def test_dynamic_scale_workspace_shared_by_both_routes():
    # one workspace serves the one-read route (words left zero after each
    # call) and the two-pass route (its own amax word, cleared before use):
    # alternate them and each must still equal the oracle
    ws = qlin.alloc_workspace()
    small = synthetic.act_entry_outliers(31, 512, 1024)     # fits on chip
    large = synthetic.act_normal(32, 9216, 4096)            # does not
    for x in (large, small, large, small):
        M, K = x.shape
        q = qlin.qlin_quantize_act_nvfp4(to_dev(x), None, qlin.alloc_nvfp4(M, K), ws)
        assert qlin.qlin_sync_status() == 0
        assert_nvfp4_equal(q, oracle.quant_nvfp4(x), f"{M}x{K}")
    assert int(ws[:12].sum()) == 0   # the one-read words are left zeroed
