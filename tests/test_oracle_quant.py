"""Pins of the oracle's quantizers and scale layout.

Sec. 4 ("Quantization"): activations and weights are quantized post-training
to NVFP4 (e2m1 codes, 16-element E4M3 block scales, FP32 tensor scale) or FP8
E4M3 with a per-tensor (activations) or per-output-channel (weights) scale.
"""
import numpy as np
import pytest

from conftest import read_golden
from paper_2609_21849_gb300 import synthetic

ml_dtypes = pytest.importorskip("ml_dtypes")


def _blocks():
    lines = read_golden("nvfp4_blocks.txt")
    out = []
    i = 0
    while i < len(lines):
        head = lines[i].split()
        assert head[0] == "block"
        name, s_dec = head[1], float(head[3])
        x = [float(v) for v in lines[i + 1].split()[1:]]
        scale = int(lines[i + 2].split()[1], 16)
        codes = [int(c, 16) for c in lines[i + 3].split()[1:]]
        assert len(x) == 16 and len(codes) == 16
        out.append((name, s_dec, x, scale, codes))
        i += 4
    return out


@pytest.mark.parametrize("case", _blocks(), ids=lambda c: c[0])
def test_nvfp4_hand_worked_blocks(oracle, case):
    name, s_dec, x, scale, codes = case
    bits = synthetic.bf16_bits(np.array([x], np.float32))
    assert np.array_equal(synthetic.bf16_to_f32(bits)[0], np.array(x, np.float32)), "fixture not bf16-exact"
    c, s, _ = oracle.quant_nvfp4(bits, s_dec)
    assert s[0, 0] == scale, (name, hex(s[0, 0]), hex(scale))
    got = [(c[0, j // 2] >> (4 * (j % 2))) & 0xF for j in range(16)]
    assert got == codes, (name, got, codes)


def test_nvfp4_packing_low_nibble_is_even_element(oracle):
    # element 0 = 6 (code 7), element 1 = 0.5 (code 1) with s_b = 1, S_dec = 1
    x = np.zeros((1, 16), np.float32)
    x[0, 0], x[0, 1] = 6.0, 0.5
    c, s, _ = oracle.quant_nvfp4(synthetic.bf16_bits(x), 1.0)
    assert c[0, 0] == 0x17 and s[0, 0] == 0x38


def test_tensor_scale_closed_forms(oracle):
    assert oracle.nvfp4_tensor_scale(2688.0) == 1.0
    assert oracle.nvfp4_tensor_scale(0.0) == 1.0
    assert oracle.fp8_tensor_scale(448.0) == 1.0
    assert oracle.fp8_tensor_scale(0.0) == 1.0
    assert oracle.nvfp4_tensor_scale(6.0) == np.float32(6.0) / np.float32(2688.0)
    assert oracle.encode_scale(0.5) == 2.0
    assert oracle.encode_scale(0.0) == np.finfo(np.float32).max
    assert oracle.encode_scale(1e-45) == np.finfo(np.float32).max


def test_block_holding_global_amax_scales_to_448(oracle):
    # With the dynamic tensor scale amax/2688, the block that holds the global
    # amax must get the largest E4M3 scale and its amax element code +-6.
    for seed in range(5):
        x = synthetic.act_entry_outliers(100 + seed, 64, 256)
        xf = synthetic.bf16_to_f32(x)
        c, s, s_dec = oracle.quant_nvfp4(x)
        assert s_dec == np.float32(np.abs(xf).max()) / np.float32(2688.0)
        r, k = np.unravel_index(np.argmax(np.abs(xf)), xf.shape)
        assert s[r, k // 16] == 0x7E
        code = (c[r, k // 2] >> (4 * (k % 2))) & 0xF
        assert code & 7 == 7 and (code >> 3) == (xf[r, k] < 0)
        assert s.max() == 0x7E  # no block scale exceeds the largest


def test_nvfp4_reconstruction_bound(oracle):
    # |x - xhat| <= half the local e2m1 grid step times the effective scale for
    # unsaturated elements, where the effective scale is s_b * S_dec.
    x = synthetic.act_entry_outliers(5, 96, 512)
    xf = synthetic.bf16_to_f32(x).astype(np.float64)
    c, s, s_dec = oracle.quant_nvfp4(x)
    deq = oracle.dequant_nvfp4(c, s, s_dec)
    scale = np.repeat(np.array([[oracle.e4m3_decode(v) for v in row] for row in s]), 16, axis=1)
    eff = scale * float(s_dec)
    grid = np.array([0, 0.5, 1, 1.5, 2, 3, 4, 6])
    step = np.diff(grid)                      # gap above each grid point
    u = np.abs(xf) / np.where(eff > 0, eff, 1)
    # local step: gap of the interval that contains |x|/eff
    idx = np.clip(np.searchsorted(grid, u, side="right") - 1, 0, 6)
    bound = 0.5 * step[idx] * eff
    ok = (u <= 6.0) & (eff > 0)
    err = np.abs(xf - deq)
    # fp32 rounding of x * r_b moves the point by ~1e-7 relative: allow it
    assert np.all(err[ok] <= bound[ok] * (1 + 1e-6) + 1e-30)
    # zero-scale blocks decode to zero
    assert np.all(deq[eff == 0] == 0)
    # saturated elements decode to the block's largest value
    sat = (u > 6.0) & (eff > 0)
    assert np.allclose(np.abs(deq[sat]), 6 * eff[sat])


def test_nvfp4_matches_ml_dtypes_elementwise_rounding(oracle):
    # Independent check of the element step: with S_dec = 1 and a block amax of
    # 6 the block scale is 1, so the codes are ml_dtypes' e2m1 rounding of x.
    rng = np.random.default_rng(9)
    x = rng.uniform(-6, 6, (64, 64)).astype(np.float32)
    x[:, ::16] = 6.0
    bits = synthetic.bf16_bits(x)
    xf = synthetic.bf16_to_f32(bits)
    c, s, _ = oracle.quant_nvfp4(bits, 1.0)
    assert np.all(s == 0x38)
    ref = xf.astype(ml_dtypes.float4_e2m1fn).view(np.uint8) & 0xF
    lo, hi = c & 0xF, c >> 4
    got = np.empty_like(ref)
    got[:, 0::2], got[:, 1::2] = lo, hi
    assert np.array_equal(got, ref)


def test_fp8_per_tensor_matches_ml_dtypes(oracle):
    x = synthetic.act_channel_gain(1, 64, 256)
    xf = synthetic.bf16_to_f32(x)
    c, s_dec = oracle.quant_fp8(x)
    assert s_dec == np.float32(np.abs(xf).max()) / np.float32(448.0)
    s_enc = oracle.encode_scale(float(s_dec))
    v = (xf * np.float32(s_enc)).astype(np.float32)     # one fp32 product
    v = np.clip(v, -448, 448)                           # saturating encoder
    ref = v.astype(ml_dtypes.float8_e4m3fn).view(np.uint8)
    assert np.array_equal(c, ref)
    # the element holding the amax maps to +-448 (code 0x7E / 0xFE)
    r, k = np.unravel_index(np.argmax(np.abs(xf)), xf.shape)
    assert c[r, k] & 0x7F == 0x7E


def test_fp8_per_channel_weights(oracle):
    (w,) = synthetic.weights(3, [(48, 128)], 0.02)
    wf = synthetic.bf16_to_f32(w)
    c, s = oracle.quant_fp8_rows(w)
    assert np.array_equal(s, (np.abs(wf).max(axis=1) / np.float32(448.0)).astype(np.float32))
    for n in range(48):
        k = np.argmax(np.abs(wf[n]))
        assert c[n, k] & 0x7F == 0x7E
    deq = oracle.dequant_fp8(c, s)
    assert np.max(np.abs(deq - wf) / s[:, None]) <= 16.0  # half an ulp at 448 is 16


def test_zero_rows_fp8(oracle):
    w = np.zeros((2, 64), np.uint16)
    c, s = oracle.quant_fp8_rows(w)
    assert np.all(c == 0) and np.all(s == 1.0)


def test_swizzle_offsets_golden(oracle):
    for line in read_golden("swizzle_offsets.txt"):
        r, c, K, off = map(int, line.split())
        assert oracle.swizzle_offset(r, c, K) == off, line


def test_swizzle_is_a_bijection_with_zero_padding(oracle):
    rows, K = 200, 256
    rng = np.random.default_rng(1)
    canon = rng.integers(1, 255, (rows, K // 16), dtype=np.uint8)
    swz = oracle.swizzle_scales(canon, K)
    assert swz.size == 2 * (K // 64) * 512
    assert np.array_equal(oracle.unswizzle_scales(swz, rows, K), canon)
    # every canonical entry lands on a distinct byte; the rest is padding (0)
    offs = {oracle.swizzle_offset(r, c, K) for r in range(rows) for c in range(K // 16)}
    assert len(offs) == rows * K // 16
    mask = np.ones(swz.size, bool)
    mask[list(offs)] = False
    assert np.all(swz[mask] == 0)


def test_amax(oracle):
    x = synthetic.act_entry_outliers(2, 32, 64)
    assert oracle.amax_bf16(x) == np.abs(synthetic.bf16_to_f32(x)).max()
