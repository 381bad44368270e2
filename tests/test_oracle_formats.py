"""Pins of the oracle's element formats (e2m1, E4M3) against the format
definitions and an independent library (ml_dtypes).

Sec. 4 ("Quantization") quantizes to FP8 and NVFP4; E4M3 follows
Micikevicius et al. 2022 and the e2m1 / E4M3-scale format follows NVIDIA's
NVFP4 description, both cited there.
"""
import math

import numpy as np
import pytest

from conftest import read_golden

ml_dtypes = pytest.importorskip("ml_dtypes")


def test_e2m1_table_matches_golden(oracle):
    for line in read_golden("e2m1_grid.txt"):
        code, val = line.split()
        code, val = int(code, 16), float(val)
        got = oracle.e2m1_decode(code)
        assert got == val and math.copysign(1, got) == math.copysign(1, val), (code, got, val)


def test_e2m1_exhaustive_round_trip(oracle):
    for code in range(16):
        assert oracle.e2m1_encode(oracle.e2m1_decode(code)) == code


def test_e2m1_matches_ml_dtypes_dense_sweep(oracle):
    # every multiple of 1/64 in [-8, 8] plus random fp32 values
    vals = np.concatenate([np.arange(-512, 513) / 64.0,
                           np.random.default_rng(7).uniform(-9, 9, 4000)]).astype(np.float32)
    ref = vals.astype(ml_dtypes.float4_e2m1fn).view(np.uint8) & 0xF
    got = np.array([oracle.e2m1_encode(float(v)) for v in vals])
    bad = np.nonzero(got != ref)[0]
    assert bad.size == 0, [(float(vals[i]), int(got[i]), int(ref[i])) for i in bad[:10]]


def test_e2m1_ties_and_saturation(oracle):
    # round to nearest, ties to the even code; saturation at 6
    cases = {0.25: 0, 0.75: 2, 1.25: 2, 1.75: 4, 2.5: 4, 3.5: 6, 5.0: 6,
             6.5: 7, 7.0: 7, 100.0: 7, -0.0: 8, -5.0: 0xE, -1e9: 0xF}
    for v, c in cases.items():
        assert oracle.e2m1_encode(v) == c, (v, oracle.e2m1_encode(v), c)


def test_e4m3_points_match_golden(oracle):
    for line in read_golden("e4m3_points.txt"):
        code, val = line.split()
        code = int(code, 16)
        got = oracle.e4m3_decode(code)
        if val == "nan":
            assert math.isnan(got)
        else:
            val = float(val)
            assert got == val and math.copysign(1, got) == math.copysign(1, val)


def test_e4m3_exhaustive_round_trip(oracle):
    for code in range(256):
        v = oracle.e4m3_decode(code)
        if math.isnan(v):
            assert code in (0x7F, 0xFF)
            assert oracle.e4m3_encode(v) & 0x7F == 0x7F
        else:
            assert oracle.e4m3_encode(v) == code, hex(code)


def test_e4m3_decode_matches_ml_dtypes(oracle):
    ref = np.arange(256, dtype=np.uint8).view(ml_dtypes.float8_e4m3fn).astype(np.float64)
    for code in range(256):
        got = oracle.e4m3_decode(code)
        if math.isnan(ref[code]):
            assert math.isnan(got)
        else:
            assert got == ref[code], hex(code)


def test_e4m3_matches_ml_dtypes_in_range(oracle):
    # ml_dtypes rounds to nearest even inside the finite range; above 448 it
    # returns NaN where a saturating encoder returns 448, so compare in range.
    rng = np.random.default_rng(11)
    grid = np.arange(0, 127, dtype=np.uint8).view(ml_dtypes.float8_e4m3fn).astype(np.float64)
    mids = (grid[:-1] + grid[1:]) / 2             # every tie point
    vals = np.concatenate([grid, mids, -mids,
                           rng.uniform(-448, 448, 3000),
                           rng.uniform(-1, 1, 3000) * 2.0 ** rng.integers(-12, 0, 3000)])
    vals = vals[np.abs(vals) <= 448].astype(np.float32)
    ref = vals.astype(ml_dtypes.float8_e4m3fn).view(np.uint8)
    got = np.array([oracle.e4m3_encode(float(v)) for v in vals], dtype=np.uint8)
    bad = np.nonzero(got != ref)[0]
    assert bad.size == 0, [(float(vals[i]), hex(got[i]), hex(ref[i])) for i in bad[:10]]


def test_e4m3_golden_encode_cases(oracle):
    for line in read_golden("fp8_encode_cases.txt"):
        f = line.split()
        v, code = float(f[0]), int(f[1], 16)
        assert oracle.e4m3_encode(v) == code, (v, hex(oracle.e4m3_encode(v)), hex(code))


def test_e4m3_brute_force_nearest(oracle):
    # independent restatement: nearest finite grid value, ties -> even code
    grid = [(c, oracle.e4m3_decode(c)) for c in range(0x7F)]
    rng = np.random.default_rng(3)
    for v in np.concatenate([rng.uniform(0, 460, 500), rng.uniform(0, 0.02, 500)]):
        v = float(np.float32(v))
        best = min(grid, key=lambda cv: (abs(cv[1] - v), cv[0] & 1))
        if v >= 448:
            best = (0x7E, 448.0)
        assert oracle.e4m3_encode(v) == best[0], (v, best)


def test_bf16_widening(oracle):
    for bits, val in [(0x3F80, 1.0), (0xC000, -2.0), (0x0000, 0.0), (0x7F7F, 3.3895313892515355e38),
                      (0x0001, 9.183549615799121e-41)]:
        assert oracle.bf16_to_f32(bits) == np.float32(val)


def test_round_bf16_matches_fp32_rounding(oracle):
    # On fp32-representable values the direct fp64 -> bf16 rounding must agree
    # with the generator's independent fp32 -> bf16 rounding.
    from paper_2609_21849_gb300 import synthetic
    rng = np.random.default_rng(5)
    v = np.concatenate([rng.standard_normal(4000) * 10.0 ** rng.integers(-30, 30, 4000),
                        [1e-40, -3e-39, 0.0, -0.0]]).astype(np.float32)
    got = oracle.round_bf16_array(v.astype(np.float64))
    assert np.array_equal(got, synthetic.bf16_bits(v))


def test_round_bf16_ties_and_single_rounding(oracle):
    assert oracle.round_bf16(1.0 + 2.0 ** -8) == 0x3F80            # tie -> even
    assert oracle.round_bf16(1.0 + 3 * 2.0 ** -8) == 0x3F82        # tie -> even (up)
    # just above a tie: a double rounding through fp32 would land on the tie
    # and go to even; rounding once from fp64 goes up
    assert oracle.round_bf16(1.0 + 2.0 ** -8 + 2.0 ** -40) == 0x3F81
    assert oracle.round_bf16(-2.0) == 0xC000
