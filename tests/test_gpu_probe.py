"""The measurement probes of libqlin_probe.so run to completion on the GPU and
return rates inside the ranges the hardware allows: the MMA probe (the
roofline ceilings), the block-scale copy issue probe and the shared-memory
fill probe (the rates behind the GEMM's copy warps and row boxes)."""
import pytest

torch = pytest.importorskip("torch")

from paper_2609_21849_gb300 import probe

pytestmark = pytest.mark.gpu


def test_mma_probe_nvfp4_pair():
    r = probe.measure(4, 1, 256, 64, iters=2048)
    # one N = 256 NVFP4 pair MMA per 128 cycles at most (2 * 256 * 256 * 64 / 2 SMs)
    assert 0 < r["flop_per_cycle_per_sm"] <= 32768 * 1.01
    assert r["cycles_per_mma"] >= 127.0


def test_scale_copy_probe():
    alone = probe.scale_copy_cycles(4, 12, 0, iters=200)
    beside = probe.scale_copy_cycles(4, 12, 4, iters=200)
    mma_only = probe.scale_copy_cycles(1, 0, 4, iters=200)
    assert alone["copy_cycles_per_iter"] > 0 and beside["copy_cycles_per_iter"] > 0
    # four MMAs of N = 256 take at least 4 x 128 cycles
    assert mma_only["mma_cycles_per_iter"] >= 4 * 127.0
    assert beside["mma_cycles_per_iter"] >= 4 * 127.0
    # copies from four warps are no slower than from one
    one = probe.scale_copy_cycles(1, 12, 0, iters=200)
    assert alone["copy_cycles_per_iter"] <= one["copy_cycles_per_iter"]


@pytest.mark.parametrize("mode", [0, 1])
def test_fill_probe(mode):
    one = probe.fill_bytes_per_cycle(mode, 1, 2, iters=200)
    four = probe.fill_bytes_per_cycle(mode, 4, 2, iters=200)
    # a 16 KB copy cannot land in fewer cycles than shared memory's width allows
    for r in (one, four):
        assert 0 < r["bytes_per_cycle_per_sm"] < 256
    assert four["bytes_per_cycle_per_sm"] >= one["bytes_per_cycle_per_sm"]
