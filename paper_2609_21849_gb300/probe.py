"""Tensor-core rate probe (include/qlin_probe.h): the measured ceiling of the
tcgen05 MMA forms the GEMMs issue, for the roofline fractions.

  python -m paper_2609_21849_gb300.probe

Each case runs back-to-back MMAs of one kind and shape from one thread per
CTA (or CTA pair) on every SM at once; the result is FLOP per SM cycle
(clock-independent), the SM clock the probe ran at (cycles / nanoseconds)
and the rate in TFLOP/s there and at the maximum SM clock.
"""
from __future__ import annotations

import ctypes
import json
import os

import torch

from . import build

_lib = None

# (name, kind, pair, n, K per instruction); kind + 100: A read from TMEM
CASES = (("nvfp4_pair_256x256x64", 4, 1, 256, 64),
         ("nvfp4_cta_128x256x64", 4, 0, 256, 64),
         ("nvfp4_cta_128x128x64", 4, 0, 128, 64),
         ("fp8_pair_256x256x32", 8, 1, 256, 32),
         ("fp8_cta_128x256x32", 8, 0, 256, 32),
         ("bf16_pair_256x256x16", 16, 1, 256, 16),
         ("nvfp4_pair_256x256x64_a_tmem", 104, 1, 256, 64),
         ("nvfp4_cta_128x256x64_a_tmem", 104, 0, 256, 64),
         ("nvfp4_cta_128x128x64_a_tmem", 104, 0, 128, 64),
         ("fp8_pair_256x256x32_a_tmem", 108, 1, 256, 32),
         ("bf16_pair_256x256x16_a_tmem", 116, 1, 256, 16))


def _load():
    global _lib
    if _lib is None:
        build.build()
        lib = ctypes.CDLL(build.PROBE_LIB)
        lib.qlin_probe_mma.restype = ctypes.c_int
        lib.qlin_probe_mma.argtypes = [ctypes.c_int] * 5 + [ctypes.c_void_p] * 3
        _lib = lib
    return _lib


def measure(kind: int, pair: int, n: int, k: int, iters: int = 16384, sm_max_mhz: float = 2070.0):
    """One probe case on every SM; returns its rates."""
    lib = _load()
    sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    ctas = sms // 2 * 2 if pair else sms
    out = torch.zeros(2 * ctas, dtype=torch.int64, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    for it in (256, iters):   # a short warm-up launch, then the measured one
        st = lib.qlin_probe_mma(kind, pair, n, ctas, it, out.data_ptr(), err.data_ptr(), s)
        if st != 0:
            raise RuntimeError(f"qlin_probe_mma({kind}, {pair}, {n}) returned {st}")
    torch.cuda.synchronize()
    if int(err.item()) != 0:
        raise RuntimeError("probe wait expired")
    issuers = ctas // 2 if pair else ctas
    v = out.view(-1, 2)[:issuers].cpu().double()
    cyc, ns = v[:, 0].mean().item(), v[:, 1].mean().item()
    m = 256 if pair else 128
    flop_per_sm = 2.0 * m * n * k * iters / (2 if pair else 1)
    fpc = flop_per_sm / cyc
    mhz = cyc / ns * 1e3
    return {"flop_per_cycle_per_sm": round(fpc, 1), "cycles_per_mma": round(cyc / iters, 2),
            "sm_mhz": round(mhz, 1), "sms": sms,
            "tflops_at_probe_clock": round(fpc * sms * mhz * 1e6 / 1e12, 1),
            "tflops_at_max_clock": round(fpc * sms * sm_max_mhz * 1e6 / 1e12, 1)}


def ceilings(sm_max_mhz: float = 2070.0) -> dict:
    return {name: measure(kind, pair, n, k, sm_max_mhz=sm_max_mhz)
            for (name, kind, pair, n, k) in CASES}


if __name__ == "__main__":
    print(json.dumps(ceilings(), indent=1))
