"""Tensor-core rate probe (include/qlin_probe.h): the measured ceiling of the
tcgen05 MMA forms the GEMMs issue, for the roofline fractions, and the issue
rates of the copies that feed them.

  python -m paper_2609_21849_gb300.probe            # MMA ceilings
  python -m paper_2609_21849_gb300.probe --copies   # block-scale copy and fill rates

Each MMA case runs back-to-back MMAs of one kind and shape from one thread per
CTA (or CTA pair) on every SM at once; the result is FLOP per SM cycle
(clock-independent), the SM clock the probe ran at (cycles / nanoseconds)
and the rate in TFLOP/s there and at the maximum SM clock.  The copy cases
give SM cycles per stage's worth of block-scale copies against the number of
issuing warps, and shared-memory fill bytes per cycle per SM against the
number of threads issuing copies.
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
        lib.qlin_probe_scale_copy.restype = ctypes.c_int
        lib.qlin_probe_scale_copy.argtypes = [ctypes.c_int] * 5 + [ctypes.c_void_p] * 3
        lib.qlin_probe_fill.restype = ctypes.c_int
        lib.qlin_probe_fill.argtypes = ([ctypes.c_int] * 5 + [ctypes.c_void_p, ctypes.c_ulonglong]
                                        + [ctypes.c_void_p] * 3)
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


def scale_copy_cycles(warps: int, copies: int = 12, mmas: int = 4, iters: int = 2000) -> dict:
    """SM cycles per iteration of `mmas` NVFP4 pair MMAs (N = 256) and, beside
    them, `copies` block-scale copies issued from `warps` warps (mmas = 0:
    the copies alone), every SM pair at once."""
    lib = _load()
    sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    ctas = sms // 2 * 2
    out = torch.zeros(ctas, dtype=torch.int64, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    for it in (64, iters):
        st = lib.qlin_probe_scale_copy(warps, copies, mmas, ctas, it, out.data_ptr(), err.data_ptr(), s)
        if st != 0:
            raise RuntimeError(f"qlin_probe_scale_copy({warps}, {copies}, {mmas}) returned {st}")
    torch.cuda.synchronize()
    if int(err.item()) != 0:
        raise RuntimeError("probe wait expired")
    v = out.view(-1, 2).cpu().double()
    mma = v[:, 0].median().item() / iters if mmas else None
    cp = v[:, 1].median().item() / iters if copies else None
    return {"warps": warps, "copies": copies, "mmas": mmas,
            "mma_cycles_per_iter": None if mma is None else round(mma, 1),
            "copy_cycles_per_iter": None if cp is None else round(cp, 1)}


def fill_bytes_per_cycle(mode: int, threads: int, depth: int, iters: int = 3000,
                         src_mb: int = 24) -> dict:
    """Shared-memory fill rate per SM (bytes per SM cycle), every SM at once,
    of `threads` threads each keeping `depth` 16 KB copies in flight: mode 0
    tiled 128-byte-swizzled tensor boxes, mode 1 plain bulk copies; the
    source (src_mb MB) stays in L2, as the GEMMs' operands do."""
    lib = _load()
    sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    nbytes = (src_mb << 20) // (1536 * 128) * (1536 * 128)
    src = torch.randint(0, 255, (nbytes,), dtype=torch.uint8, device="cuda")
    out = torch.zeros(sms, dtype=torch.int64, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    for it in (64, iters):
        st = lib.qlin_probe_fill(mode, threads, depth, sms, it, src.data_ptr(), nbytes,
                                 out.data_ptr(), err.data_ptr(), s)
        if st != 0:
            raise RuntimeError(f"qlin_probe_fill({mode}, {threads}, {depth}) returned {st}")
    torch.cuda.synchronize()
    if int(err.item()) != 0:
        raise RuntimeError("probe wait expired")
    cyc = out.cpu().double().median().item()
    return {"mode": ("tiled_128B_box", "bulk")[mode], "threads": threads, "depth": depth,
            "bytes_per_cycle_per_sm": round(threads * iters * 16384 / cyc, 1)}


def copy_rates() -> dict:
    cp = [scale_copy_cycles(w, 12, 0) for w in (1, 2, 4, 6)]
    cp += [scale_copy_cycles(w, 12, 4) for w in (1, 2, 4, 6)]
    cp += [scale_copy_cycles(1, 0, 4)]
    fill = [fill_bytes_per_cycle(m, t, d) for m in (0, 1)
            for (t, d) in ((1, 2), (1, 8), (2, 4), (4, 2), (6, 2), (8, 1))]
    return {"scale_copy": cp, "fill": fill}


if __name__ == "__main__":
    import sys
    print(json.dumps(copy_rates() if "--copies" in sys.argv[1:] else ceilings(), indent=1))
