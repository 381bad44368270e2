"""Runs one libqlin kernel on a fixed workload a given number of times, for
profilers (ncu) and quick timing:

  python -m paper_2609_21849_gb300.profile_case CASE [--warmup W] [--launches L]

Cases (seeded synthetic inputs, shapes of the paper's workloads):
  quant_nvfp4      static-scale NVFP4 quantization of x [4608, 3072]
  quant_nvfp4_dyn  dynamic (amax + quantize) of the same
  quant_fp8        static-scale FP8 quantization of x [4608, 3072]
  gemm_nvfp4       NVFP4 GEMM 4608 x 12288 x 3072, bf16 out
  fused_nvfp4      the same with the fused NVFP4 re-quantization
  gemm_fp8         FP8 GEMM 4608 x 3072 x 3072
  small_nvfp4      NVFP4 GEMM 512 x 2560 x 1024 (translator shape)
Prints the mean device time per launch (CUDA events, not for use under a
profiler).
"""
from __future__ import annotations

import argparse

import numpy as np
import torch

from . import build, qlin, synthetic


def _dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def make_case(name: str):
    if name.startswith("quant"):
        x = _dev(synthetic.act_entry_outliers(2, 4608, 3072))
        if name == "quant_fp8":
            out = qlin.alloc_fp8(4608, 3072, False)
            sc = torch.tensor([np.float32(0.05)], device="cuda")
            return lambda: qlin.qlin_quantize_act_fp8(x, sc, out)
        out = qlin.alloc_nvfp4(4608, 3072)
        if name == "quant_nvfp4_dyn":
            ws = qlin.alloc_workspace()
            return lambda: qlin.qlin_quantize_act_nvfp4(x, None, out, ws)
        sc = torch.tensor([np.float32(0.01)], device="cuda")
        return lambda: qlin.qlin_quantize_act_nvfp4(x, sc, out)
    if name in ("gemm_nvfp4", "fused_nvfp4"):
        xb, wb = synthetic.nvfp4_mlp_up()
        A = qlin.qlin_quantize_act_nvfp4(_dev(xb))
        W = qlin.qlin_quantize_weight(_dev(wb), qlin.QLIN_FMT_NVFP4)
        y = torch.empty((A.rows, W.rows), dtype=torch.bfloat16, device="cuda")
        if name == "gemm_nvfp4":
            return lambda: qlin.qlin_gemm_nvfp4(A, W, y)
        yq = qlin.alloc_nvfp4(A.rows, W.rows)
        sc = torch.tensor([np.float32(0.002)], device="cuda")
        return lambda: qlin.qlin_linear_fused(A, W, y, sc, yq)
    if name == "gemm_fp8":
        xb, wb = synthetic.fp8_linear()
        A = qlin.qlin_quantize_act_fp8(_dev(xb))
        W = qlin.qlin_quantize_weight(_dev(wb), qlin.QLIN_FMT_FP8)
        y = torch.empty((A.rows, W.rows), dtype=torch.bfloat16, device="cuda")
        return lambda: qlin.qlin_gemm_fp8(A, W, y)
    if name == "small_nvfp4":
        x1, _, w1, _ = synthetic.translator()
        A = qlin.qlin_quantize_act_nvfp4(_dev(x1))
        W = qlin.qlin_quantize_weight(_dev(w1), qlin.QLIN_FMT_NVFP4)
        y = torch.empty((A.rows, W.rows), dtype=torch.bfloat16, device="cuda")
        return lambda: qlin.qlin_gemm_nvfp4(A, W, y)
    raise SystemExit(f"unknown case {name}")


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("case")
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--launches", type=int, default=3)
    a = ap.parse_args()
    build.build()
    fn = make_case(a.case)
    torch.cuda.synchronize()
    for _ in range(a.warmup):
        fn()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(a.launches):
        fn()
    e1.record()
    e1.synchronize()
    st = qlin.qlin_sync_status()
    if st != 0:
        raise SystemExit(f"device status {qlin.qlin_status_str(st)}")
    print(f"{a.case}: {e0.elapsed_time(e1) * 1e3 / a.launches:.2f} us per launch")


if __name__ == "__main__":
    main()
