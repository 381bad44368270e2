"""The embedding translator's MLP forward on the quantized small-M path.

The paper's translator (Sec. 3, Table 1) maps the 0.6B encoder's per-token
features (1024 wide) to the 4B encoder's conditioning space (2560 wide); its
best variant, d3072, is a single 3072-wide MLP.  Here that forward runs as two
chained quantized linears on the 512 tokens of a prompt batch:

  x [512, 1024] bf16 --(dynamic quantization)--> x_q
  h = x_q W1^T  [512, 3072]   (epilogue re-quantizes h to h_q, static scale)
  y = h_q W2^T  [512, 2560]   bf16 out

in NVFP4 (W4A4, qlin_linear_fused) or FP8 (W8A8 with per-channel weight
scales, qlin_linear_fused_fp8).  Reading where the paper is silent: it gives
the MLP's widths but neither its activation function nor norms, so the
forward keeps the two linears only, as the denoiser's linear stack does; the
hidden activations' static scale comes from a calibration pass (post-training
quantization, Sec. 4).  Trained weights are not available: the weights are
seeded random matrices of the translator's shapes.

Host-side orchestration only: every step runs in libqlin's kernels.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np
import torch

from . import qlin


@dataclass
class TranslatorMLP:
    fmt: str                      # "nvfp4" or "fp8"
    M: int
    W1: object                    # quantized [hidden, in]
    W2: object                    # quantized [out, hidden]
    x_q: object                   # quantized input [M, in]
    h_q: object                   # re-quantized hidden [M, hidden]
    h: torch.Tensor               # bf16 hidden (written only when asked)
    y: torch.Tensor               # bf16 output [M, out]
    h_scale: torch.Tensor         # fp32 [1]: static S_dec of h_q
    workspace: torch.Tensor

    @property
    def flops(self) -> int:
        return 2 * self.M * (self.W1.rows * self.W1.K + self.W2.rows * self.W2.K)

    def forward(self, x: torch.Tensor, stream=None, write_hidden: bool = False) -> torch.Tensor:
        """x [M, in] bf16 -> y [M, out] bf16 (dynamic input scale; the hidden
        activations' bf16 values are written only with write_hidden)."""
        h = self.h if write_hidden else None
        if self.fmt == "nvfp4":
            qlin.qlin_quantize_act_nvfp4(x, None, self.x_q, self.workspace, stream)
            qlin.qlin_linear_fused(self.x_q, self.W1, h, self.h_scale, self.h_q, 0, stream)
            qlin.qlin_gemm_nvfp4(self.h_q, self.W2, self.y, stream)
        else:
            qlin.qlin_quantize_act_fp8(x, None, self.x_q, self.workspace, stream)
            qlin.qlin_linear_fused_fp8(self.x_q, self.W1, h, self.h_scale, self.h_q, 0, stream)
            qlin.qlin_gemm_fp8(self.h_q, self.W2, self.y, stream)
        return self.y

    def calibrate(self, x: torch.Tensor) -> float:
        """Post-training calibration on the GPU: the hidden activations'
        dynamic tensor scale on x becomes the static scale."""
        if self.fmt == "nvfp4":
            qlin.qlin_quantize_act_nvfp4(x, None, self.x_q, self.workspace)
            qlin.qlin_gemm_nvfp4(self.x_q, self.W1, self.h)
            q = qlin.qlin_quantize_act_nvfp4(self.h, None, None, self.workspace)
            self.h_scale.copy_(q.tensor_scale)
        else:
            qlin.qlin_quantize_act_fp8(x, None, self.x_q, self.workspace)
            qlin.qlin_gemm_fp8(self.x_q, self.W1, self.h)
            q = qlin.qlin_quantize_act_fp8(self.h, None, None, self.workspace)
            self.h_scale.copy_(q.scale)
        torch.cuda.synchronize()
        return float(self.h_scale.item())

    def set_hidden_scale(self, s: float):
        self.h_scale.fill_(float(np.float32(s)))


def build_translator(fmt: str, w1_bits: np.ndarray, w2_bits: np.ndarray, M: int = 512,
                     device="cuda") -> TranslatorMLP:
    """Quantize the two weights on the GPU (offline step) and allocate the
    activations of an M-token forward."""
    if fmt not in ("nvfp4", "fp8"):
        raise ValueError("fmt must be 'nvfp4' or 'fp8'")
    dev = lambda b: torch.from_numpy(np.ascontiguousarray(b).view(np.int16)).to(device).view(
        torch.bfloat16)
    hidden, k_in = w1_bits.shape
    out = w2_bits.shape[0]
    if w2_bits.shape[1] != hidden:
        raise ValueError("W2 must take W1's output width")
    ws = qlin.alloc_workspace(device)
    if fmt == "nvfp4":
        W1 = qlin.qlin_quantize_weight(dev(w1_bits), qlin.QLIN_FMT_NVFP4, workspace=ws)
        W2 = qlin.qlin_quantize_weight(dev(w2_bits), qlin.QLIN_FMT_NVFP4, workspace=ws)
        x_q, h_q = qlin.alloc_nvfp4(M, k_in, device), qlin.alloc_nvfp4(M, hidden, device)
    else:
        W1 = qlin.qlin_quantize_weight(dev(w1_bits), qlin.QLIN_FMT_FP8)
        W2 = qlin.qlin_quantize_weight(dev(w2_bits), qlin.QLIN_FMT_FP8)
        x_q, h_q = qlin.alloc_fp8(M, k_in, False, device), qlin.alloc_fp8(M, hidden, False, device)
    t = TranslatorMLP(fmt, M, W1, W2, x_q, h_q,
                      torch.empty((M, hidden), dtype=torch.bfloat16, device=device),
                      torch.empty((M, out), dtype=torch.bfloat16, device=device),
                      torch.ones(1, dtype=torch.float32, device=device), ws)
    torch.cuda.synchronize()
    return t
