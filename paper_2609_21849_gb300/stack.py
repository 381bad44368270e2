"""The denoise-step linear stack: 8 transformer blocks, each QKV (3072 -> 9216),
out-projection (3072 -> 3072), MLP up (3072 -> 12288) and down (12288 -> 3072),
all NVFP4 W4A4 with chained fused re-quantization (Sec. 4: the quantized
denoising transformer; its linears are the step's compute).

Reading where the paper is silent: attention, norms, activations and residuals
are left out (they are not linear layers), so the only shape gap is QKV
(N = 9216) -> out-projection (K = 3072).  The QKV epilogue re-quantizes the
value columns 6144..9215, which feed the out-projection.

Host-side orchestration only: every step runs in libqlin's kernels.  The
static next-layer scales come from a calibration pass (post-training
quantization) or from the caller.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch

from . import qlin, synthetic

V_COL0 = 2 * synthetic.HIDDEN  # first value column of the QKV output


@dataclass
class Layer:
    block: int
    name: str
    W: qlin.NVFP4Tensor
    N: int
    K: int
    rq_col0: int
    rq_cols: int
    y: torch.Tensor                    # bf16 [M, N]
    out_q: qlin.NVFP4Tensor            # re-quantized input of the next layer
    next_scale: torch.Tensor           # fp32 [1], static S_dec of out_q


@dataclass
class LinearStack:
    M: int
    layers: list = field(default_factory=list)
    a0: qlin.NVFP4Tensor | None = None
    workspace: torch.Tensor | None = None

    @property
    def flops(self) -> int:
        return sum(2 * self.M * l.N * l.K for l in self.layers)

    def quantize_input(self, x: torch.Tensor, stream=None):
        """Dynamic NVFP4 quantization of the stack input (amax + quantize)."""
        qlin.qlin_quantize_act_nvfp4(x, None, self.a0, self.workspace, stream)

    def forward(self, x: torch.Tensor | None = None, stream=None, write_y: bool = True):
        """One pass: (optionally) quantize x, then the 32 fused linears."""
        if x is not None:
            self.quantize_input(x, stream)
        a = self.a0
        for l in self.layers:
            qlin.qlin_linear_fused(a, l.W, l.y if write_y else None, l.next_scale, l.out_q,
                                   l.rq_col0, stream)
            a = l.out_q

    def set_next_scales(self, scales):
        for l, s in zip(self.layers, scales):
            l.next_scale.fill_(float(np.float32(s)))

    def calibrate(self, x: torch.Tensor):
        """Post-training calibration on the GPU: run the chain with plain GEMMs
        and dynamic quantization of each output window; the dynamic tensor
        scales become the static next-layer scales."""
        self.quantize_input(x)
        a = self.a0
        for l in self.layers:
            qlin.qlin_gemm_nvfp4(a, l.W, l.y)
            win = l.y[:, l.rq_col0:l.rq_col0 + l.rq_cols].contiguous()
            qlin.qlin_quantize_act_nvfp4(win, None, l.out_q, self.workspace)
            l.next_scale.copy_(l.out_q.tensor_scale)
            a = l.out_q
        torch.cuda.synchronize()


def build_stack(B: int = 1, n_blocks: int = 8, seed: int = 4, weights=None,
                device="cuda") -> LinearStack:
    """Quantize the stack's weights on the GPU (offline step) and allocate
    every activation buffer.  ``weights``: optional iterable of
    (block, name, bf16 bits) overriding the seeded generator."""
    M = synthetic.M_TOKENS * B
    st = LinearStack(M=M)
    st.workspace = qlin.alloc_workspace(device)
    st.a0 = qlin.alloc_nvfp4(M, synthetic.HIDDEN, device)
    src = weights if weights is not None else synthetic.stack_weights(n_blocks, seed)
    for b, name, wbits in src:
        N, K = wbits.shape
        w = torch.from_numpy(np.ascontiguousarray(wbits).view(np.int16)).to(device).view(torch.bfloat16)
        W = qlin.qlin_quantize_weight(w, qlin.QLIN_FMT_NVFP4, workspace=st.workspace)
        del w
        rq0, rqn = (V_COL0, N - V_COL0) if name == "qkv" else (0, N)
        st.layers.append(Layer(b, name, W, N, K, rq0, rqn,
                               torch.empty((M, N), dtype=torch.bfloat16, device=device),
                               qlin.alloc_nvfp4(M, rqn, device),
                               torch.ones(1, dtype=torch.float32, device=device)))
    torch.cuda.synchronize()
    return st
