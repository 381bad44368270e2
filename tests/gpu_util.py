"""Helpers shared by the GPU parity tests: move seeded inputs to the device,
read results back, and compare the CUDA path with the CPU oracle."""
import numpy as np
import torch

import oracle
from paper_2609_21849_gb300 import qlin

# GEMM tolerance: |y_gpu - y_exact| / (||a_m||_2 * ||w_n||_2) <= 2e-3, the
# row-L2-normalised bound of the quantized linear (norms over the
# dequantized, scaled operands).
GEMM_TOL = 2e-3


def to_dev(bits: np.ndarray) -> torch.Tensor:
    """bf16 bit array (uint16) -> contiguous bf16 CUDA tensor."""
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def u8(t: torch.Tensor) -> np.ndarray:
    return t.cpu().numpy()


def f32(t: torch.Tensor) -> np.ndarray:
    return t.cpu().numpy().astype(np.float32)


def nvfp4_to_host(q: qlin.NVFP4Tensor):
    """(codes, canonical scales, S_dec) of a device NVFP4 operand."""
    codes = u8(q.codes)
    canon = oracle.unswizzle_scales(u8(q.scales), q.rows, q.K)
    return codes, canon, np.float32(f32(q.tensor_scale)[0])


def assert_nvfp4_equal(gpu: qlin.NVFP4Tensor, ref, what=""):
    codes, canon, s = nvfp4_to_host(gpu)
    rc, rs, rsd = ref
    assert s.view(np.uint32) == np.float32(rsd).view(np.uint32), (what, s, rsd)
    bad = np.argwhere(canon != rs)
    assert bad.size == 0, (what, "scales differ", bad[:5], canon[tuple(bad[0])], rs[tuple(bad[0])])
    bad = np.argwhere(codes != rc)
    assert bad.size == 0, (what, "codes differ", bad[:5], hex(codes[tuple(bad[0])]), hex(rc[tuple(bad[0])]))


def gemm_errors(y_gpu_bits: np.ndarray, y_ref: np.ndarray, na: np.ndarray, nw: np.ndarray):
    """Normalised error per output, and the fraction of outputs equal to the
    correctly rounded bf16 of the exact result."""
    yg = (y_gpu_bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    denom = np.outer(na, nw)
    denom[denom == 0] = 1.0
    err = np.abs(yg - y_ref) / denom
    exact = np.mean(y_gpu_bits == oracle.round_bf16_array(y_ref))
    return err, exact


def sample_rows(M: int, n: int, seed: int = 0) -> np.ndarray:
    """First, last and random rows (sorted, unique)."""
    rng = np.random.default_rng(seed)
    rows = {0, M - 1} | set(rng.choice(M, size=min(n, M), replace=False).tolist())
    return np.array(sorted(rows), np.int64)


def requant_agreement(gpu_codes, gpu_canon, y16_gpu, y16_ref, s_next):
    """Compare re-quantized blocks of the GPU with the oracle's quantization of
    its own bf16 rounding of the exact result.  Blocks whose 16 bf16 inputs
    agree must be identical; returns the fraction of identical blocks."""
    rows, K = y16_ref.shape
    rc, rs, _ = oracle.quant_nvfp4(y16_ref, s_next)
    same_in = (y16_gpu == y16_ref).reshape(rows, K // 16, 16).all(axis=2)
    same_out = (gpu_canon == rs) & (gpu_codes == rc).reshape(rows, K // 16, 8).all(axis=2)
    bad = np.argwhere(same_in & ~same_out)
    assert bad.size == 0, ("re-quantized block differs on identical inputs", bad[:5])
    return same_out.mean()
