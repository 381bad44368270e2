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


def stratified_rows(M: int, n: int, seed: int = 0) -> np.ndarray:
    """Rows covering every 128-row M tile, cycling through the four 32-lane
    quarters of the tile's TMEM accumulator from tile to tile, plus the first
    and last rows, topped up with random rows to about n (sorted, unique)."""
    rng = np.random.default_rng(seed)
    rows = {0, M - 1}
    for t in range((M + 127) // 128):
        q = t % 4
        r = t * 128 + q * 32 + int(rng.integers(0, 32))
        rows.add(min(r, M - 1))
    extra = max(0, n - len(rows))
    if extra:
        rows |= set(rng.choice(M, size=min(extra, M), replace=False).tolist())
    return np.array(sorted(rows), np.int64)


def assert_requant_exact(gpu_codes, gpu_canon, y16_gpu, s_next, what=""):
    """The fused re-quantization of a layer's own bf16 output: its codes and
    scales must equal the oracle's NVFP4 quantization of that same bf16
    output with the same static tensor scale, bit for bit (every block)."""
    ref = oracle.quant_nvfp4(np.ascontiguousarray(y16_gpu), s_next)
    bad = np.argwhere(gpu_canon != ref[1])
    assert bad.size == 0, (what, "re-quantized scales differ", bad[:5])
    bad = np.argwhere(gpu_codes != ref[0])
    assert bad.size == 0, (what, "re-quantized codes differ", bad[:5])
    return ref


def check_stack_layers(st, x_bits, wqs, rows, s0, what=""):
    """Per-layer oracle parity of a linear stack's forward on the given token
    rows.  Layer i's input is checked bit-exactly against the oracle's
    quantization of the previous layer's bf16 output (for the first layer, of
    the stack input x with tensor scale s0), and its bf16 output is checked
    within GEMM_TOL against the oracle's exact fp64 product of that input and
    the oracle-quantized weight wqs[i].  Returns the worst normalised error."""
    Rt = torch.from_numpy(rows).cuda()
    a_ref = oracle.quant_nvfp4(np.ascontiguousarray(x_bits[rows]), s0)
    codes, canon, s = nvfp4_to_host(st.a0)
    assert s == np.float32(s0), (what, "input tensor scale")
    assert np.array_equal(codes[rows], a_ref[0]) and np.array_equal(canon[rows], a_ref[1]), \
        (what, "stack input quantization")
    worst = 0.0
    for i, l in enumerate(st.layers):
        yref, na, nw = oracle.gemm_nvfp4(a_ref, wqs[i])
        yb = bf16_bits(l.y.index_select(0, Rt))
        err, exact = gemm_errors(yb, yref, na, nw)
        assert err.max() <= GEMM_TOL, (what, i, l.block, l.name, err.max())
        worst = max(worst, float(err.max()))
        s_next = np.float32(f32(l.next_scale)[0])
        codes, canon, s = nvfp4_to_host(l.out_q)
        assert s == s_next, (what, i, "re-quantized tensor scale")
        win = np.ascontiguousarray(yb[:, l.rq_col0:l.rq_col0 + l.rq_cols])
        a_ref = assert_requant_exact(codes[rows], canon[rows], win, s_next, (what, i))
    return worst


def oracle_stack_scales(x_bits, wlist, wqs, rows, v_col0):
    """Static next-layer scales of a linear stack, calibrated by the oracle:
    its own chain on the given token rows (exact GEMM, bf16 rounding, dynamic
    tensor scale of each re-quantized window), as post-training calibration
    does.  Returns (input tensor scale s0, per-layer next scales)."""
    s0 = oracle.nvfp4_tensor_scale(oracle.amax_bf16(x_bits))
    a = oracle.quant_nvfp4(np.ascontiguousarray(x_bits[rows]), s0)
    scales = []
    for (_, name, _), wq in zip(wlist, wqs):
        yref, _, _ = oracle.gemm_nvfp4(a, wq)
        c0 = v_col0 if name == "qkv" else 0
        win = np.ascontiguousarray(oracle.round_bf16_array(yref)[:, c0:])
        s_next = oracle.nvfp4_tensor_scale(oracle.amax_bf16(win))
        scales.append(s_next)
        a = oracle.quant_nvfp4(win, s_next)
    return s0, scales
