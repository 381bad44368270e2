"""GPU parity of the denoise-step linear stack (8 blocks x QKV / out / up /
down, NVFP4 W4A4, chained fused re-quantization), batch 1 and 4 (M = 4608,
18432), in the launch configuration the benchmark times.

The oracle runs the same chain on a few sampled token rows (every layer is
row-local once its static input scale is fixed): exact fp64 GEMM, its own bf16
rounding, and re-quantization with the next-layer scale calibrated on those
rows.  The GPU runs all rows with the same static scales."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2609_21849_gb300 import qlin, stack, synthetic

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from gpu_util import (GEMM_TOL, assert_nvfp4_equal, bf16_bits, gemm_errors, nvfp4_to_host,
                          requant_agreement, sample_rows, to_dev)


_WEIGHTS = {}


def _weights():
    """The stack's seeded weights and the oracle's quantization of them
    (shared by the batch sizes)."""
    if not _WEIGHTS:
        wlist = list(synthetic.stack_weights(8, 4))
        _WEIGHTS["w"] = wlist
        _WEIGHTS["q"] = [oracle.quant_nvfp4(w) for (_, _, w) in wlist]
    return _WEIGHTS["w"], _WEIGHTS["q"]


@pytest.mark.parametrize("B", [1, 4])
def test_stack_chain(B):
    M = synthetic.M_TOKENS * B
    R = sample_rows(M, 6, seed=9 + B)
    x = synthetic.stack_input(B)
    wlist, wqs = _weights()

    # ---- oracle chain on the sampled rows
    s0 = oracle.nvfp4_tensor_scale(oracle.amax_bf16(x))
    a_rows = oracle.quant_nvfp4(np.ascontiguousarray(x[R]), s0)
    a0_ref = a_rows
    refs, wq0 = [], None
    for i, (b, name, w) in enumerate(wlist):
        wq = wqs[i]
        if i < 4:
            wq0 = (wq0 or []) + [wq]
        yref, na, nw = oracle.gemm_nvfp4(a_rows, wq)
        y16 = oracle.round_bf16_array(yref)
        c0 = stack.V_COL0 if name == "qkv" else 0
        win = np.ascontiguousarray(y16[:, c0:])
        s_next = oracle.nvfp4_tensor_scale(oracle.amax_bf16(win))
        refs.append((yref, na, nw, win, s_next, c0))
        a_rows = oracle.quant_nvfp4(win, s_next)

    # ---- GPU: all rows, same weights and static scales
    st = stack.build_stack(B, weights=wlist)
    st.set_next_scales([r[4] for r in refs])
    st.forward(to_dev(x))
    assert qlin.qlin_sync_status() == 0

    for i in range(4):   # first block's weights bit-exact
        assert_nvfp4_equal(st.layers[i].W, wq0[i], f"W{i}")
    codes, canon, s = nvfp4_to_host(st.a0)
    assert s == np.float32(s0)
    assert np.array_equal(codes[R], a0_ref[0]) and np.array_equal(canon[R], a0_ref[1])

    Rt = torch.from_numpy(R).cuda()
    worst, agree_min = 0.0, 1.0
    for i, l in enumerate(st.layers):
        yref, na, nw, win, s_next, c0 = refs[i]
        yb = bf16_bits(l.y.index_select(0, Rt))
        err, exact = gemm_errors(yb, yref, na, nw)
        assert err.max() <= GEMM_TOL, (i, l.block, l.name, err.max())
        codes, canon, s = nvfp4_to_host(l.out_q)
        assert s == np.float32(s_next)
        agree = requant_agreement(codes[R], canon[R], np.ascontiguousarray(yb[:, c0:]), win, s_next)
        assert agree >= 0.99, (i, agree)
        worst, agree_min = max(worst, err.max()), min(agree_min, agree)
    print(f"stack B={B}: worst normalised error {worst:.2e}, min requant agreement {agree_min:.5f}")
