"""GPU parity of the denoise-step linear stack (8 blocks x QKV / out / up /
down, NVFP4 W4A4, chained fused re-quantization), batch 1 and 4 (M = 4608,
18432), in the launch configuration the benchmark times.

Every layer is checked on 256 token rows that cover every 128-row M tile (and
cycle through the TMEM lane quarters), against all output columns:
- its quantized input equals, bit for bit, the oracle's NVFP4 quantization of
  the previous layer's bf16 output (the stack input x for the first layer);
- its bf16 output is within the GEMM tolerance of the oracle's exact fp64
  product of that input and the oracle-quantized weight;
- its re-quantized output is checked the same way as the next layer's input.
The static next-layer scales come from the oracle's own chain on 64 rows of
the same kind (post-training calibration)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2609_21849_gb300 import qlin, stack, synthetic

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from gpu_util import (assert_nvfp4_equal, check_stack_layers, oracle_stack_scales,
                          stratified_rows, to_dev)


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
    R = stratified_rows(M, 256, seed=9 + B)
    x = synthetic.stack_input(B)
    wlist, wqs = _weights()
    cal = stratified_rows(M, 64, seed=30 + B)
    s0, scales = oracle_stack_scales(x, wlist, wqs, cal, stack.V_COL0)

    st = stack.build_stack(B, weights=wlist)
    st.set_next_scales(scales)
    st.forward(to_dev(x))
    assert qlin.qlin_sync_status() == 0
    for i in range(4):   # the first block's weights, bit-exact
        assert_nvfp4_equal(st.layers[i].W, wqs[i], f"W{i}")
    worst = check_stack_layers(st, x, wqs, R, s0, f"stack B={B}")
    print(f"stack B={B}: {len(R)} rows per layer, worst normalised error {worst:.2e}")
