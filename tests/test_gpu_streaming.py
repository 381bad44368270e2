"""Weight streaming on the GPU (Sec. 4, "Weight streaming"): the streamed
forward of the linear stack must give outputs bit-identical to the fully
resident forward, since only where the weights live changes, and each
streamed layer must match the oracle."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2609_21849_gb300 import qlin, stack, streaming, synthetic

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from gpu_util import check_stack_layers, oracle_stack_scales, stratified_rows, to_dev


def _outputs(st):
    return [(l.y.clone(), l.out_q.codes.clone(), l.out_q.scales.clone(),
             l.out_q.tensor_scale.clone()) for l in st.layers]


def _assert_same(st, ref, tag):
    for i, (l, (y, c, s, ts)) in enumerate(zip(st.layers, ref)):
        assert torch.equal(l.y.view(torch.int16), y.view(torch.int16)), (tag, i, "y")
        assert torch.equal(l.out_q.codes, c), (tag, i, "codes")
        assert torch.equal(l.out_q.scales, s), (tag, i, "scales")
        assert torch.equal(l.out_q.tensor_scale, ts), (tag, i, "tensor scale")


@pytest.mark.parametrize("B", [1])
def test_streamed_forward_bit_identical(B):
    st = stack.build_stack(B, n_blocks=2, seed=11)
    x = torch.randn(st.M, synthetic.HIDDEN, generator=torch.Generator().manual_seed(5))
    x = x.to(torch.bfloat16).cuda()
    st.calibrate(x)
    st.forward(x)
    torch.cuda.synchronize()
    assert qlin.qlin_sync_status() == 0
    ref = _outputs(st)

    for frac, slots, release in [(0.75, 2, False), (0.5, 2, False), (0.25, 2, False),
                                 (0.25, 3, False), (0.0, 3, False), (0.0, 2, True)]:
        for l in st.layers:                        # stale outputs must be overwritten
            l.y.zero_(); l.out_q.codes.zero_(); l.out_q.scales.zero_()
        ss = streaming.StreamedStack(st, frac, release=release, n_slots=slots)
        s = torch.cuda.Stream()
        with torch.cuda.stream(s):
            ss.forward(x, s)
            ss.forward(x, s)                       # slots reused across forwards
        torch.cuda.synchronize()
        assert qlin.qlin_sync_status() == 0
        _assert_same(st, ref, (frac, slots))
    assert all(l.W is None for l in st.layers)     # released: only the slots remain


def test_streamed_forward_in_cuda_graph():
    st = stack.build_stack(1, n_blocks=1, seed=12)
    x = torch.randn(st.M, synthetic.HIDDEN, generator=torch.Generator().manual_seed(6))
    x = x.to(torch.bfloat16).cuda()
    st.calibrate(x)
    st.forward(x)
    torch.cuda.synchronize()
    ref = _outputs(st)
    ss = streaming.StreamedStack(st, 0.25)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        ss.forward(x, s)                          # warm-up outside capture
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        ss.forward(x, s)
    for l in st.layers:
        l.y.zero_(); l.out_q.codes.zero_(); l.out_q.scales.zero_()
    torch.cuda.synchronize()
    g.replay(); g.replay()
    torch.cuda.synchronize()
    assert qlin.qlin_sync_status() == 0
    _assert_same(st, ref, "graph")


@pytest.mark.parametrize("frac,slots", [(0.25, 2), (0.0, 3)])
def test_streamed_forward_matches_oracle(frac, slots):
    # Seeded 2-block stack (the stack's own weight and input recipes), static
    # scales calibrated by the oracle; after a streamed forward (most layers
    # copied from pinned host memory into the device slots), every layer is
    # checked against the oracle on rows covering every 128-row tile.
    wlist = list(synthetic.stack_weights(2, 4))
    wqs = [oracle.quant_nvfp4(w) for (_, _, w) in wlist]
    x = synthetic.stack_input(1)
    M = x.shape[0]
    s0, scales = oracle_stack_scales(x, wlist, wqs, stratified_rows(M, 48, seed=3), stack.V_COL0)
    st = stack.build_stack(1, weights=wlist)
    st.set_next_scales(scales)
    ss = streaming.StreamedStack(st, frac, n_slots=slots)
    s = torch.cuda.Stream()
    xd = to_dev(x)
    with torch.cuda.stream(s):
        ss.forward(xd, s)
    torch.cuda.synchronize()
    assert qlin.qlin_sync_status() == 0
    assert sum(not r for r in ss.resident) >= 6, ss.resident   # most layers streamed
    worst = check_stack_layers(st, x, wqs, stratified_rows(M, 128, seed=4), s0,
                               f"streamed {frac} x{slots}")
    print(f"streamed forward ({frac:.2f} resident, {slots} slots): worst error {worst:.2e}")
