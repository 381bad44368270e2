"""Weight streaming on the GPU (Sec. 4, "Weight streaming"): the streamed
forward of the linear stack must give outputs bit-identical to the fully
resident forward, since only where the weights live changes."""
import pytest

torch = pytest.importorskip("torch")

from paper_2609_21849_gb300 import qlin, stack, streaming, synthetic

pytestmark = pytest.mark.gpu


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
