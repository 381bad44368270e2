"""Weight streaming for the denoise-step linear stack (Sec. 4, "Weight
streaming"): only a resident subset of the layers' weights stays in device
memory; the others live in pinned host memory and are copied into a small
ring of device slots (two at the memory floor) ahead of use, on a copy stream, overlapped with the compute of
the layers in between.  Only where the weights live changes, so the outputs
are bit-identical to a fully resident run.

The paper's model of the cost, restated:
  lambda = L * M / W    (L: compute time between successive linears,
                         M: host -> device rate, W: a layer's weight bytes)
  lambda >= 1: every copy hides behind compute;
  lambda <  1: the reservoir drains, and the awaited copies add
               Delta = (N - K) * W / M   (N layers, K of them overlapped).
  Device memory floor: T_min = 2 * W_max + A_max (two weight slots plus the
  largest activation that coexists with them).

Host orchestration only: the linears are libqlin's fused NVFP4 kernels; the
copies are stream-ordered device copies of caller-owned pinned buffers.
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

from . import qlin


# ------------------------------------------------------------ pure model ---

def resident_layers(n_layers: int, fraction: float) -> list[bool]:
    """Which layers stay resident for a residency fraction in [0, 1]: the
    resident ones are spread evenly over the execution order, so every
    streamed layer's copy overlaps the compute of resident layers too."""
    k = max(0, min(n_layers, round(fraction * n_layers)))
    res = [False] * n_layers
    for j in range(k):
        res[(j * n_layers) // k] = True
    return res


def copy_plan(resident: list[bool], n_slots: int = 2) -> list[tuple[int, int]]:
    """(layer, slot) for each streamed layer in execution order; streamed
    layers take the device slots round-robin (two slots: layers i and i+1 of
    the paper's memory floor)."""
    plan, k = [], 0
    for i, r in enumerate(resident):
        if not r:
            plan.append((i, k % n_slots))
            k += 1
    return plan


def reservoir_lambda(L_s: float, M_bytes_per_s: float, W_bytes: float) -> float:
    """The reservoir decay factor lambda = L * M / W."""
    return L_s * M_bytes_per_s / W_bytes


def predicted_overhead(n_layers: int, k_overlapped: int, W_bytes: float,
                       M_bytes_per_s: float) -> float:
    """Delta = (N - K) * W / M (seconds): the added latency when lambda < 1."""
    return (n_layers - k_overlapped) * W_bytes / M_bytes_per_s


def simulate(resident: list[bool], L_s, copy_s, n_slots: int = 2) -> tuple[float, int]:
    """Event-level timing of the slot schedule that StreamedStack runs (not
    the paper's closed form): one copy engine takes the streamed layers'
    copies in order; the copy into a slot starts once the layer that last read
    the slot has finished; a streamed layer starts once its copy has landed.
    ``L_s`` / ``copy_s``: per-layer compute and copy times (scalars or lists).
    Returns (finish time, number of streamed layers that waited on their
    copy): the latter is N - K in the paper's Delta."""
    n = len(resident)
    L = L_s if isinstance(L_s, (list, tuple)) else [L_s] * n
    C = copy_s if isinstance(copy_s, (list, tuple)) else [copy_s] * n
    plan = copy_plan(resident, n_slots)
    landed, slot_free = {}, [0.0] * n_slots
    engine = 0.0
    t = 0.0
    def issue(j):
        nonlocal engine
        layer, slot = plan[j]
        engine = max(engine, slot_free[slot]) + C[layer]
        landed[layer] = engine
    for j in range(min(n_slots, len(plan))):
        issue(j)
    k = awaited = 0
    for i in range(n):
        if not resident[i]:
            awaited += landed[i] > t
            t = max(t, landed[i])
        t += L[i]
        if not resident[i]:
            slot_free[plan[k][1]] = t
            if k + n_slots < len(plan):
                issue(k + n_slots)
            k += 1
    return t, awaited


def t_min(w_max_bytes: int, a_max_bytes: int, n_slots: int = 2) -> int:
    """Device memory floor of streaming: the weight slots (two in the paper)
    plus the peak activation."""
    return n_slots * w_max_bytes + a_max_bytes


# ------------------------------------------------------------- runtime ---

@dataclass
class _Host:
    codes: torch.Tensor          # pinned uint8
    scales: torch.Tensor         # pinned uint8
    tensor_scale: torch.Tensor   # pinned float32 [1]


class StreamedStack:
    """A LinearStack whose non-resident layers' NVFP4 weights are held in
    pinned host memory and streamed through ``n_slots`` device slots (two by
    default, the paper's floor; a third lets each copy start one layer
    earlier, which pays when the copy engine is the bound).  With
    ``release`` the stack's device copies of those weights are dropped (the
    stack then runs only through this object)."""

    def __init__(self, stack, fraction: float, release: bool = True, n_slots: int = 2):
        if n_slots < 2:
            raise ValueError("weight streaming needs at least two device slots")
        self.n_slots = n_slots
        self.stack = stack
        n = len(stack.layers)
        self.resident = resident_layers(n, fraction)
        self.plan = copy_plan(self.resident, n_slots)
        self.host: dict[int, _Host] = {}
        self.weights = [l.W for l in stack.layers]     # resident layers keep theirs
        cb = sb = 0
        for i, l in enumerate(stack.layers):
            if self.resident[i]:
                continue
            W = l.W
            self.host[i] = _Host(W.codes.cpu().pin_memory(), W.scales.cpu().pin_memory(),
                                 W.tensor_scale.cpu().pin_memory())
            cb, sb = max(cb, W.codes.numel()), max(sb, W.scales.numel())
            self.weights[i] = None                       # device copy released
        dev = stack.a0.codes.device
        ns = n_slots if self.plan else 0
        self.slot_codes = [torch.empty(cb, dtype=torch.uint8, device=dev) for _ in range(ns)]
        self.slot_scales = [torch.empty(sb, dtype=torch.uint8, device=dev) for _ in range(ns)]
        self.slot_ts = [torch.empty(1, dtype=torch.float32, device=dev) for _ in range(ns)]
        self.copy_stream = torch.cuda.Stream(device=dev)
        self.copied = [torch.cuda.Event() for _ in range(ns)]   # slot filled
        self.freed = [torch.cuda.Event() for _ in range(ns)]    # slot's last reader done
        if release:
            for l, w in zip(stack.layers, self.weights):
                if w is None:
                    l.W = None
        torch.cuda.synchronize(dev)

    @property
    def slot_bytes(self) -> int:
        return sum(t.numel() for t in self.slot_codes + self.slot_scales)

    def _issue_copy(self, layer: int, slot: int):
        h, l = self.host[layer], self.stack.layers[layer]
        cs = self.copy_stream
        cs.wait_event(self.freed[slot])
        with torch.cuda.stream(cs):
            self.slot_codes[slot][:h.codes.numel()].copy_(h.codes.view(-1), non_blocking=True)
            self.slot_scales[slot][:h.scales.numel()].copy_(h.scales, non_blocking=True)
            self.slot_ts[slot].copy_(h.tensor_scale, non_blocking=True)
        self.copied[slot].record(cs)

    def _slot_tensor(self, layer: int, slot: int) -> qlin.NVFP4Tensor:
        h, l = self.host[layer], self.stack.layers[layer]
        codes = self.slot_codes[slot][:h.codes.numel()].view(l.N, l.K // 2)
        return qlin.NVFP4Tensor(codes, self.slot_scales[slot][:h.scales.numel()],
                                self.slot_ts[slot], l.N, l.K)

    def forward(self, x: torch.Tensor | None = None, stream=None, write_y: bool = True):
        """The stack's forward with streamed weights (same kernels, same
        operands, so the same outputs)."""
        st = self.stack
        stream = stream if stream is not None else torch.cuda.current_stream()
        for e in self.freed:
            e.record(stream)
        # the first n_slots streamed layers' copies start at once
        for layer, slot in self.plan[:self.n_slots]:
            self._issue_copy(layer, slot)
        if x is not None:
            st.quantize_input(x, stream)
        a = st.a0
        k = 0
        for i, l in enumerate(st.layers):
            if self.resident[i]:
                W = self.weights[i]
            else:
                slot = self.plan[k][1]
                stream.wait_event(self.copied[slot])
                W = self._slot_tensor(i, slot)
            qlin.qlin_linear_fused(a, W, l.y if write_y else None, l.next_scale, l.out_q,
                                   l.rq_col0, stream)
            if not self.resident[i]:
                self.freed[slot].record(stream)
                if k + self.n_slots < len(self.plan):  # refill this slot
                    self._issue_copy(*self.plan[k + self.n_slots])
                k += 1
            a = l.out_q
        if self.plan:                                  # join the copy stream back
            stream.wait_stream(self.copy_stream)
