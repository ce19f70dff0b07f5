"""Device buffers and the call sequence of one adaptation step (steps a1..a12).

Plumbing only: torch allocates the caller-owned device buffers the C ABI writes
into, and ``StepRunner`` issues the seven library calls of one step in order on
one stream -- eight with the router backward (``router_grad=True``), which adds
the gradient of the gating network.  No arithmetic of the method happens here.
"""
from __future__ import annotations

import copy

import torch

from . import (VMOE_BF16, vmoe_combine, vmoe_dispatch, vmoe_expert_bwd,
               vmoe_expert_bwd_workspace_size, vmoe_expert_fwd, vmoe_problem_capacity, vmoe_route,
               vmoe_router_bwd)


class Buffers:
    """Every intermediate and output of one step for problem ``p`` on ``device``."""

    def __init__(self, p, device="cuda"):
        T, N, d, f, E, k = p.T, p.N, p.d_model, p.d_ff, p.E, p.k
        C = vmoe_problem_capacity(p)
        dt = torch.bfloat16 if p.dtype == VMOE_BF16 else torch.float32
        self.C = C
        self.dtype = dt
        f32, i32 = torch.float32, torch.int32
        e = lambda *shape, dtype=dt: torch.empty(shape, dtype=dtype, device=device)  # noqa: E731
        self.logits = e(T, N, E, dtype=f32)
        self.idx = e(T, N, k, dtype=i32)
        self.gate = e(T, N, k, dtype=f32)
        self.slot = e(T, N, k, dtype=i32)
        self.load = e(T, E, dtype=i32)
        self.xe = e(T, E, C, d)
        self.h = e(T, E, C, f)
        self.a = e(T, E, C, f)
        self.ye = e(T, E, C, d)
        self.y = e(T, N, d)
        self.dye = e(T, E, C, d)
        self.dxe = e(T, E, C, d)
        self.dw1 = e(T, E, d, f)
        self.dw2 = e(T, E, f, d)
        self.dx = e(T, N, d)
        # router backward
        self.dgate = e(T, N, k, dtype=f32)
        self.dlogits = e(T, N, E, dtype=f32)
        self.dw_router = e(T, d, E, dtype=f32)
        self.dbias = e(T, E, dtype=f32)
        self.workspace = torch.empty(vmoe_expert_bwd_workspace_size(p), dtype=torch.uint8,
                                     device=device)


class StepRunner:
    """Issues the library calls of one forward + backward step.

    ``inputs`` holds device tensors x, dy [T,N,d], w_router [T,d,E], bias [T,E]
    or None, w1 [T,E,d,f], w2 [T,E,f,d].  With ``router_grad`` the backward also
    produces dW_r and dbias and adds the router's share to dX.
    """

    def __init__(self, p, inputs, bufs: Buffers | None = None, router_grad: bool = False):
        self.p = p
        self.inp = inputs
        self.router_grad = router_grad
        self.b = bufs if bufs is not None else Buffers(p, inputs["x"].device)

    def forward(self, stream=None):
        p, i, b = self.p, self.inp, self.b
        vmoe_route(p, i["x"], i["w_router"], i.get("bias"), b.logits, b.idx, b.gate, b.slot,
                   b.load, stream)
        vmoe_dispatch(p, i["x"], None, b.idx, b.slot, b.load, b.xe, stream)
        vmoe_expert_fwd(p, b.xe, i["w1"], i["w2"], b.load, b.h, b.a, b.ye, stream)
        vmoe_combine(p, b.ye, b.gate, b.idx, b.slot, b.y, stream)

    def backward(self, stream=None):
        p, i, b = self.p, self.inp, self.b
        vmoe_dispatch(p, i["dy"], b.gate, b.idx, b.slot, b.load, b.dye, stream)
        vmoe_expert_bwd(p, b.xe, b.h, b.a, i["w1"], i["w2"], b.dye, b.load, b.dxe, b.dw1, b.dw2,
                        b.workspace, stream=stream)
        vmoe_combine(p, b.dxe, None, b.idx, b.slot, b.dx, stream)
        if self.router_grad:
            self.router_backward(stream)

    def router_backward(self, stream=None):
        p, i, b = self.p, self.inp, self.b
        vmoe_router_bwd(p, i["x"], i["w_router"], b.logits, b.idx, b.gate, b.slot, i["dy"], b.ye,
                        b.dgate, b.dlogits, b.dw_router, b.dbias, b.dx, stream)

    def step(self, stream=None):
        self.forward(stream)
        self.backward(stream)


class HostPipeline:
    """Steps from pinned host inputs to pinned host outputs, with the host<->device
    copies overlapped with compute.

    Two slots each hold device copies of x, dY, y and dX; everything else (weights,
    activations, gradients) is shared, as the steps run in order on one compute
    stream.  The copies run on their own stream: step i+1's x and dY upload while
    step i computes, y of step i is read back while its backward runs, and dX as
    soon as it is done.  ``weights`` holds w_router, bias, w1, w2 on the device.
    """

    def __init__(self, p, weights, bufs: Buffers | None = None, device="cuda",
                 router_grad: bool = False):
        self.p = p
        base = bufs if bufs is not None else Buffers(p, device)
        self.slots = []
        for _ in range(2):
            b = copy.copy(base)
            b.y = torch.empty_like(base.y)
            b.dx = torch.empty_like(base.dx)
            inp = dict(weights)
            inp["x"] = torch.empty_like(base.y)
            inp["dy"] = torch.empty_like(base.y)
            self.slots.append(StepRunner(p, inp, b, router_grad=router_grad))
        self.copy_stream = torch.cuda.Stream(device)
        ev = lambda: [torch.cuda.Event() for _ in range(2)]  # noqa: E731
        self.h2d, self.fwd, self.done, self.d2h = ev(), ev(), ev(), ev()

    def _upload(self, slot, x_host, dy_host):
        r = self.slots[slot]
        with torch.cuda.stream(self.copy_stream):
            r.inp["x"].copy_(x_host, non_blocking=True)
            r.inp["dy"].copy_(dy_host, non_blocking=True)
        self.h2d[slot].record(self.copy_stream)

    def run(self, inputs, outputs, stream=None):
        """inputs[i] = (x, dY) and outputs[i] = (y, dX): pinned host tensors of
        step i.  Enqueues every step and returns; synchronise the copy stream (or
        the device) before reading the outputs."""
        cs = stream if stream is not None else torch.cuda.current_stream()
        steps = len(inputs)
        if steps == 0:
            return
        self._upload(0, *inputs[0])
        for i in range(steps):
            s = i % 2
            r = self.slots[s]
            cs.wait_event(self.h2d[s])
            if i >= 2:  # this slot's y / dX of step i-2 have been read back
                cs.wait_event(self.d2h[s])
            r.forward(cs)
            self.fwd[s].record(cs)
            r.backward(cs)
            self.done[s].record(cs)
            if i + 1 < steps:  # the other slot is free once step i-1 has finished
                if i >= 1:
                    self.copy_stream.wait_event(self.done[s ^ 1])
                self._upload(s ^ 1, *inputs[i + 1])
            y_host, dx_host = outputs[i]
            self.copy_stream.wait_event(self.fwd[s])
            with torch.cuda.stream(self.copy_stream):
                y_host.copy_(r.b.y, non_blocking=True)
            self.copy_stream.wait_event(self.done[s])
            with torch.cuda.stream(self.copy_stream):
                dx_host.copy_(r.b.dx, non_blocking=True)
            self.d2h[s].record(self.copy_stream)
