"""Python binding of libvmoe: one adaptation step of T concurrent V-MoE expert layers on GB300.

Argument marshalling only.  Every step of the path runs in the CUDA kernels of
``libvmoe.so`` (built in-tree by ``_build.build()``); there is no Python, PyTorch
or CPU fallback, and importing a function whose library is missing raises.

The functions carry the C names (``vmoe_route``, ``vmoe_dispatch``,
``vmoe_expert_fwd``, ``vmoe_expert_bwd``, ``vmoe_combine``) and take torch tensors
(device memory, any dtype matching the problem) or raw integer device pointers;
``stream`` is a ``torch.cuda.Stream``, a raw ``cudaStream_t`` integer, or None for
the current torch stream.  A non-zero status raises ``VmoeError``.
"""
from __future__ import annotations

import ctypes
import os

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.environ.get("VMOE_LIBRARY", os.path.join(PKG, "libvmoe.so"))

VMOE_OK = 0
VMOE_ERR_INVALID = -1
VMOE_ERR_UNSUPPORTED = -2
VMOE_ERR_CUDA = -3
VMOE_ERR_DEVICE_TIMEOUT = -4

VMOE_F32 = 0
VMOE_BF16 = 1

VMOE_LOGITS_IN = 1 << 0
VMOE_NO_RENORM = 1 << 1
VMOE_GELU_TANH = 1 << 2

# Every symbol include/vmoe.h declares.
EXPORTS = ("vmoe_version", "vmoe_status_string", "vmoe_problem_capacity", "vmoe_route",
           "vmoe_dispatch", "vmoe_expert_fwd", "vmoe_expert_bwd_workspace_size",
           "vmoe_expert_bwd_min_workspace_size",
           "vmoe_expert_bwd", "vmoe_expert_bwd_static_scratch", "vmoe_combine", "vmoe_router_bwd", "vmoe_plan_slices", "vmoe_plan_shares",
           "vmoe_attn_expert_fwd", "vmoe_attn_expert_bwd", "vmoe_attn_expert_bwd_workspace_size",
           "vmoe_device_status", "vmoe_selftest_bounded_wait", "vmoe_trace_enable",
           "vmoe_trace_disable", "vmoe_trace_get")


class VmoeError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__("%s: %s" % (where, status_string(status)))


class VmoeProblem(ctypes.Structure):
    """Mirror of ``vmoe_problem`` in include/vmoe.h."""
    _fields_ = [("T", ctypes.c_int32), ("N", ctypes.c_int32), ("d_model", ctypes.c_int32),
                ("d_ff", ctypes.c_int32), ("E", ctypes.c_int32), ("k", ctypes.c_int32),
                ("capacity_factor", ctypes.c_double), ("capacity", ctypes.c_int32),
                ("dtype", ctypes.c_int32), ("flags", ctypes.c_uint32)]


_lib = None
_P = ctypes.c_void_p


def library():
    """The loaded libvmoe (ctypes.CDLL).  Raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                "libvmoe.so not found at %s: build it first with "
                "`python -c 'import __graft_entry__ as g; g.build()'`" % LIB_PATH)
        lib = ctypes.CDLL(LIB_PATH)
        PP = ctypes.POINTER(VmoeProblem)
        sig = {
            "vmoe_version": (ctypes.c_int, []),
            "vmoe_status_string": (ctypes.c_char_p, [ctypes.c_int]),
            "vmoe_problem_capacity": (ctypes.c_int, [PP]),
            "vmoe_route": (ctypes.c_int, [PP] + [_P] * 8 + [_P]),
            "vmoe_dispatch": (ctypes.c_int, [PP] + [_P] * 6 + [_P]),
            "vmoe_expert_fwd": (ctypes.c_int, [PP] + [_P] * 7 + [_P]),
            "vmoe_expert_bwd_workspace_size": (ctypes.c_size_t, [PP]),
            "vmoe_expert_bwd_min_workspace_size": (ctypes.c_size_t, [PP]),
            "vmoe_expert_bwd": (ctypes.c_int, [PP] + [_P] * 11 + [ctypes.c_size_t, _P]),
            "vmoe_expert_bwd_static_scratch": (ctypes.c_int, [PP] + [_P] * 10 + [_P]),
            "vmoe_combine": (ctypes.c_int, [PP] + [_P] * 5 + [_P]),
            "vmoe_router_bwd": (ctypes.c_int, [PP] + [_P] * 13 + [_P]),
            "vmoe_attn_expert_fwd": (ctypes.c_int, [PP, ctypes.c_int] + [_P] * 9),
            "vmoe_attn_expert_bwd_workspace_size": (ctypes.c_size_t, [PP, ctypes.c_int]),
            "vmoe_attn_expert_bwd": (ctypes.c_int, [PP, ctypes.c_int] + [_P] * 12 + [ctypes.c_size_t, _P]),
            "vmoe_plan_slices": (ctypes.c_int, [ctypes.c_int, _P, _P, ctypes.c_int64,
                                                ctypes.c_double, ctypes.c_double, _P, _P]),
            "vmoe_plan_shares": (ctypes.c_int, [ctypes.c_int, _P, _P, _P, ctypes.c_int32, _P]),
            "vmoe_device_status": (ctypes.c_int, [ctypes.c_int]),
            "vmoe_selftest_bounded_wait": (ctypes.c_int, [ctypes.c_longlong, _P]),
            "vmoe_trace_enable": (ctypes.c_int, [ctypes.c_int]),
            "vmoe_trace_disable": (ctypes.c_int, []),
            "vmoe_trace_get": (ctypes.c_int, [ctypes.c_int, ctypes.POINTER(ctypes.c_char_p),
                                              ctypes.POINTER(ctypes.c_float)]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def status_string(status: int) -> str:
    try:
        return library().vmoe_status_string(int(status)).decode()
    except Exception:  # library not loadable
        return "status %d" % status


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(st: int, where: str):
    if st != VMOE_OK:
        raise VmoeError(st, where)


def problem(T, N, d_model, d_ff, E, k, capacity_factor, dtype="bf16", flags=0, capacity=0):
    """Build a VmoeProblem; ``dtype`` is "bf16", "f32" or a VMOE_* code."""
    if isinstance(dtype, str):
        dtype = {"bf16": VMOE_BF16, "f32": VMOE_F32}[dtype]
    return VmoeProblem(int(T), int(N), int(d_model), int(d_ff), int(E), int(k),
                       float(capacity_factor), int(capacity), int(dtype), int(flags))


def vmoe_version() -> int:
    return library().vmoe_version()


def vmoe_problem_capacity(p: VmoeProblem) -> int:
    c = library().vmoe_problem_capacity(ctypes.byref(p))
    if c < 0:
        raise VmoeError(c, "vmoe_problem_capacity")
    return c


def vmoe_expert_bwd_workspace_size(p: VmoeProblem) -> int:
    return int(library().vmoe_expert_bwd_workspace_size(ctypes.byref(p)))


def vmoe_expert_bwd_min_workspace_size(p: VmoeProblem) -> int:
    return int(library().vmoe_expert_bwd_min_workspace_size(ctypes.byref(p)))


def vmoe_route(p, x, w_router, logit_bias, logits, expert_idx, gate, slot, load, stream=None):
    _check(library().vmoe_route(ctypes.byref(p), _ptr(x), _ptr(w_router), _ptr(logit_bias),
                                _ptr(logits), _ptr(expert_idx), _ptr(gate), _ptr(slot),
                                _ptr(load), _stream(stream)), "vmoe_route")


def vmoe_dispatch(p, src, weight, expert_idx, slot, load, dst, stream=None):
    _check(library().vmoe_dispatch(ctypes.byref(p), _ptr(src), _ptr(weight), _ptr(expert_idx),
                                   _ptr(slot), _ptr(load), _ptr(dst), _stream(stream)),
           "vmoe_dispatch")


def vmoe_expert_fwd(p, xe, w1, w2, load, h, a, ye, stream=None):
    _check(library().vmoe_expert_fwd(ctypes.byref(p), _ptr(xe), _ptr(w1), _ptr(w2), _ptr(load),
                                     _ptr(h), _ptr(a), _ptr(ye), _stream(stream)),
           "vmoe_expert_fwd")


def vmoe_expert_bwd(p, xe, h, a, w1, w2, dye, load, dxe, dw1, dw2, workspace, workspace_bytes=None,
                    stream=None):
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    _check(library().vmoe_expert_bwd(ctypes.byref(p), _ptr(xe), _ptr(h), _ptr(a), _ptr(w1),
                                     _ptr(w2), _ptr(dye), _ptr(load), _ptr(dxe), _ptr(dw1),
                                     _ptr(dw2), _ptr(workspace), int(workspace_bytes),
                                     _stream(stream)), "vmoe_expert_bwd")


VMOE_STATIC_SCRATCH_BYTES = 64 << 20


def vmoe_expert_bwd_static_scratch(p, xe, h, a, w1, w2, dye, load, dxe, dw1, dw2, stream=None):
    """vmoe_expert_bwd with its dH scratch in the library's own 64 MiB device
    array, for callers that cannot allocate device memory (see include/vmoe.h)."""
    _check(library().vmoe_expert_bwd_static_scratch(
        ctypes.byref(p), _ptr(xe), _ptr(h), _ptr(a), _ptr(w1), _ptr(w2), _ptr(dye), _ptr(load),
        _ptr(dxe), _ptr(dw1), _ptr(dw2), _stream(stream)), "vmoe_expert_bwd_static_scratch")


def vmoe_combine(p, src, weight, expert_idx, slot, dst, stream=None):
    _check(library().vmoe_combine(ctypes.byref(p), _ptr(src), _ptr(weight), _ptr(expert_idx),
                                  _ptr(slot), _ptr(dst), _stream(stream)), "vmoe_combine")


def vmoe_attn_expert_fwd(p, heads, xe, wqkv, wo, load, qkv, o, lse, ye, stream=None):
    """Attention experts, forward (see include/vmoe.h)."""
    _check(library().vmoe_attn_expert_fwd(ctypes.byref(p), int(heads), _ptr(xe), _ptr(wqkv), _ptr(wo),
                                          _ptr(load), _ptr(qkv), _ptr(o), _ptr(lse), _ptr(ye),
                                          _stream(stream)), "vmoe_attn_expert_fwd")


def vmoe_attn_expert_bwd_workspace_size(p, heads) -> int:
    return int(library().vmoe_attn_expert_bwd_workspace_size(ctypes.byref(p), int(heads)))


def vmoe_attn_expert_bwd(p, heads, xe, qkv, o, lse, wqkv, wo, dye, load, dxe, dwqkv, dwo, workspace,
                         workspace_bytes=None, stream=None):
    """Attention experts, backward (see include/vmoe.h)."""
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    _check(library().vmoe_attn_expert_bwd(
        ctypes.byref(p), int(heads), _ptr(xe), _ptr(qkv), _ptr(o), _ptr(lse), _ptr(wqkv), _ptr(wo),
        _ptr(dye), _ptr(load), _ptr(dxe), _ptr(dwqkv), _ptr(dwo), _ptr(workspace), int(workspace_bytes),
        _stream(stream)), "vmoe_attn_expert_bwd")


def vmoe_router_bwd(p, x, w_router, logits, expert_idx, gate, slot, dy, ye, dgate, dlogits,
                    dw_router, dbias=None, dx=None, stream=None):
    """Router backward with the routing fixed; dx (if given) is updated in place."""
    _check(library().vmoe_router_bwd(
        ctypes.byref(p), _ptr(x), _ptr(w_router), _ptr(logits), _ptr(expert_idx), _ptr(gate),
        _ptr(slot), _ptr(dy), _ptr(ye), _ptr(dgate), _ptr(dlogits), _ptr(dw_router), _ptr(dbias),
        _ptr(dx), _stream(stream)), "vmoe_router_bwd")


def vmoe_plan_slices(weight, lifespan, capacity: int, eta: float = 0.0, budget: float = 0.0):
    """Host-side slice planner (see include/vmoe.h); returns a list of slices,
    each a list of item indices."""
    import numpy as np
    w = np.ascontiguousarray(weight, dtype=np.int64)
    r = np.ascontiguousarray(lifespan, dtype=np.float64)
    n = int(w.size)
    order = np.zeros(max(n, 1), dtype=np.int32)
    start = np.zeros(n + 2, dtype=np.int32)
    ns = library().vmoe_plan_slices(n, w.ctypes.data, r.ctypes.data, int(capacity), float(eta),
                                    float(budget), order.ctypes.data, start.ctypes.data)
    _check(ns if ns < 0 else 0, "vmoe_plan_slices")
    return [order[start[s]:start[s + 1]].tolist() for s in range(ns)]


def vmoe_plan_shares(work, minimum, saturation, budget: int):
    """Host-side fill-clamp-refill allocation (see include/vmoe.h); returns the
    list of whole-unit shares."""
    import numpy as np
    w = np.ascontiguousarray(work, dtype=np.float64)
    mn = np.ascontiguousarray(minimum, dtype=np.int32)
    sat = np.ascontiguousarray(saturation, dtype=np.int32)
    n = int(w.size)
    out = np.zeros(max(n, 1), dtype=np.int32)
    r = library().vmoe_plan_shares(n, w.ctypes.data, mn.ctypes.data, sat.ctypes.data, int(budget),
                                   out.ctypes.data)
    _check(r if r < 0 else 0, "vmoe_plan_shares")
    return out[:n].tolist()


def vmoe_device_status(reset: bool = False) -> int:
    return library().vmoe_device_status(1 if reset else 0)


def vmoe_selftest_bounded_wait(limit_ns: int, stream=None):
    _check(library().vmoe_selftest_bounded_wait(int(limit_ns), _stream(stream)),
           "vmoe_selftest_bounded_wait")


def vmoe_trace_enable(max_records: int):
    _check(library().vmoe_trace_enable(int(max_records)), "vmoe_trace_enable")


def vmoe_trace_disable() -> int:
    return library().vmoe_trace_disable()


def vmoe_trace_get(i: int):
    name = ctypes.c_char_p()
    ms = ctypes.c_float()
    _check(library().vmoe_trace_get(int(i), ctypes.byref(name), ctypes.byref(ms)),
           "vmoe_trace_get")
    return name.value.decode(), ms.value


from .step import Buffers, HostPipeline, StepRunner  # noqa: E402  (needs the names above)
