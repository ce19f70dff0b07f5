"""fp64 CPU oracle for one adaptation step of T multiplexed V-MoE expert layers.

TEST INFRASTRUCTURE, NOT PRODUCT CODE.  Only ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline / reference legs of ``bench.py`` may import this package.  It
shares no code with the CUDA library in ``paper_2608_16188_gb300`` and neither
imports the other.

The arithmetic lives in ``vmoe_oracle.c`` (plain C, double precision, each
function citing the paper section it follows); this module only compiles it with
gcc on first use and marshals numpy arrays.  Inputs are widened to float64 before
the call, so bf16 / fp32 values enter the oracle exactly.

Parity status (what pins each function, see ``tests/test_oracle_pins.py``):
  capacity        closed-form values and clamps
  router_logits   numpy matmul on random inputs
  route           brute-force k-permutation enumeration, rank-by-sort slot rule,
                  hand-derived golden fixture, invariants (softmax sums, shifts)
  dispatch/combine  identity-expert invariant, brute-force scatter on tiny inputs
  expert_fwd/bwd  torch float64 autograd on the dense special case (E=1, k=1,
                  C=N) and central finite differences of the composed forward
  router_bwd      torch float64 autograd of the whole routed layer (routing fixed,
                  gates differentiable) and central finite differences
  plan_slices     (planner.py, plain Python) brute-force subset enumeration, a
                  textbook knapsack instance, equal-weight closed forms
  attention_expert_fwd / _bwd  (attention.py, numpy) torch float64 autograd
                  through scaled_dot_product_attention, central finite
                  differences, one-token and zero-query closed forms,
                  permutation equivariance, padding rows and empty groups
  fill_clamp_refill / integer_shares  (planner.py) the closed form
                  min(sat, min + lambda w) with lambda found by bisection, a
                  hand-worked example (tests/golden/shares_example.json), sums
                  and bounds, rounding within one unit
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

from .planner import plan_slices  # noqa: F401  (cross-task slice planner, Section 3.2.1)
from .planner import fill_clamp_refill, integer_shares  # noqa: F401  (Section 3.2.2)

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "vmoe_oracle.c")
_LIB = os.path.join(_HERE, "_liboracle.so")
_lock = threading.Lock()
_lib = None

FLAG_NO_RENORM = 2
FLAG_GELU_TANH = 4

_DP = ctypes.POINTER(ctypes.c_double)
_IP = ctypes.POINTER(ctypes.c_int32)


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2 -fopenmp) into ``oracle/_liboracle.so``."""
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    tmp = _LIB + ".%d.tmp" % os.getpid()
    cmd = ["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c11", "-D_DEFAULT_SOURCE",
           "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            lib.oracle_capacity.restype = ctypes.c_int
            lib.oracle_capacity.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                            ctypes.c_double, ctypes.c_int]
            lib.oracle_num_threads.restype = ctypes.c_int
            for name in ("oracle_router_logits", "oracle_route", "oracle_dispatch",
                         "oracle_expert_fwd", "oracle_combine", "oracle_expert_bwd",
                         "oracle_router_bwd"):
                getattr(lib, name).restype = None
            _lib = lib
    return _lib


def _d(a):
    """Contiguous float64 copy-or-view and its pointer."""
    a = np.ascontiguousarray(np.asarray(a, dtype=np.float64))
    return a, a.ctypes.data_as(_DP)


def _i(a):
    a = np.ascontiguousarray(np.asarray(a, dtype=np.int32))
    return a, a.ctypes.data_as(_IP)


def _as_np64(t):
    """torch tensor (any float dtype, any device) or array -> float64 numpy."""
    try:
        import torch
        if isinstance(t, torch.Tensor):
            return t.detach().to("cpu", torch.float64).numpy()
    except ImportError:  # pragma: no cover
        pass
    return np.asarray(t, dtype=np.float64)


def num_threads() -> int:
    return int(_load().oracle_num_threads())


def capacity(N: int, E: int, k: int, capacity_factor: float, capacity_override: int = 0) -> int:
    return int(_load().oracle_capacity(int(N), int(E), int(k), float(capacity_factor),
                                       int(capacity_override)))


def router_logits(x, w_router, bias=None):
    """x [T,N,d], w_router [T,d,E], bias [T,E] or None -> logits [T,N,E] float64."""
    x, px = _d(_as_np64(x))
    w, pw = _d(_as_np64(w_router))
    T, N, d = x.shape
    E = w.shape[2]
    pb = None
    if bias is not None:
        b, pb = _d(_as_np64(bias))
    out = np.empty((T, N, E), np.float64)
    _load().oracle_router_logits(T, N, d, E, px, pw, pb, out.ctypes.data_as(_DP))
    return out


def route(logits, k: int, C: int, flags: int = 0):
    """logits [T,N,E] -> (idx [T,N,k] int32, gate [T,N,k] f64, slot [T,N,k] int32, load [T,E] int32)."""
    lg, pl = _d(_as_np64(logits))
    T, N, E = lg.shape
    idx = np.empty((T, N, k), np.int32)
    gate = np.empty((T, N, k), np.float64)
    slot = np.empty((T, N, k), np.int32)
    load = np.empty((T, E), np.int32)
    _load().oracle_route(T, N, E, k, C, flags, pl, idx.ctypes.data_as(_IP),
                         gate.ctypes.data_as(_DP), slot.ctypes.data_as(_IP),
                         load.ctypes.data_as(_IP))
    return idx, gate, slot, load


def dispatch(src, weight, idx, slot, E: int, C: int):
    """src [T,N,d], weight [T,N,k] or None -> dst [T,E,C,d] float64 (padding rows zero)."""
    s, ps = _d(_as_np64(src))
    T, N, d = s.shape
    ix, pix = _i(idx)
    sl, psl = _i(slot)
    k = ix.shape[2]
    pw = None
    if weight is not None:
        w, pw = _d(_as_np64(weight))
    out = np.empty((T, E, C, d), np.float64)
    _load().oracle_dispatch(T, N, d, E, k, C, ps, pw, pix, psl, out.ctypes.data_as(_DP))
    return out


def combine(src, weight, idx, slot, N: int):
    """src [T,E,C,d], weight [T,N,k] or None -> dst [T,N,d] float64."""
    s, ps = _d(_as_np64(src))
    T, E, C, d = s.shape
    ix, pix = _i(idx)
    sl, psl = _i(slot)
    k = ix.shape[2]
    pw = None
    if weight is not None:
        w, pw = _d(_as_np64(weight))
    out = np.empty((T, N, d), np.float64)
    _load().oracle_combine(T, N, d, E, k, C, ps, pw, pix, psl, out.ctypes.data_as(_DP))
    return out


def expert_fwd(xe, w1, w2, load, flags: int = 0):
    """xe [G,C,d], w1 [G,d,f], w2 [G,f,d], load [G] -> (h, a [G,C,f], ye [G,C,d]) float64.

    Leading dims may be [T,E,...]; they are flattened to G = T*E and restored.
    """
    xe = _as_np64(xe)
    lead = xe.shape[:-2]
    C, d = xe.shape[-2:]
    f = np.shape(w1)[-1]
    x, px = _d(xe.reshape(-1, C, d))
    G = x.shape[0]
    a1, p1 = _d(_as_np64(w1).reshape(G, d, f))
    a2, p2 = _d(_as_np64(w2).reshape(G, f, d))
    ld, pld = _i(np.asarray(load).reshape(G))
    h = np.empty((G, C, f), np.float64)
    a = np.empty((G, C, f), np.float64)
    ye = np.empty((G, C, d), np.float64)
    _load().oracle_expert_fwd(G, C, d, f, flags, px, p1, p2, pld, h.ctypes.data_as(_DP),
                              a.ctypes.data_as(_DP), ye.ctypes.data_as(_DP))
    return (h.reshape(*lead, C, f), a.reshape(*lead, C, f), ye.reshape(*lead, C, d))


def expert_bwd(xe, h, a, w1, w2, dye, load, flags: int = 0):
    """-> (dh [G,C,f], dxe [G,C,d], dw1 [G,d,f], dw2 [G,f,d]) float64, leading dims kept."""
    xe = _as_np64(xe)
    lead = xe.shape[:-2]
    C, d = xe.shape[-2:]
    f = np.shape(w1)[-1]
    x, px = _d(xe.reshape(-1, C, d))
    G = x.shape[0]
    hh, ph = _d(_as_np64(h).reshape(G, C, f))
    aa, pa = _d(_as_np64(a).reshape(G, C, f))
    a1, p1 = _d(_as_np64(w1).reshape(G, d, f))
    a2, p2 = _d(_as_np64(w2).reshape(G, f, d))
    dy, pdy = _d(_as_np64(dye).reshape(G, C, d))
    ld, pld = _i(np.asarray(load).reshape(G))
    dh = np.empty((G, C, f), np.float64)
    dxe = np.empty((G, C, d), np.float64)
    dw1 = np.empty((G, d, f), np.float64)
    dw2 = np.empty((G, f, d), np.float64)
    _load().oracle_expert_bwd(G, C, d, f, flags, px, ph, pa, p1, p2, pdy, pld,
                              dh.ctypes.data_as(_DP), dxe.ctypes.data_as(_DP),
                              dw1.ctypes.data_as(_DP), dw2.ctypes.data_as(_DP))
    return (dh.reshape(*lead, C, f), dxe.reshape(*lead, C, d),
            dw1.reshape(*lead, d, f), dw2.reshape(*lead, f, d))


def router_bwd(x, w_router, logits, idx, gate, slot, dy, ye, flags: int = 0):
    """Router backward with routing fixed.  ye [T,E,C,d] (or [G,C,d]).

    Returns (dgate [T,N,k], dlogits [T,N,E], dw_router [T,d,E], dbias [T,E],
    dx_router [T,N,d]) in float64.
    """
    xx, px = _d(_as_np64(x))
    T, N, d = xx.shape
    w, pw = _d(_as_np64(w_router))
    E = w.shape[2]
    lg, pl = _d(_as_np64(logits))
    ix, pix = _i(idx)
    k = ix.shape[2]
    g, pg = _d(_as_np64(gate))
    sl, psl = _i(slot)
    dyy, pdy = _d(_as_np64(dy))
    y_e = _as_np64(ye)
    C = y_e.shape[-2]
    yy, pye = _d(y_e.reshape(T, E, C, d))
    dgate = np.empty((T, N, k), np.float64)
    dl = np.empty((T, N, E), np.float64)
    dw = np.empty((T, d, E), np.float64)
    db = np.empty((T, E), np.float64)
    dxr = np.empty((T, N, d), np.float64)
    _load().oracle_router_bwd(T, N, d, E, k, C, flags, px, pw, pl, pix, pg, psl, pdy, pye,
                              dgate.ctypes.data_as(_DP), dl.ctypes.data_as(_DP),
                              dw.ctypes.data_as(_DP), db.ctypes.data_as(_DP),
                              dxr.ctypes.data_as(_DP))
    return dgate, dl, dw, db, dxr


def step(x, w_router, bias, w1, w2, dy, k: int, C: int, flags: int = 0, logits=None):
    """One full adaptation step a1..a12 in fp64.

    If ``logits`` is given (parity mode) routing uses those values instead of the
    oracle's own fp64 router logits, so routing can be compared bit-exactly with a
    device run that produced them.  Returns a dict of float64 / int32 arrays.
    """
    T, N, d = np.shape(x)
    E = np.shape(w_router)[2]
    own_logits = router_logits(x, w_router, bias)
    lg = own_logits if logits is None else _as_np64(logits)
    idx, gate, slot, load = route(lg, k, C, flags)
    xe = dispatch(x, None, idx, slot, E, C)
    h, a, ye = expert_fwd(xe, w1, w2, load, flags)
    y = combine(ye, gate, idx, slot, N)
    dye = dispatch(dy, gate, idx, slot, E, C)
    dh, dxe, dw1, dw2 = expert_bwd(xe, h, a, w1, w2, dye, load, flags)
    dx = combine(dxe, None, idx, slot, N)
    return dict(logits=own_logits, idx=idx, gate=gate, slot=slot, load=load, xe=xe, h=h, a=a,
                ye=ye, y=y, dye=dye, dh=dh, dxe=dxe, dw1=dw1, dw2=dw2, dx=dx)
