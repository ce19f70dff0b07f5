"""Group tails of the expert GEMMs against the fp64 oracle.

The grouped GEMMs load only a group's valid rows: row-mode A tiles load
16 ceil(load / 16) rows as 64-, 32- and 16-row boxes, and the resident-B
weight-gradient kernels (one SM, and SM pairs) load a group's last k-block
with a 16-, 32- or 48-row box.  Here every group of one launch has its own
load, covering each residue (0, 1, 15-17, 31-33, ..., 127, 128 rows of a
128-row capacity; up to 256 rows of a 256-row one), and every
padding row of the inputs (rows s >= load of xe, dye and the workspace) holds
NaN: padding contents must not reach any output.  The forward outputs' padding
rows must keep what the caller left there (they are not written).  The bf16
backward runs with the full workspace and with the smallest one (the sliced
path); the two must agree bitwise.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import np64, rel_err, rms_err

pytestmark = pytest.mark.gpu

LOADS = [0, 1, 15, 16, 17, 31, 32, 33, 47, 48, 49, 63, 64, 65, 79, 80, 96, 111, 112, 113, 127, 128]
# capacity 256: every residue of the last of up to four k-blocks
LOADS_256 = [0, 1, 16, 33, 64, 65, 100, 127, 128, 129, 143, 160, 191, 192, 193, 209, 224, 239, 255, 256]
# capacity 32 (the SM-pair kernel for dW2 too): one partial k-block per group
LOADS_32 = [0, 1, 2, 7, 8, 15, 16, 17, 24, 31, 32, 0, 5]
LOADS_BY_C = {32: LOADS_32, 128: LOADS, 256: LOADS_256}
SENTINEL = 7.0


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()


def _inputs(dtype, d, f, loads, C, seed=90):
    g = torch.Generator().manual_seed(seed)
    G = len(loads)
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    load = torch.tensor(loads, dtype=torch.int32).reshape(1, G)
    valid = torch.arange(C)[None, :] < load.reshape(G, 1)  # [G, C]

    def rows(width, scale):
        v = torch.randn(1, G, C, width, generator=g) * scale
        v[0][~valid] = float("nan")  # padding rows: NaN
        return v.to(tdt)

    xe = rows(d, 1.0)
    dye = rows(d, 1.0)
    w1 = (torch.randn(1, G, d, f, generator=g) / d ** 0.5).to(tdt)
    w2 = (torch.randn(1, G, f, d, generator=g) / f ** 0.5).to(tdt)
    return load, valid, xe, dye, w1, w2


def _zero_pad(t, valid):
    t = np64(t).copy()
    t[0][~valid.numpy()] = 0.0
    return t


# d 128 / f 256 and d 256 / f 384: the one-SM weight-gradient kernels (resident B,
# and streaming with 128-column tiles); d 256 / f 512 and d 512 / f 256: the
# SM-pair kernel for dW1 (C 128: two resident B tiles; C 256: one) and for dW2
# (C 32 and C 256; with C 128 dW2 streams).  With C 256 the row-mode GEMMs run on
# SM pairs (256-row tiles), with 256-column tiles (d 512 / f 256) and 128-column
# ones (d 384 / f 640, whose weight gradients stream).
@pytest.mark.parametrize("dtype,d,f,C", [("bf16", 128, 256, 128), ("bf16", 256, 384, 128),
                                         ("bf16", 256, 512, 128), ("bf16", 512, 256, 256),
                                         ("bf16", 256, 512, 32), ("bf16", 384, 640, 256),
                                         ("f32", 40, 72, 128)])
def test_group_tails(dtype, d, f, C):
    _check_tails(dtype, d, f, C, LOADS_BY_C[C])


# More groups than SM pairs at C 256, so that each pair takes several units in a
# row: the SM-pair dW1 kernel's single resident B tile is then released and
# refilled one k-block at a time while the previous unit's last row tile still
# runs (d 512: two row tiles per unit; d 256: one).
@pytest.mark.parametrize("d,f,G", [(512, 512, 96), (256, 768, 160)])
def test_wgrad_pair_units_in_a_row(d, f, G):
    rng = np.random.default_rng(7 + d)
    loads = [int(v) for v in rng.integers(0, 257, size=G)]
    loads[:4] = [0, 256, 129, 1]  # group 0 empty: its dW must be zeros
    _check_tails("bf16", d, f, 256, loads)


def _check_tails(dtype, d, f, C, loads):
    import paper_2608_16188_gb300 as vm
    G = len(loads)
    p = vm.problem(1, C, d, f, G, 1, 1.0, dtype, capacity=C)
    assert vm.vmoe_problem_capacity(p) == C
    load, valid, xe, dye, w1, w2 = _inputs(dtype, d, f, loads, C)
    dev = "cuda"
    tdt = xe.dtype
    xe_d, dye_d, w1_d, w2_d, load_d = (t.to(dev) for t in (xe, dye, w1, w2, load))
    h = torch.full((1, G, C, f), SENTINEL, dtype=tdt, device=dev)
    a = torch.full((1, G, C, f), SENTINEL, dtype=tdt, device=dev)
    ye = torch.full((1, G, C, d), SENTINEL, dtype=tdt, device=dev)
    vm.vmoe_expert_fwd(p, xe_d, w1_d, w2_d, load_d, h, a, ye)
    torch.cuda.synchronize()

    vmask = valid.numpy()[None]  # [1, G, C]
    pad = ~vmask
    for name, t in (("h", h), ("a", a), ("ye", ye)):
        assert np.all(np64(t)[pad] == SENTINEL), name + ": padding rows were written"

    tol, agg = (2e-2, 5e-3) if dtype == "bf16" else (1e-5, 2.5e-6)
    xe0, dye0 = _zero_pad(xe, valid), _zero_pad(dye, valid)
    r_h, r_a, r_ye = oracle.expert_fwd(xe0, np64(w1), np64(w2), loads)
    for name, gpu, ref in (("h", h, r_h), ("a", a, r_a), ("ye", ye, r_ye)):
        g64 = np64(gpu)
        assert np.all(np.isfinite(g64[vmask])), name
        e = rel_err(g64, ref, vmask, G)
        assert e < tol, (name, e)
        assert rms_err(g64, ref, vmask, G) < agg, name

    # backward: the oracle takes the forward outputs this call received
    h_in = _zero_pad(h.cpu(), valid)
    a_in = _zero_pad(a.cpu(), valid)
    _, r_dxe, r_dw1, r_dw2 = oracle.expert_bwd(xe0, h_in, a_in, np64(w1), np64(w2), dye0, loads)
    full = vm.vmoe_expert_bwd_workspace_size(p)
    sizes = [full] + ([vm.vmoe_expert_bwd_min_workspace_size(p)] if dtype == "bf16" else [])
    results = []
    for ws_bytes in sizes:
        ws = torch.full((ws_bytes // 4,), float("nan"), dtype=torch.float32, device=dev)
        dxe = torch.full((1, G, C, d), SENTINEL, dtype=tdt, device=dev)
        dw1 = torch.empty((1, G, d, f), dtype=tdt, device=dev)
        dw2 = torch.empty((1, G, f, d), dtype=tdt, device=dev)
        vm.vmoe_expert_bwd(p, xe_d, h, a, w1_d, w2_d, dye_d, load_d, dxe, dw1, dw2, ws, ws_bytes)
        torch.cuda.synchronize()
        assert vm.vmoe_device_status() == 0
        assert np.all(np64(dxe)[pad] == SENTINEL), "dxe: padding rows were written"
        results.append((dxe.cpu(), dw1.cpu(), dw2.cpu()))
        for name, gpu, ref, m in (("dxe", dxe, r_dxe, vmask), ("dw1", dw1, r_dw1, None),
                                  ("dw2", dw2, r_dw2, None)):
            g64 = np64(gpu)
            sel = g64[m] if m is not None else g64
            assert np.all(np.isfinite(sel)), name + ": NaN from padding rows"
            e = rel_err(g64, ref, m, G)
            assert e < tol, (name, ws_bytes, e)
            assert rms_err(g64, ref, m, G) < agg, name
        assert np.all(np64(dw1)[0, 0] == 0.0) and np.all(np64(dw2)[0, 0] == 0.0)  # load 0
    if len(results) == 2:  # the sliced run is bitwise the full one
        for x, y in zip(results[0], results[1]):
            assert torch.equal(x, y)

