"""Full-size parity: the 17-task ViT-B step, the Zipf-skewed step, the 6-task ViT-B
step (two row tiles per group) and the 4-task ViT-S step (128-wide column tiles), in the launch
configuration the benchmark times, checked against the fp64 oracle.

Routing is compared bit-exactly for every token of every task.  The expert FFN
(forward and all three gradients) is compared on sampled (task, expert) groups
that the oracle recomputes one by one -- the first, a middle and the last group,
the fullest group and, where present, an empty one.  Dispatch and combine are
checked on whole tasks, and at full size through the property that they move and
gate-weight rows only (the oracle's combine of the GPU's own expert outputs).  As in the small cases,
each stage's oracle gets the inputs the GPU call got, and every (task, expert)
group, or token row of y and dX, is its own output for the RMS normalisation.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads
from gpu_helpers import (BF16_RMS_TOL, BF16_TOL, np64, rel_err, report, run_step, to_dev,
                         valid_rows)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()


def _ok(name, g, r, mask=None, errs=None, groups=None, case="fullsize"):
    e = report(case, name, g, r, mask, groups)
    if errs is not None:
        errs[name] = e
    return e[0] <= BF16_TOL and e[1] <= BF16_RMS_TOL


@pytest.mark.parametrize("name", ["vitb_t17", "skew_t8", "vitb_t6", "vits_t4"])
def test_fullsize_sampled_parity(name):
    cfg = workloads.CONFIGS[name]
    inp = workloads.make_inputs(cfg)
    p, b = run_step(cfg, to_dev(inp))
    T, N, E, k, C = cfg.T, cfg.N, cfg.E, cfg.k, b.C
    load = b.load.cpu().numpy()

    # routing, all tokens of all tasks, from the GPU's fp32 logits
    ridx, rgate, rslot, rload = oracle.route(b.logits.cpu().numpy(), k, C, cfg.flags)
    assert np.array_equal(b.idx.cpu().numpy(), ridx)
    assert np.array_equal(b.slot.cpu().numpy(), rslot)
    assert np.array_equal(load, rload)
    np.testing.assert_allclose(np64(b.gate), rgate, rtol=1e-6)
    if name == "skew_t8":
        assert (rslot < 0).sum() > 0.5 * rslot.size  # the skew really overflows
    # router logits of the first and last task against the fp64 router
    for t in (0, T - 1):
        lg = oracle.router_logits(inp["x"][t:t + 1], inp["w_router"][t:t + 1],
                                  None if inp["bias"] is None else inp["bias"][t:t + 1])
        assert rel_err(b.logits[t:t + 1], lg) < 1e-5

    # dispatch of whole tasks is exact; weighted dispatch within bf16 rounding
    errs = {}
    for t in (0, T - 1):
        xe_ref = oracle.dispatch(inp["x"][t:t + 1], None, ridx[t:t + 1], rslot[t:t + 1], E, C)
        assert np.array_equal(np64(b.xe[t:t + 1]), xe_ref)
        dye_ref = oracle.dispatch(inp["dy"][t:t + 1], rgate[t:t + 1], ridx[t:t + 1],
                                  rslot[t:t + 1], E, C)
        assert _ok("dye", b.dye[t:t + 1], dye_ref, errs=errs, groups=E, case=name), errs

    # combine at full size from the GPU's own expert outputs
    y_ref = oracle.combine(b.ye, rgate, ridx, rslot, N)
    assert _ok("y", b.y, y_ref, errs=errs, groups=T * N, case=name), errs
    dx_ref = oracle.combine(b.dxe, None, ridx, rslot, N)
    assert _ok("dx", b.dx, dx_ref, errs=errs, groups=T * N, case=name), errs

    # sampled groups through the whole expert FFN, forward and backward
    G = T * E
    flat = load.reshape(-1)
    picks = {0, G // 2, G - 1, int(np.argmax(flat))}
    empty = np.flatnonzero(flat == 0)
    if empty.size:
        picks.add(int(empty[0]))
    picks = sorted(picks)
    tt = [g // E for g in picks]
    ee = [g % E for g in picks]
    xe = b.xe.view(G, C, cfg.d)[picks]
    dye = b.dye.view(G, C, cfg.d)[picks]
    w1 = inp["w1"][tt, ee]
    w2 = inp["w2"][tt, ee]
    ld = flat[picks]
    view = lambda t_, w: t_.view(G, C, w)[picks]  # noqa: E731
    # stage-wise: the oracle gets the inputs each GPU call got
    h, a, ye = oracle.expert_fwd(xe, w1, w2, ld, cfg.flags)
    _, dxe, dw1, dw2 = oracle.expert_bwd(xe, view(b.h, cfg.f), view(b.a, cfg.f), w1, w2, dye, ld,
                                         cfg.flags)
    rows = np.arange(C)[None, :] < ld[:, None]
    checks = [("h", view(b.h, cfg.f), h, rows), ("a", view(b.a, cfg.f), a, rows),
              ("ye", view(b.ye, cfg.d), ye, rows), ("dxe", view(b.dxe, cfg.d), dxe, rows),
              ("dw1", b.dw1.view(G, cfg.d, cfg.f)[picks], dw1, None),
              ("dw2", b.dw2.view(G, cfg.f, cfg.d)[picks], dw2, None)]
    ng = len(picks)
    bad = [nm for nm, g_, r_, m_ in checks if not _ok(nm, g_, r_, m_, errs, groups=ng, case=name)]
    assert not bad, (name, picks, ld.tolist(), errs)
    if empty.size:
        e0 = int(empty[0])
        assert torch.all(b.dw1.view(G, cfg.d, cfg.f)[e0] == 0)
        assert torch.all(b.dw2.view(G, cfg.f, cfg.d)[e0] == 0)
    print(name, "loads", ld.tolist(), {k_: tuple(round(v, 5) for v in e) for k_, e in errs.items()})
