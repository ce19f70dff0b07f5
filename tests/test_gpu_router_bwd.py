"""Parity of the router backward (vmoe_router_bwd) with the fp64 oracle, on a GB300.

The router backward completes the adaptation gradient of Section 3.1 with the
gating network's share: dgate, dlogits, dW_r, dbias and the router's term of dX,
with the routing of the forward held fixed.  Stage-wise, as for the other calls:
the oracle gets the logits, indices, gates, slots and expert outputs Ye that the
GPU produced, and dX is compared against the GPU's dX before the call plus the
oracle's router term.  dgate, dlogits, dW_r and dbias are fp32 outputs with no
bf16 rounding of their own (bf16 problems give them bf16 inputs, which the
oracle reads exactly), so every problem holds them to the fp32 bar, 1e-5 of
their RMS; dX is a bf16 output in bf16 problems, held to the usual 2e-2.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads
from gpu_helpers import (BF16_RMS_TOL, BF16_TOL, F32_RMS_TOL, F32_TOL, np64, problem_of, rel_err,
                         rms_err, to_dev)

pytestmark = pytest.mark.gpu

Config = workloads.Config

CASES = {
    "tiny_fp32": workloads.CONFIGS["tiny_fp32"],
    # ragged N (300 = 4 x 64 + 44) and d (200 = 3 x 64 + 8); two choices, drops
    "fp32_ragged": Config("fp32_ragged", 60, T=2, N=300, d=200, f=96, E=6, k=2, cf=1.0,
                          dtype="f32", bias="drift"),
    "bf16_drops_drift": Config("bf16_drops_drift", 61, T=3, N=200, d=384, f=640, E=8, k=2,
                               cf=1.0, dtype="bf16", bias="drift"),
    # V-MoE gating without renormalisation: dlogits over all E experts
    "bf16_norenorm": Config("bf16_norenorm", 62, T=2, N=160, d=128, f=384, E=4, k=2, cf=1.5,
                            dtype="bf16", flags=2),
    # top-1, most assignments dropped, most groups empty
    "bf16_skew_top1": Config("bf16_skew_top1", 63, T=2, N=100, d=128, f=256, E=16, k=1, cf=1.0,
                             dtype="bf16", bias="zipf"),
    # E = 96 spans two expert tiles of dW_r with a ragged tail; k = 3
    "bf16_e96_k3": Config("bf16_e96_k3", 64, T=2, N=130, d=256, f=128, E=96, k=3, cf=2.0,
                          dtype="bf16"),
    # the largest expert count and top-k
    "k8_of_256_experts": Config("k8_of_256_experts", 65, T=2, N=300, d=128, f=128, E=256, k=8,
                                cf=2.0, dtype="bf16", bias="drift"),
    "k8_norenorm": Config("k8_norenorm", 66, T=1, N=90, d=128, f=128, E=64, k=8, cf=1.0,
                          dtype="bf16", flags=2),
    "capacity_one": Config("capacity_one", 67, T=2, N=50, d=128, f=256, E=4, k=2, cf=1.0,
                           dtype="bf16", capacity=1),
    "one_token": Config("one_token", 68, T=3, N=1, d=256, f=128, E=4, k=2, cf=1.0,
                        dtype="bf16"),
    # E = 32 takes the tcgen05 dW_r kernel: N = 131 gives the two ranks of a
    # cluster 65 and 66 tokens (a full and a partial k-block each), d = 256 two slices
    "bf16_e32_ragged": Config("bf16_e32_ragged", 69, T=3, N=131, d=256, f=128, E=32, k=2, cf=1.25,
                              dtype="bf16", bias="drift"),
    # one token: the first rank of every cluster has no tokens at all
    "bf16_e32_one_token": Config("bf16_e32_one_token", 70, T=2, N=1, d=128, f=128, E=32, k=2,
                                 cf=1.0, dtype="bf16"),
}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()


def _forward_backward(cfg):
    """Runs a1..a12 on the GPU; returns (problem, runner, inputs on CPU, dX before the call)."""
    import paper_2608_16188_gb300 as vm
    inp = workloads.make_inputs(cfg)
    p = problem_of(cfg)
    r = vm.StepRunner(p, to_dev(inp))
    r.step()
    torch.cuda.synchronize()
    return p, r, inp, r.b.dx.clone()


def _check(cfg, r, inp, dx_before):
    b = r.b
    T, N = cfg.T, cfg.N
    ref = oracle.router_bwd(inp["x"], inp["w_router"], b.logits, b.idx.cpu(), b.gate, b.slot.cpu(),
                            inp["dy"], b.ye, cfg.flags)
    r_dgate, r_dl, r_dw, r_db, r_dx = ref
    f32 = cfg.dtype == "f32"
    tol, rtol = F32_TOL, F32_RMS_TOL  # fp32 outputs in every problem
    xtol, xrtol = (F32_TOL, F32_RMS_TOL) if f32 else (BF16_TOL, BF16_RMS_TOL)
    checks = {  # name: (gpu, reference, number of separate outputs, tolerances)
        "dgate": (b.dgate, r_dgate, T, tol, rtol),
        "dlogits": (b.dlogits, r_dl, T, tol, rtol),
        "dw_router": (b.dw_router, r_dw, T, tol, rtol),
        "dbias": (b.dbias, r_db, T, tol, rtol),
        "dx": (b.dx, np64(dx_before) + r_dx, T * N, xtol, xrtol),
    }
    errs, bad = {}, {}
    for n, (g, rr, groups, t1, t2) in checks.items():
        errs[n] = (rel_err(g, rr, None, groups), rms_err(g, rr))
        if not (errs[n][0] <= t1 and errs[n][1] <= t2):
            bad[n] = errs[n]
    print(cfg.name, {n: (float("%.3g" % v[0]), float("%.3g" % v[1])) for n, v in errs.items()})
    assert not bad, (cfg.name, bad)
    # dropped choices have exactly zero dgate; unchosen experts exactly zero dlogits
    slot = b.slot.cpu().numpy()
    assert np.all(b.dgate.cpu().numpy()[slot < 0] == 0)
    if not (cfg.flags & 2):
        chosen = np.zeros((T, N, cfg.E), bool)
        np.put_along_axis(chosen, b.idx.cpu().numpy().astype(np.int64), True, axis=2)
        assert np.all(b.dlogits.cpu().numpy()[~chosen] == 0)
    return errs


@pytest.mark.parametrize("name", list(CASES))
def test_router_bwd_parity(name):
    cfg = CASES[name]
    p, r, inp, dx0 = _forward_backward(cfg)
    r.router_backward()
    torch.cuda.synchronize()
    _check(cfg, r, inp, dx0)


@pytest.mark.parametrize("name", ["vitb_t17", "skew_t8"])
def test_router_bwd_fullsize(name):
    """Every output at full size, in the step configuration the benchmark times."""
    cfg = workloads.CONFIGS[name]
    p, r, inp, dx0 = _forward_backward(cfg)
    r.router_backward()
    torch.cuda.synchronize()
    _check(cfg, r, inp, dx0)


def test_router_bwd_optional_outputs_and_determinism():
    """dbias and dx may be NULL (dx then stays untouched); two runs agree bitwise;
    the softmax-backward identity sum_e dlogits = 0 holds per token."""
    import paper_2608_16188_gb300 as vm
    cfg = CASES["bf16_drops_drift"]
    p, r, inp, dx0 = _forward_backward(cfg)
    b, i = r.b, r.inp
    outs = []
    for _ in range(2):
        dg = torch.full_like(b.dgate, float("nan"))
        dl = torch.full_like(b.dlogits, float("nan"))
        dw = torch.full_like(b.dw_router, float("nan"))
        vm.vmoe_router_bwd(p, i["x"], None, None, b.idx, b.gate, b.slot, i["dy"], b.ye, dg, dl,
                           dw, None, None)
        torch.cuda.synchronize()
        outs.append((dg, dl, dw))
    assert torch.equal(b.dx, dx0)
    for a, c in zip(outs[0], outs[1]):
        assert torch.equal(a, c) and not torch.isnan(a).any()
    # sum_j gate_j (dgate_j - s) = 0 since the renormalised gates sum to 1; fp32
    # rounding leaves a residue of a few ulp of sum_j gate_j (|dgate_j| + |s|)
    g, dgd = b.gate.double(), outs[0][0].double()
    s_tok = (g * dgd).sum(dim=2, keepdim=True)
    scale = (g * (dgd.abs() + s_tok.abs())).sum(dim=2) + 1e-30
    resid = outs[0][1].double().sum(dim=2).abs() / scale
    assert float(resid.max()) < 1e-5
    # the full call agrees bitwise with the one without the optional outputs
    r.router_backward()
    torch.cuda.synchronize()
    assert torch.equal(b.dgate, outs[0][0]) and torch.equal(b.dlogits, outs[0][1])
    assert torch.equal(b.dw_router, outs[0][2])


def test_router_bwd_argument_errors():
    import paper_2608_16188_gb300 as vm
    cfg = CASES["bf16_norenorm"]
    p, r, inp, dx0 = _forward_backward(cfg)
    b, i = r.b, r.inp
    args = [p, i["x"], i["w_router"], b.logits, b.idx, b.gate, b.slot, i["dy"], b.ye, b.dgate,
            b.dlogits, b.dw_router, b.dbias, b.dx]
    bad_logits = list(args)
    bad_logits[3] = None  # VMOE_NO_RENORM reads the logits
    with pytest.raises(vm.VmoeError) as e:
        vm.vmoe_router_bwd(*bad_logits)
    assert e.value.status == vm.VMOE_ERR_INVALID
    bad_w = list(args)
    bad_w[2] = None  # dx given without W_r
    with pytest.raises(vm.VmoeError) as e:
        vm.vmoe_router_bwd(*bad_w)
    assert e.value.status == vm.VMOE_ERR_INVALID
    torch.cuda.synchronize()
    assert torch.equal(b.dx, dx0)  # nothing launched
