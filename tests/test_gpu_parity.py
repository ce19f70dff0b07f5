"""Parity of the CUDA path (through the C ABI) with the fp64 oracle, on a GB300.

Routing indices, slots and loads must match bit-exactly when the oracle routes
from the GPU's own fp32 logits; gates within 1e-6 relative.  Every other output
of every ABI call must be within 2e-2 (bf16) or 1e-5 (fp32) of the oracle given
the same inputs, the error of each element normalised by max(rms, |ref|) of its
own output -- a (task, expert) group's slice of an expert tensor, or one token's
row of y and dX; y and dX also end to end against the pure oracle.
The small cases span several tiles in M, N and K with ragged tails, drops, empty
groups and both N-tile widths of the tensor-core path.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads
from gpu_helpers import (BF16_RMS_TOL, BF16_TOL, F32_RMS_TOL, F32_TOL, GATE_RTOL, np64, problem_of,
                         rel_err, report, rms_err, run_step, to_dev, valid_rows)

pytestmark = pytest.mark.gpu

Config = workloads.Config

SMALL = {
    # fp32 correctness configuration (CUDA-core path)
    "tiny_fp32": workloads.CONFIGS["tiny_fp32"],
    # 2 M-tiles per group (C = 188), ragged K tail in the weight gradients, N = 512 (BN 256)
    "bf16_two_mtiles": Config("bf16_two_mtiles", 20, T=2, N=300, d=256, f=512, E=4, k=2, cf=1.25,
                              dtype="bf16"),
    # d = 384 and f = 640: N-tiles of 128 in every GEMM, drops at cf = 1.0
    "bf16_bn128_drops": Config("bf16_bn128_drops", 21, T=3, N=200, d=384, f=640, E=8, k=2, cf=1.0,
                               dtype="bf16", bias="drift"),
    # skewed load: most groups empty or tiny, top-1
    "bf16_skew_empty": Config("bf16_skew_empty", 22, T=2, N=100, d=128, f=256, E=16, k=1, cf=1.0,
                              dtype="bf16", bias="zipf"),
    # V-MoE gating (no renormalisation) and tanh GELU
    "bf16_norenorm_tanh": Config("bf16_norenorm_tanh", 23, T=2, N=160, d=128, f=384, E=4, k=2,
                                 cf=1.5, dtype="bf16", flags=2 | 4),
}


# Cases whose end-to-end dW1 / dW2 meet the per-element bar (measured: 0.007-0.019);
# the others (bf16_bn128_drops, capacity_one, k8_of_256_experts) sit at 0.021-0.031,
# the floor that bf16 A and dYe set, and are held to the aggregate bar.
E2E_DW_ELEMENTWISE = {"bf16_two_mtiles", "bf16_skew_empty", "bf16_norenorm_tanh", "k_equals_E",
                      "one_token", "1024_groups"}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()


def _compare_step(cfg, inp_cpu, b, flags):
    """Stage-wise parity of every ABI call (the oracle gets the same inputs the
    GPU call got) plus end-to-end parity of y and dX with the pure fp64 oracle."""
    tol = F32_TOL if cfg.dtype == "f32" else BF16_TOL
    rms_tol = F32_RMS_TOL if cfg.dtype == "f32" else BF16_RMS_TOL
    T, N, E, k, C, d, f = cfg.T, cfg.N, cfg.E, cfg.k, b.C, cfg.d, cfg.f
    G = T * E
    ref = oracle.step(inp_cpu["x"], inp_cpu["w_router"], inp_cpu["bias"], inp_cpu["w1"],
                      inp_cpu["w2"], inp_cpu["dy"], k, C, flags, logits=b.logits)
    # routing: bit-exact from the same fp32 logits
    assert np.array_equal(b.idx.cpu().numpy(), ref["idx"])
    assert np.array_equal(b.slot.cpu().numpy(), ref["slot"])
    assert np.array_equal(b.load.cpu().numpy(), ref["load"])
    np.testing.assert_allclose(np64(b.gate), ref["gate"], rtol=GATE_RTOL, atol=0)
    assert rel_err(b.logits, ref["logits"]) < 1e-5  # vs the fp64 router
    load = ref["load"]
    rows = valid_rows(load, C)
    gate, idx, slot = np64(b.gate), ref["idx"], ref["slot"]
    # stage inputs as the GPU saw them
    xe_g, h_g, a_g, ye_g = b.xe, b.h, b.a, b.ye
    dye_g, dxe_g = b.dye, b.dxe
    s_dye = oracle.dispatch(inp_cpu["dy"], gate, idx, slot, E, C)
    s_h, s_a, s_ye = oracle.expert_fwd(xe_g, inp_cpu["w1"], inp_cpu["w2"], load, flags)
    s_y = oracle.combine(ye_g, gate, idx, slot, N)
    _, s_dxe, s_dw1, s_dw2 = oracle.expert_bwd(xe_g, h_g, a_g, inp_cpu["w1"], inp_cpu["w2"], dye_g,
                                               load, flags)
    s_dx = oracle.combine(dxe_g, None, idx, slot, N)
    assert np.array_equal(np64(xe_g), ref["xe"])  # dispatch is a pure copy
    checks = {  # name: (gpu, reference, row mask, number of separate outputs)
        "dye": (dye_g, s_dye, None, G), "h": (h_g, s_h, rows, G), "a": (a_g, s_a, rows, G),
        "ye": (ye_g, s_ye, rows, G), "y_stage": (b.y, s_y, None, T * N),
        "dxe": (dxe_g, s_dxe, rows, G), "dw1": (b.dw1, s_dw1, None, G),
        "dw2": (b.dw2, s_dw2, None, G), "dx_stage": (b.dx, s_dx, None, T * N),
        "y_e2e": (b.y, ref["y"], None, T * N), "dx_e2e": (b.dx, ref["dx"], None, T * N),
    }
    errs = {n: report(cfg.name, n, g, r, m, gr) for n, (g, r, m, gr) in checks.items()}
    # end-to-end weight gradients: their inputs A and dYe are bf16 by the ABI, and a
    # CPU emulation of exactly those roundings reaches 0.021-0.031 per element on the
    # cases with the fewest rows per group and the largest cancellation; those are held
    # to the aggregate bar, every other case also to the per-element one
    e_dw1 = report(cfg.name, "dw1_e2e", b.dw1, ref["dw1"], None, G)
    e_dw2 = report(cfg.name, "dw2_e2e", b.dw2, ref["dw2"], None, G)
    if cfg.name in E2E_DW_ELEMENTWISE or cfg.dtype == "f32":
        errs["dw1_e2e"], errs["dw2_e2e"] = e_dw1, e_dw2
    else:
        errs["dw1_e2e_rms"], errs["dw2_e2e_rms"] = (0.0, e_dw1[1]), (0.0, e_dw2[1])
    bad = {n: v for n, v in errs.items() if not (v[0] <= tol and v[1] <= rms_tol)}
    print(cfg.name, {n: (round(v[0], 5), round(v[1], 6)) for n, v in errs.items()})
    assert not bad, (cfg.name, bad)
    # padding rows of the dispatched buffers are exactly zero
    pad = torch.from_numpy(~rows)
    assert torch.all(b.xe.cpu()[pad] == 0)
    assert torch.all(b.dye.cpu()[pad] == 0)
    # empty groups have exactly-zero weight gradients
    empty = torch.from_numpy(load == 0)
    if empty.any():
        assert torch.all(b.dw1.cpu()[empty] == 0) and torch.all(b.dw2.cpu()[empty] == 0)
    return errs


@pytest.mark.parametrize("name", list(SMALL))
def test_step_parity_small(name):
    cfg = SMALL[name]
    inp = workloads.make_inputs(cfg)
    p, b = run_step(cfg, to_dev(inp))
    _compare_step(cfg, inp, b, cfg.flags)


def test_route_ties_from_given_logits():
    """VMOE_LOGITS_IN with logits quantised to three values: many exact ties,
    which must go to the lower expert index, and a capacity that drops."""
    import paper_2608_16188_gb300 as vm
    T, N, E, k = 3, 257, 8, 3
    g = torch.Generator().manual_seed(5)
    lg = torch.randint(-1, 2, (T, N, E), generator=g).to(torch.float32) * 0.5
    p = vm.problem(T, N, 64, 128, E, k, 0.75, "bf16", flags=vm.VMOE_LOGITS_IN)
    C = vm.vmoe_problem_capacity(p)
    assert C == oracle.capacity(N, E, k, 0.75)
    dl = lg.cuda()
    idx = torch.empty(T, N, k, dtype=torch.int32, device="cuda")
    gate = torch.empty(T, N, k, dtype=torch.float32, device="cuda")
    slot = torch.empty_like(idx)
    load = torch.empty(T, E, dtype=torch.int32, device="cuda")
    vm.vmoe_route(p, None, None, None, dl, idx, gate, slot, load)
    torch.cuda.synchronize()
    ridx, rgate, rslot, rload = oracle.route(lg.numpy(), k, C)
    assert np.array_equal(idx.cpu().numpy(), ridx)
    assert np.array_equal(slot.cpu().numpy(), rslot)
    assert np.array_equal(load.cpu().numpy(), rload)
    np.testing.assert_allclose(gate.cpu().numpy(), rgate, rtol=GATE_RTOL)
    assert (rslot < 0).any()


def test_identity_experts_dispatch_combine():
    """combine(dispatch(x), gate) = x * (kept gate mass) and combine(dispatch(x))
    = x * (kept count), through the GPU kernels alone."""
    import paper_2608_16188_gb300 as vm
    cfg = SMALL["bf16_bn128_drops"]
    inp = to_dev(workloads.make_inputs(cfg, with_weights=False))
    p = problem_of(cfg)
    b = vm.Buffers(p)
    vm.vmoe_route(p, inp["x"], inp["w_router"], inp["bias"], b.logits, b.idx, b.gate, b.slot,
                  b.load)
    vm.vmoe_dispatch(p, inp["x"], None, b.idx, b.slot, b.load, b.xe)
    vm.vmoe_combine(p, b.xe, b.gate, b.idx, b.slot, b.y)
    vm.vmoe_combine(p, b.xe, None, b.idx, b.slot, b.dx)
    torch.cuda.synchronize()
    kept = (b.slot >= 0)
    mass = torch.where(kept, b.gate, torch.zeros_like(b.gate)).sum(-1, dtype=torch.float64)
    x64 = inp["x"].double()
    ref_y = (x64 * mass[..., None]).cpu().numpy()
    assert rel_err(b.y, ref_y) <= BF16_TOL and rms_err(b.y, ref_y) <= BF16_RMS_TOL
    cnt = kept.sum(-1).double()
    # unweighted sums of at most k bf16 copies of the same value are exact in fp32
    assert torch.equal(b.dx.double(), (x64 * cnt[..., None]).to(torch.bfloat16).double())
    assert (cnt < cfg.k).any()


def test_determinism_bitwise():
    cfg = SMALL["bf16_two_mtiles"]
    inp = to_dev(workloads.make_inputs(cfg))
    _, b1 = run_step(cfg, inp)
    rows = torch.from_numpy(valid_rows(b1.load, b1.C)).cuda()
    outs1 = [t.clone() for t in (b1.y, b1.dx, b1.dw1, b1.dw2, b1.h[rows], b1.gate)]
    _, b2 = run_step(cfg, inp)
    assert torch.equal(b1.load, b2.load)
    for t1, t2 in zip(outs1, (b2.y, b2.dx, b2.dw1, b2.dw2, b2.h[rows], b2.gate)):
        assert torch.equal(t1, t2)


def test_argument_errors_launch_nothing():
    import paper_2608_16188_gb300 as vm
    cfg = SMALL["bf16_two_mtiles"]
    p = problem_of(cfg)
    b = vm.Buffers(p)
    inp = to_dev(workloads.make_inputs(cfg))
    with pytest.raises(vm.VmoeError) as ei:  # workspace too small
        vm.vmoe_expert_bwd(p, b.xe, b.h, b.a, inp["w1"], inp["w2"], b.dye, b.load, b.dxe, b.dw1,
                           b.dw2, b.workspace, workspace_bytes=16)
    assert ei.value.status == vm.VMOE_ERR_INVALID
    with pytest.raises(vm.VmoeError) as ei:  # misaligned pointer
        vm.vmoe_combine(p, b.ye.data_ptr() + 2, b.gate, b.idx, b.slot, b.y)
    assert ei.value.status == vm.VMOE_ERR_INVALID
    bad = vm.problem(2, 300, 200, 512, 4, 2, 1.25, "bf16")  # d % 128 != 0 on the bf16 path
    with pytest.raises(vm.VmoeError) as ei:
        vm.vmoe_expert_fwd(bad, b.xe, inp["w1"], inp["w2"], b.load, b.h, b.a, b.ye)
    assert ei.value.status == vm.VMOE_ERR_UNSUPPORTED
    assert vm.vmoe_device_status(reset=True) == 0
