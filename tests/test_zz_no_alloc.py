"""vmoe_expert_bwd_static_scratch: the expert backward for callers that cannot
allocate device memory (a plug-in whose host framework owns every device buffer,
or a deployment that forbids device allocation after start-up).

The entry point keeps its dH scratch in a fixed device array inside the library
instead of a caller-supplied workspace.  This file checks, through the C ABI, that
two calls in a row give the same dX, dW1 and dW2 as vmoe_expert_bwd with an
allocated workspace (within the tolerance the parity tests use), that a bf16 problem
whose dH exceeds the array runs in slices with bitwise the same results, and that
a problem that cannot fit is refused before anything is launched.  The file name
makes pytest collect it last; it also passes alone in a fresh process.
"""
import pytest
import torch

import workloads
from gpu_helpers import BF16_TOL, F32_TOL, problem_of, rel_err, to_dev

pytestmark = pytest.mark.gpu

CASES = {
    "bf16": workloads.Config("noalloc_bf16", 40, T=2, N=300, d=256, f=512, E=4, k=2, cf=1.25,
                             dtype="bf16", bias="drift"),
    "fp32": workloads.CONFIGS["tiny_fp32"],
}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()


@pytest.mark.parametrize("case", list(CASES))
def test_static_scratch_matches_workspace_backward(case):
    import paper_2608_16188_gb300 as vm
    cfg = CASES[case]
    tol = F32_TOL if cfg.dtype == "f32" else BF16_TOL
    p = problem_of(cfg)
    assert vm.vmoe_expert_bwd_workspace_size(p) <= vm.VMOE_STATIC_SCRATCH_BYTES
    inp = to_dev(workloads.make_inputs(cfg))
    run = vm.StepRunner(p, inp)
    run.step()  # forward, dispatch of dY, and the reference backward with a workspace
    b = run.b
    ref = [t.clone() for t in (b.dxe, b.dw1, b.dw2)]
    rows = (torch.arange(b.C, device="cuda")[None, None, :] < b.load[:, :, None])
    for call in range(2):  # the array keeps the previous call's contents
        outs = [torch.full_like(t, float("nan")) for t in ref]
        vm.vmoe_expert_bwd_static_scratch(p, b.xe, b.h, b.a, inp["w1"], inp["w2"], b.dye, b.load,
                                          *outs)
        torch.cuda.synchronize()
        assert vm.vmoe_device_status() == 0
        assert rel_err(outs[0][rows], ref[0][rows].double().cpu().numpy()) <= tol, call
        assert rel_err(outs[1], ref[1].double().cpu().numpy()) <= tol, call
        assert rel_err(outs[2], ref[2].double().cpu().numpy()) <= tol, call


def test_static_scratch_runs_in_slices_beyond_its_size():
    """A bf16 problem whose dH (195 MB) exceeds the 64 MiB array runs in slices of
    groups planned to fit it, with results bitwise equal to the backward with a
    full workspace."""
    import paper_2608_16188_gb300 as vm
    cfg = workloads.CONFIGS["vitb_t17"].with_(name="vitb_t4", T=4)
    p = problem_of(cfg)
    assert vm.vmoe_expert_bwd_workspace_size(p) > vm.VMOE_STATIC_SCRATCH_BYTES
    inp = to_dev(workloads.make_inputs(cfg, with_weights=False))
    inp["w1"], inp["w2"] = workloads.make_weights_fast(cfg, "cuda", seed=11)
    run = vm.StepRunner(p, inp)
    run.step()
    b = run.b
    ref = [t.clone() for t in (b.dxe, b.dw1, b.dw2)]
    rows = (torch.arange(b.C, device="cuda")[None, None, :] < b.load[:, :, None])
    outs = [torch.full_like(t, float("nan")) for t in ref]
    vm.vmoe_expert_bwd_static_scratch(p, b.xe, b.h, b.a, inp["w1"], inp["w2"], b.dye, b.load, *outs)
    torch.cuda.synchronize()
    assert vm.vmoe_device_status() == 0
    assert torch.equal(outs[0][rows], ref[0][rows])
    assert torch.equal(outs[1], ref[1]) and torch.equal(outs[2], ref[2])


def test_static_scratch_rejects_problems_beyond_its_size():
    """Refused on the host, before anything is launched: an fp32 problem whose dH
    exceeds the array (fp32 has no sliced path), and a bf16 problem one of whose
    groups alone needs more than the array."""
    import paper_2608_16188_gb300 as vm
    fake = 1 << 20  # aligned non-null pointers: the size check comes before any use
    for p in (problem_of(workloads.CONFIGS["vitb_t17"].with_(dtype="f32")),
              vm.problem(1, 8192, 128, 8192, 1, 1, 1.0, "bf16")):
        assert vm.vmoe_expert_bwd_min_workspace_size(p) > vm.VMOE_STATIC_SCRATCH_BYTES
        with pytest.raises(vm.VmoeError) as ei:
            vm.vmoe_expert_bwd_static_scratch(p, *([fake] * 10))
        assert ei.value.status == vm.VMOE_ERR_UNSUPPORTED
