"""The expert backward under a dH budget: with a workspace smaller than
vmoe_expert_bwd_workspace_size, the groups run in slices planned by the
cross-task DP (Section 3.2.1) and dA, dX and dW1 address a compact dH buffer.
Every group's GEMMs are the same as in the unsliced run, so dXe (valid rows), dW1
and dW2 must be bitwise equal to it -- at the smallest workspace (about one group
per slice), at a third of the full size, for groups of two row tiles (the
streaming weight-gradient kernel), with empty groups, with 512 groups, and with
1024 groups whose first slice holds more than 256 entries.
"""
import pytest
import torch

import workloads
from gpu_helpers import problem_of, to_dev

pytestmark = pytest.mark.gpu

Config = workloads.Config
CASES = {
    "two_row_tiles": Config("sl_two_mtiles", 80, T=2, N=300, d=256, f=512, E=4, k=2, cf=1.25,
                            dtype="bf16"),
    "skew_empty": Config("sl_skew_empty", 81, T=2, N=100, d=128, f=256, E=16, k=1, cf=1.0,
                         dtype="bf16", bias="zipf"),
    "drift_bn128": Config("sl_bn128", 82, T=3, N=200, d=384, f=640, E=8, k=2, cf=1.0,
                          dtype="bf16", bias="drift"),
    "512_groups": Config("sl_512", 83, T=2, N=300, d=128, f=128, E=256, k=8, cf=2.0,
                         dtype="bf16", bias="drift"),
    # 1024 groups, most of them empty: the empty groups join the first slice, so
    # its plan (more than 256 entries) reaches the device in several parts
    "1024_groups_mostly_empty": Config("sl_1024", 84, T=4, N=64, d=128, f=128, E=256, k=2,
                                       cf=2.0, dtype="bf16", bias="drift"),
}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()


@pytest.mark.parametrize("name", list(CASES))
def test_sliced_backward_is_bitwise_the_full_one(name):
    import paper_2608_16188_gb300 as vm
    cfg = CASES[name]
    p = problem_of(cfg)
    inp = to_dev(workloads.make_inputs(cfg))
    run = vm.StepRunner(p, inp)
    run.step()
    torch.cuda.synchronize()
    b = run.b
    ref = [t.clone() for t in (b.dxe, b.dw1, b.dw2)]
    rows = (torch.arange(b.C, device="cuda")[None, None, :] < b.load[:, :, None])
    full = vm.vmoe_expert_bwd_workspace_size(p)
    smallest = vm.vmoe_expert_bwd_min_workspace_size(p)
    assert smallest < full
    for ws_bytes in (smallest, max(smallest, full // 3)):
        ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
        outs = [torch.full_like(t, float("nan")) for t in ref]
        vm.vmoe_expert_bwd(p, b.xe, b.h, b.a, inp["w1"], inp["w2"], b.dye, b.load, *outs, ws)
        torch.cuda.synchronize()
        assert vm.vmoe_device_status() == 0
        assert torch.equal(outs[0][rows], ref[0][rows]), ws_bytes
        assert torch.equal(outs[1], ref[1]), ws_bytes
        assert torch.equal(outs[2], ref[2]), ws_bytes


def test_sliced_backward_rejects_a_workspace_below_the_minimum():
    import paper_2608_16188_gb300 as vm
    cfg = CASES["two_row_tiles"]
    p = problem_of(cfg)
    inp = to_dev(workloads.make_inputs(cfg))
    run = vm.StepRunner(p, inp)
    run.forward()
    b = run.b
    ws = torch.empty(vm.vmoe_expert_bwd_min_workspace_size(p) - 256, dtype=torch.uint8,
                     device="cuda")
    with pytest.raises(vm.VmoeError) as e:
        vm.vmoe_expert_bwd(p, b.xe, b.h, b.a, inp["w1"], inp["w2"], b.dye, b.load, b.dxe, b.dw1,
                           b.dw2, ws)
    assert e.value.status == vm.VMOE_ERR_INVALID


def test_sliced_backward_at_the_17_task_step():
    """The benchmark's budgeted backward: the 17-task ViT-B step through the 64 MiB
    static array (8 slices) is bitwise the full-workspace backward."""
    import paper_2608_16188_gb300 as vm
    cfg = workloads.CONFIGS["vitb_t17"]
    p = problem_of(cfg)
    inp = to_dev(workloads.make_inputs(cfg, with_weights=False))
    inp["w1"], inp["w2"] = workloads.make_weights_fast(cfg, "cuda", seed=5)
    run = vm.StepRunner(p, inp)
    run.step()
    torch.cuda.synchronize()
    b = run.b
    ref = [t.clone() for t in (b.dxe, b.dw1, b.dw2)]
    rows = (torch.arange(b.C, device="cuda")[None, None, :] < b.load[:, :, None])
    outs = [torch.full_like(t, float("nan")) for t in ref]
    vm.vmoe_expert_bwd_static_scratch(p, b.xe, b.h, b.a, inp["w1"], inp["w2"], b.dye, b.load, *outs)
    torch.cuda.synchronize()
    assert vm.vmoe_device_status() == 0
    assert torch.equal(outs[0][rows], ref[0][rows])
    assert torch.equal(outs[1], ref[1]) and torch.equal(outs[2], ref[2])
