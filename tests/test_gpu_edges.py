"""Edge cases of the CUDA path against the fp64 oracle, and the device failure path.

Limits and degenerate shapes: the largest expert count (E = 256, several router
passes), the largest top-k (k = 8), every expert chosen (k = E), a capacity of one
slot, a single token per task, 1024 (task, expert) groups with most of them empty,
and an odd-sized fp32 problem.  Each runs the whole step through the C ABI and is
checked stage by stage like the main parity tests.  The last test makes a device
wait run out on purpose (a barrier nothing signals, 20 ms limit) and checks that the
library reports it and the context stays usable.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads
from gpu_helpers import GATE_RTOL, np64, problem_of, rel_err, run_step, to_dev
from test_gpu_parity import _compare_step

pytestmark = pytest.mark.gpu

Config = workloads.Config

EDGES = {
    "k8_of_256_experts": Config("k8_of_256_experts", 50, T=2, N=300, d=128, f=128, E=256, k=8,
                                cf=2.0, dtype="bf16", bias="drift"),
    "capacity_one": Config("capacity_one", 51, T=2, N=50, d=128, f=256, E=4, k=2, cf=1.0,
                           dtype="bf16", capacity=1),
    "one_token": Config("one_token", 52, T=3, N=1, d=256, f=128, E=4, k=2, cf=1.0, dtype="bf16"),
    "k_equals_E": Config("k_equals_E", 53, T=2, N=64, d=128, f=256, E=4, k=4, cf=1.0,
                         dtype="bf16"),
    "1024_groups": Config("1024_groups", 54, T=4, N=256, d=128, f=128, E=256, k=1, cf=1.0,
                          dtype="bf16", bias="zipf"),
    "fp32_odd": Config("fp32_odd", 55, T=2, N=37, d=24, f=20, E=3, k=2, cf=1.0, dtype="f32"),
}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()


@pytest.mark.parametrize("name", list(EDGES))
def test_edge_case_step(name):
    cfg = EDGES[name]
    inp = workloads.make_inputs(cfg)
    p, b = run_step(cfg, to_dev(inp))
    _compare_step(cfg, inp, b, cfg.flags)


def test_nan_logits_keep_indices_in_range():
    """A NaN logit is never chosen (treated as -inf); indices and slots stay valid."""
    import paper_2608_16188_gb300 as vm
    T, N, E, k = 2, 100, 8, 2
    g = torch.Generator().manual_seed(9)
    lg = torch.randn((T, N, E), generator=g)
    lg[0, :10, 0] = float("nan")
    lg[1, 5, :] = float("nan")  # a token whose logits are all NaN
    p = vm.problem(T, N, 64, 128, E, k, 1.0, "bf16", flags=vm.VMOE_LOGITS_IN)
    dl = lg.cuda()
    idx = torch.empty(T, N, k, dtype=torch.int32, device="cuda")
    gate = torch.empty(T, N, k, dtype=torch.float32, device="cuda")
    slot = torch.empty_like(idx)
    load = torch.empty(T, E, dtype=torch.int32, device="cuda")
    vm.vmoe_route(p, None, None, None, dl, idx, gate, slot, load)
    torch.cuda.synchronize()
    i = idx.cpu()
    assert int(i.min()) >= 0 and int(i.max()) < E
    assert torch.all(i[0, :10] != 0)  # the NaN expert never wins while finite logits exist
    assert torch.equal(i[1, 5], torch.tensor([0, 1], dtype=torch.int32))  # all -inf: lowest indices
    C = vm.vmoe_problem_capacity(p)
    assert int(load.max()) <= C and int(slot.max()) < C
    # the rest of the routing still matches the oracle on the rows without NaN
    clean = torch.where(torch.isnan(lg), torch.full_like(lg, -np.inf), lg)
    ridx, _, rslot, rload = oracle.route(clean.numpy(), k, C)
    assert np.array_equal(i.numpy(), ridx)
    assert np.array_equal(slot.cpu().numpy(), rslot)
    assert np.array_equal(load.cpu().numpy(), rload)
    assert vm.vmoe_device_status() == 0


def test_bounded_wait_reports_timeout_and_context_survives():
    import paper_2608_16188_gb300 as vm
    assert vm.vmoe_device_status(reset=True) == 0
    vm.vmoe_selftest_bounded_wait(20_000_000)  # 20 ms, nothing will ever signal the barrier
    torch.cuda.synchronize()
    assert vm.vmoe_device_status(reset=True) == vm.VMOE_ERR_DEVICE_TIMEOUT
    assert vm.vmoe_device_status() == 0
    with pytest.raises(vm.VmoeError):
        vm.vmoe_selftest_bounded_wait(0)
    # the context is intact: a full step still runs and matches the oracle
    cfg = EDGES["k_equals_E"]
    inp = workloads.make_inputs(cfg)
    p, b = run_step(cfg, to_dev(inp))
    _compare_step(cfg, inp, b, cfg.flags)
    assert vm.vmoe_device_status() == 0
