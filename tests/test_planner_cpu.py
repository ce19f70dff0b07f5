"""The library's slice planner (vmoe_plan_slices, host C++) against the oracle's
(CPU only): identical slices, item for item, on random instances and on the
expert-backward instances the library plans (one item per (task, expert) group,
weight = its dH rows in units of 8, lifespan = its load)."""
import random

import numpy as np
import pytest

import oracle


@pytest.fixture(scope="module")
def vm():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_16188_gb300 as vm
    return vm


@pytest.mark.parametrize("seed", range(30))
def test_random_instances_match_oracle(vm, seed):
    rng = random.Random(100 + seed)
    n = rng.randint(0, 60)
    w = [rng.choice([0, rng.randint(1, 40)]) for _ in range(n)]
    r = [rng.choice([rng.random(), float(rng.randint(0, 5))]) for _ in range(n)]
    cap = max(w + [0]) + rng.randint(0, 80)
    eta = rng.choice([0.0, 0.02, 0.5, -0.1])
    budget = rng.choice([0.0, float(cap) * 1.5])
    got = vm.vmoe_plan_slices(w, r, cap, eta, budget)
    ref = oracle.plan_slices(w, r, cap, eta, budget if budget > 0 else None)
    assert got == ref


def test_expert_backward_instance_matches_oracle(vm):
    g = np.random.default_rng(7)
    load = np.minimum(g.poisson(72, size=544), 124)
    load[g.choice(544, 20, replace=False)] = 0
    w = [int(-(-2 * int(L) // 8)) for L in load]   # ceil(2 L / 8)
    r = [float(L) for L in load]
    cap = (64 << 20) // (3072 * 2) // 8
    got = vm.vmoe_plan_slices(w, r, cap, 0.0, 0.0)
    ref = oracle.plan_slices(w, r, cap, 0.0)
    assert got == ref
    assert sorted(i for s in got for i in s) == list(range(544))


def test_refusals(vm):
    with pytest.raises(vm.VmoeError) as e:
        vm.vmoe_plan_slices([5], [1.0], 4)
    assert e.value.status == vm.VMOE_ERR_UNSUPPORTED
    with pytest.raises(vm.VmoeError) as e:
        vm.vmoe_plan_slices([-1], [1.0], 4)
    assert e.value.status == vm.VMOE_ERR_INVALID
    assert vm.vmoe_plan_slices([], [], 4) == []


@pytest.mark.parametrize("seed", range(40))
def test_plan_shares_matches_oracle(vm, seed):
    """vmoe_plan_shares (host C++) against the oracle's fill-clamp-refill rounded to
    whole units (Section 3.2.2): identical shares on random instances, and on the
    instances the budgeted backward builds (one expert per (task, expert) group of a
    slice, work from its load, one to twelve SM pairs, 76 pairs)."""
    rng = random.Random(500 + seed)
    if seed % 2:
        n = rng.randint(0, 30)
        work = [rng.choice([0.0, rng.random() * 100, float(rng.randint(1, 9))]) for _ in range(n)]
        mn = [rng.randint(0, 3) for _ in range(n)]
        sat = [m + rng.randint(0, 10) for m in mn]
        budget = sum(mn) + rng.randint(0, 60)
    else:
        n = rng.randint(1, 76)
        loads = [rng.randint(0, 124) for _ in range(n)]
        work = [12 * (3 * 256 * 256 * 2 + L * (768 * 2 + 1024)) for L in loads]
        mn, sat, budget = [1] * n, [12] * n, 76
    got = vm.vmoe_plan_shares(work, mn, sat, budget)
    assert got == oracle.integer_shares(work, mn, sat, budget)


def test_plan_shares_errors(vm):
    with pytest.raises(vm.VmoeError) as ei:
        vm.vmoe_plan_shares([1.0, 1.0], [3, 3], [5, 5], 5)  # minima above the budget
    assert ei.value.status == vm.VMOE_ERR_UNSUPPORTED
    with pytest.raises(vm.VmoeError) as ei:
        vm.vmoe_plan_shares([1.0, float("nan")], [0, 0], [5, 5], 5)
    assert ei.value.status == vm.VMOE_ERR_INVALID
    with pytest.raises(vm.VmoeError) as ei:
        vm.vmoe_plan_shares([1.0], [3], [2], 5)  # saturation below minimum
    assert ei.value.status == vm.VMOE_ERR_INVALID
    assert vm.vmoe_plan_shares([], [], [], 7) == []
