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
