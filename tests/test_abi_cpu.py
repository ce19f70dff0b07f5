"""The C ABI on a machine without a GPU: the library loads, exports every function
include/vmoe.h declares, applies the capacity rule of the oracle, and rejects
invalid arguments on the host before any CUDA call (no compute is launched here).
"""
import ctypes
import os
import re

import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def vm():
    from paper_2608_16188_gb300 import _build
    _build.build()
    import paper_2608_16188_gb300 as vm
    vm.library()
    return vm


def _declared_functions():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if not fn.endswith(".h"):
            continue
        text = open(os.path.join(ROOT, "include", fn)).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names.update(re.findall(r"\b(vmoe_[a-z_0-9]+)\s*\(", text))
    return names


def test_every_declared_symbol_is_exported(vm):
    declared = _declared_functions()
    assert {"vmoe_route", "vmoe_dispatch", "vmoe_expert_fwd", "vmoe_expert_bwd",
            "vmoe_combine"} <= declared
    lib = ctypes.CDLL(vm.LIB_PATH)
    missing = [n for n in sorted(declared) if not hasattr(lib, n)]
    assert not missing
    assert set(vm.EXPORTS) == declared  # the binding covers exactly the header
    assert vm.vmoe_version() == 1


@pytest.mark.parametrize("N,E,k,cf,override", [
    (64, 4, 2, 2.0, 0), (1576, 8, 2, 1.25, 0), (3152, 32, 2, 1.25, 0), (1576, 32, 2, 1.25, 0),
    (1576, 64, 1, 1.0, 0), (100, 10, 1, 1.0, 0), (10, 4, 2, 1e-9, 0), (10, 1, 2, 8.0, 0),
    (10, 4, 2, 1.0, 7), (197, 7, 3, 0.3, 0), (1, 1, 1, 1.0, 0)])
def test_capacity_rule_matches_oracle(vm, N, E, k, cf, override):
    k = min(k, E)
    p = vm.problem(2, N, 64, 128, E, k, cf, "bf16", capacity=override)
    assert vm.vmoe_problem_capacity(p) == oracle.capacity(N, E, k, cf, override)


def test_invalid_problems_are_rejected_on_host(vm):
    lib = vm.library()
    good = dict(T=2, N=64, d_model=128, d_ff=256, E=4, k=2, capacity_factor=1.25)
    bad_cases = [
        dict(T=0), dict(N=0), dict(E=0), dict(k=0), dict(k=5), dict(k=9, E=16),
        dict(d_model=0), dict(capacity_factor=0.0), dict(capacity_factor=float("nan")),
    ]
    for bad in bad_cases:
        kw = dict(good, **bad)
        p = vm.problem(kw["T"], kw["N"], kw["d_model"], kw["d_ff"], kw["E"], kw["k"],
                       kw["capacity_factor"], "bf16")
        assert lib.vmoe_problem_capacity(ctypes.byref(p)) == vm.VMOE_ERR_INVALID, bad
        assert vm.vmoe_expert_bwd_workspace_size(p) == 0
    p = vm.problem(**good)
    p.flags = 1 << 7  # unknown flag
    assert lib.vmoe_problem_capacity(ctypes.byref(p)) == vm.VMOE_ERR_INVALID
    big = vm.problem(2, 64, 128, 256, 300, 2, 1.0)  # E > 256
    assert lib.vmoe_problem_capacity(ctypes.byref(big)) == vm.VMOE_ERR_UNSUPPORTED
    odd = vm.problem(2, 64, 100, 256, 4, 2, 1.0)  # d % 8 != 0
    assert lib.vmoe_problem_capacity(ctypes.byref(odd)) == vm.VMOE_ERR_UNSUPPORTED


def test_null_and_misaligned_pointers_are_rejected_without_cuda(vm):
    """Argument checks run before any CUDA call, so they work with no GPU at all."""
    lib = vm.library()
    p = vm.problem(2, 64, 128, 256, 4, 2, 1.25, "bf16")
    P = 1 << 20  # an aligned, never dereferenced address
    st = lib.vmoe_route(ctypes.byref(p), None, P, None, P, P, P, P, P, None)
    assert st == vm.VMOE_ERR_INVALID  # x missing without VMOE_LOGITS_IN
    st = lib.vmoe_dispatch(ctypes.byref(p), P + 4, None, P, P, P, P, None)
    assert st == vm.VMOE_ERR_INVALID  # misaligned source
    st = lib.vmoe_combine(ctypes.byref(p), P, None, P, None, P, None)
    assert st == vm.VMOE_ERR_INVALID  # slot missing
    st = lib.vmoe_expert_fwd(ctypes.byref(p), P, P, P, P, P, P, None, None)
    assert st == vm.VMOE_ERR_INVALID  # ye missing
    ws_min = vm.vmoe_expert_bwd_min_workspace_size(p)
    st = lib.vmoe_expert_bwd(ctypes.byref(p), P, P, P, P, P, P, P, P, P, P, P, ws_min - 1, None)
    assert st == vm.VMOE_ERR_INVALID  # workspace one byte short of the sliced minimum
    pf = vm.problem(2, 64, 128, 256, 4, 2, 1.25, "f32")
    ws = vm.vmoe_expert_bwd_workspace_size(pf)
    assert vm.vmoe_expert_bwd_min_workspace_size(pf) == ws  # fp32: no sliced path
    st = lib.vmoe_expert_bwd(ctypes.byref(pf), P, P, P, P, P, P, P, P, P, P, P, ws - 1, None)
    assert st == vm.VMOE_ERR_INVALID  # fp32 workspace one byte short
    odd = vm.problem(2, 64, 64, 256, 4, 2, 1.25, "bf16")  # bf16 path needs d % 128 == 0
    st = lib.vmoe_expert_fwd(ctypes.byref(odd), P, P, P, P, P, P, P, None)
    assert st == vm.VMOE_ERR_UNSUPPORTED
    st = lib.vmoe_expert_bwd_static_scratch(
        ctypes.byref(vm.problem(17, 1576, 768, 3072, 32, 2, 1.25, "f32")), P, P, P, P, P, P, P, P,
        P, P, None)
    assert st == vm.VMOE_ERR_UNSUPPORTED  # fp32 dH larger than the static array (no slices)
    big = vm.problem(1, 8192, 128, 8192, 1, 1, 1.0)  # one group's dH (2 x 8192 x 8192 bf16) > 64 MiB
    st = lib.vmoe_expert_bwd_static_scratch(ctypes.byref(big), P, P, P, P, P, P, P, P, P, P, None)
    assert st == vm.VMOE_ERR_UNSUPPORTED
    # the 17-task bf16 step fits in slices: one group's dH plus the plan
    t17 = vm.problem(17, 1576, 768, 3072, 32, 2, 1.25)
    assert vm.vmoe_expert_bwd_min_workspace_size(t17) == 4352 + 248 * 3072 * 2
    # router backward: W_r is required with dx, logits with VMOE_NO_RENORM
    st = lib.vmoe_router_bwd(ctypes.byref(p), P, None, None, P, P, P, P, P, P, P, P, None, P, None)
    assert st == vm.VMOE_ERR_INVALID
    nr = vm.problem(2, 64, 128, 256, 4, 2, 1.25, "bf16", flags=vm.VMOE_NO_RENORM)
    st = lib.vmoe_router_bwd(ctypes.byref(nr), P, P, None, P, P, P, P, P, P, P, P, None, None, None)
    assert st == vm.VMOE_ERR_INVALID
    st = lib.vmoe_router_bwd(ctypes.byref(p), P, None, None, P, P, P, P, P, P, P, P + 8, None, None,
                             None)
    assert st == vm.VMOE_ERR_INVALID  # misaligned dW_r
    # bf16: dH as (bf16 value, bf16 residual) pairs
    assert vm.vmoe_expert_bwd_workspace_size(p) == 2 * 4 * oracle.capacity(64, 4, 2, 1.25) * 256 * 2 * 2
    for s in (0, -1, -2, -3, -4, 7):
        assert isinstance(vm.status_string(s), str) and vm.status_string(s)


def test_attention_expert_arguments_rejected_on_host(vm):
    """Attention experts: bf16, an even head count, d % 128 == 0 and C <= 512, else
    VMOE_ERR_UNSUPPORTED; null pointers and a short workspace are VMOE_ERR_INVALID."""
    lib = vm.library()
    P = 1 << 20
    p = vm.problem(2, 300, 256, 1, 4, 2, 1.25, "bf16")
    ws = vm.vmoe_attn_expert_bwd_workspace_size(p, 2)
    C = oracle.capacity(300, 4, 2, 1.25)
    assert ws == 8 * C * 128 * 2 + 8 * C * 384 * 2 + 8 * 2 * C * 4  # dO, dQKV, D
    assert lib.vmoe_attn_expert_fwd(ctypes.byref(p), 2, P, P, P, P, P, P, P, None, None) == vm.VMOE_ERR_INVALID
    assert lib.vmoe_attn_expert_fwd(ctypes.byref(p), 3, P, P, P, P, P, P, P, P, None) == vm.VMOE_ERR_UNSUPPORTED
    assert lib.vmoe_attn_expert_fwd(ctypes.byref(p), 0, P, P, P, P, P, P, P, P, None) == vm.VMOE_ERR_INVALID
    pf = vm.problem(2, 300, 256, 1, 4, 2, 1.25, "f32")
    assert lib.vmoe_attn_expert_fwd(ctypes.byref(pf), 2, P, P, P, P, P, P, P, P, None) == vm.VMOE_ERR_UNSUPPORTED
    wide = vm.problem(1, 4096, 256, 1, 2, 1, 1.0, "bf16")  # C = 2048 > 512
    assert vm.vmoe_attn_expert_bwd_workspace_size(wide, 2) == 0
    args = [P] * 12
    assert lib.vmoe_attn_expert_bwd(ctypes.byref(p), 2, *args, ws - 1, None) == vm.VMOE_ERR_INVALID
