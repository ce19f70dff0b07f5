"""Pins of the fp64 oracle against things other than itself (CPU only).

Every check here comes from the mathematics, a library routine or a hand-derived
fixture, so that a dropped term, a wrong sign, a swapped index or a transposed
operand anywhere in the oracle fails at least one of them:
  * capacity        closed form for the five workloads, override and clamps
  * router logits   numpy einsum
  * top-k           brute-force enumeration of ordered k-tuples (E <= 6), and the
                    dominance characterisation of the chosen set
  * gates           scipy softmax, shift invariance, k=1 renormalised gate = 1
  * capacity scan   rank-by-stable-argsort rule, a hand-derived golden fixture
  * dispatch/combine  brute-force placement check, identity-expert invariant
  * expert FFN      torch float64 autograd on the dense case (E=1, k=1, C=N),
                    erf and tanh GELU, and central finite differences of the
                    composed routed forward with routing frozen
"""
import itertools
import json
import os

import numpy as np
import pytest
import scipy.special
import torch

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_capacity_closed_form():
    # ceil(cf*k*N/E): 2*2*64/4 = 64; 1.25*2*1576/8 = 492.5; 1.25*2*3152/32 = 246.25;
    # 1.25*2*1576/32 = 123.125; 1*1*1576/64 = 24.625
    assert oracle.capacity(64, 4, 2, 2.0) == 64
    assert oracle.capacity(1576, 8, 2, 1.25) == 493
    assert oracle.capacity(3152, 32, 2, 1.25) == 247
    assert oracle.capacity(1576, 32, 2, 1.25) == 124
    assert oracle.capacity(1576, 64, 1, 1.0) == 25
    assert oracle.capacity(100, 10, 1, 1.0) == 10       # exact product, no rounding up
    assert oracle.capacity(10, 4, 2, 1e-9) == 1          # clamp to >= 1
    assert oracle.capacity(10, 1, 2, 8.0) == 10          # clamp to <= N
    assert oracle.capacity(10, 4, 2, 1.0, 7) == 7        # explicit override


def test_router_logits_match_einsum():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((3, 7, 5))
    w = rng.standard_normal((3, 5, 4))
    b = rng.standard_normal((3, 4))
    ref = np.einsum("tnd,tde->tne", x, w) + b[:, None, :]
    np.testing.assert_allclose(oracle.router_logits(x, w, b), ref, rtol=1e-13, atol=1e-13)
    np.testing.assert_allclose(oracle.router_logits(x, w, None),
                               np.einsum("tnd,tde->tne", x, w), rtol=1e-13, atol=1e-13)


def _brute_topk(l, k):
    """The ordered k-tuple of distinct experts whose key (l[e0], -e0, l[e1], -e1, ...)
    is lexicographically largest."""
    best, best_key = None, None
    for tup in itertools.permutations(range(len(l)), k):
        key = tuple(v for e in tup for v in (l[e], -e))
        if best_key is None or key > best_key:
            best, best_key = tup, key
    return list(best)


@pytest.mark.parametrize("E,k", [(2, 1), (3, 2), (4, 2), (5, 3), (6, 2), (6, 1)])
@pytest.mark.parametrize("quantised", [False, True])
def test_topk_brute_force(E, k, quantised):
    rng = np.random.default_rng(E * 10 + k + (100 if quantised else 0))
    N = 40
    lg = rng.standard_normal((1, N, E))
    if quantised:  # only 3 distinct values: many ties
        lg = np.round(lg).clip(-1, 1)
    idx, gate, slot, load = oracle.route(lg, k, C=N)
    for n in range(N):
        l = list(lg[0, n])
        assert list(idx[0, n]) == _brute_topk(l, k)
        chosen = set(idx[0, n])
        for c in chosen:
            for u in set(range(E)) - chosen:
                assert l[c] > l[u] or (l[c] == l[u] and c < u)


def test_gates_closed_forms():
    rng = np.random.default_rng(7)
    T, N, E, k = 2, 30, 8, 3
    lg = rng.standard_normal((T, N, E)) * 2.0
    idx, gate, _, _ = oracle.route(lg, k, C=N)
    idx_nr, gate_nr, _, _ = oracle.route(lg, k, C=N, flags=oracle.FLAG_NO_RENORM)
    assert np.array_equal(idx, idx_nr)
    p = scipy.special.softmax(lg, axis=-1)
    sel = np.take_along_axis(p, idx.astype(np.int64), axis=-1)
    np.testing.assert_allclose(gate_nr, sel, rtol=1e-14)
    # renormalised gates are the softmax of the selected logits alone
    sel_l = np.take_along_axis(lg, idx.astype(np.int64), axis=-1)
    np.testing.assert_allclose(gate, scipy.special.softmax(sel_l, axis=-1), rtol=1e-13)
    np.testing.assert_allclose(gate.sum(-1), 1.0, rtol=1e-14)
    assert np.all(gate_nr.sum(-1) <= 1.0 + 1e-14)
    assert np.all(np.diff(gate, axis=-1) <= 0)  # ordered like the logits
    # shift invariance of softmax gating
    idx2, gate2, _, _ = oracle.route(lg + 123.5, k, C=N)
    assert np.array_equal(idx, idx2)
    np.testing.assert_allclose(gate, gate2, rtol=1e-12)
    # top-1 renormalised gate is exactly 1
    _, g1, _, _ = oracle.route(lg, 1, C=N)
    assert np.all(g1 == 1.0)


def _slots_by_rank(idx, E, C):
    """Slot rule written independently: in choice-major order p = j*N + n, the
    assignment's slot is its rank among earlier assignments to the same expert,
    or -1 once that rank reaches C."""
    T, N, k = idx.shape
    slot = np.empty_like(idx)
    load = np.zeros((T, E), np.int32)
    for t in range(T):
        seq = idx[t].T.reshape(-1)  # choice-major
        order = np.argsort(seq, kind="stable")
        ranks = np.empty(len(seq), np.int64)
        sorted_e = seq[order]
        starts = np.searchsorted(sorted_e, np.arange(E), side="left")
        ranks[order] = np.arange(len(seq)) - starts[sorted_e]
        s = np.where(ranks < C, ranks, -1)
        slot[t] = s.reshape(k, N).T
        load[t] = np.minimum(np.bincount(seq, minlength=E), C)
    return slot, load


@pytest.mark.parametrize("T,N,E,k,C", [(1, 50, 4, 2, 9), (3, 64, 8, 2, 5), (2, 33, 5, 3, 40),
                                       (2, 100, 16, 1, 3), (1, 20, 2, 2, 1)])
def test_capacity_scan_rank_rule(T, N, E, k, C):
    rng = np.random.default_rng(T * 1000 + N + E + k + C)
    lg = rng.standard_normal((T, N, E))
    idx, gate, slot, load = oracle.route(lg, k, C)
    ref_slot, ref_load = _slots_by_rank(idx, E, C)
    assert np.array_equal(slot, ref_slot)
    assert np.array_equal(load, ref_load)
    assert np.all(load <= C)
    for t in range(T):  # kept slots of each expert are exactly 0..load-1
        for e in range(E):
            s = np.sort(slot[t][(idx[t] == e) & (slot[t] >= 0)])
            assert np.array_equal(s, np.arange(load[t, e]))


def test_route_golden_fixture():
    with open(os.path.join(GOLDEN, "route_tiny.json")) as fh:
        g = json.load(fh)
    idx, gate, slot, load = oracle.route(np.array(g["logits"]), g["k"], g["C"])
    assert idx.tolist() == g["idx"]
    assert slot.tolist() == g["slot"]
    assert load.tolist() == g["load"]
    np.testing.assert_allclose(gate, np.array(g["gate_renorm"]), rtol=1e-15)
    _, gate_nr, _, _ = oracle.route(np.array(g["logits"]), g["k"], g["C"],
                                    flags=oracle.FLAG_NO_RENORM)
    l = np.array(g["logits"])[0]
    p = np.exp(l) / np.exp(l).sum(-1, keepdims=True)
    for n in range(g["N"]):
        for j in range(g["k"]):
            assert abs(gate_nr[0, n, j] - p[n, g["idx"][0][n][j]]) < 1e-15


def _tiny_routing(seed, T=2, N=24, E=4, k=2, C=8, d=6):
    rng = np.random.default_rng(seed)
    lg = rng.standard_normal((T, N, E))
    idx, gate, slot, load = oracle.route(lg, k, C)
    x = rng.standard_normal((T, N, d))
    return x, idx, gate, slot, load, E, C


def test_dispatch_brute_force_placement():
    x, idx, gate, slot, load, E, C = _tiny_routing(3)
    T, N, d = x.shape
    xe = oracle.dispatch(x, None, idx, slot, E, C)
    xw = oracle.dispatch(x, gate, idx, slot, E, C)
    for t in range(T):
        for e in range(E):
            for s in range(C):
                src = [(n, j) for n in range(N) for j in range(idx.shape[2])
                       if idx[t, n, j] == e and slot[t, n, j] == s]
                assert len(src) <= 1
                if s < load[t, e]:
                    (n, j), = src
                    assert np.array_equal(xe[t, e, s], x[t, n])
                    np.testing.assert_allclose(xw[t, e, s], gate[t, n, j] * x[t, n], rtol=1e-15)
                else:
                    assert not src
                    assert np.all(xe[t, e, s] == 0) and np.all(xw[t, e, s] == 0)


def test_combine_of_identity_experts():
    x, idx, gate, slot, load, E, C = _tiny_routing(4)
    N = x.shape[1]
    xe = oracle.dispatch(x, None, idx, slot, E, C)
    kept_mass = np.where(slot >= 0, gate, 0.0).sum(-1)
    kept_count = (slot >= 0).sum(-1)
    y = oracle.combine(xe, gate, idx, slot, N)
    np.testing.assert_allclose(y, x * kept_mass[..., None], rtol=1e-14, atol=1e-15)
    y1 = oracle.combine(xe, None, idx, slot, N)
    np.testing.assert_allclose(y1, x * kept_count[..., None], rtol=1e-14, atol=1e-15)
    assert np.any(kept_count < 2)  # the case really has drops


@pytest.mark.parametrize("tanh", [False, True])
def test_dense_special_case_against_torch_autograd(tanh):
    """E=1, k=1, C=N: every token goes to the single expert with gate 1, so the
    layer is a dense Linear-GELU-Linear MLP; torch float64 autograd is the
    independent reference for the forward and all three gradients."""
    rng = np.random.default_rng(11)
    T, N, d, f = 2, 9, 5, 7
    flags = oracle.FLAG_GELU_TANH if tanh else 0
    x = rng.standard_normal((T, N, d))
    wr = rng.standard_normal((T, d, 1))
    w1 = rng.standard_normal((T, 1, d, f)) / np.sqrt(d)
    w2 = rng.standard_normal((T, 1, f, d)) / np.sqrt(f)
    dy = rng.standard_normal((T, N, d))
    C = oracle.capacity(N, 1, 1, 1.0)
    assert C == N
    out = oracle.step(x, wr, None, w1, w2, dy, k=1, C=C, flags=flags)
    assert np.all(out["slot"][..., 0] == np.arange(N)) and np.all(out["gate"] == 1.0)

    tx = torch.tensor(x, requires_grad=True)
    t1 = torch.tensor(w1[:, 0], requires_grad=True)
    t2 = torch.tensor(w2[:, 0], requires_grad=True)
    th = tx @ t1
    th.retain_grad()
    ta = torch.nn.functional.gelu(th, approximate="tanh" if tanh else "none")
    ty = ta @ t2
    (ty * torch.tensor(dy)).sum().backward()
    np.testing.assert_allclose(out["h"][:, 0], th.detach().numpy(), rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(out["a"][:, 0], ta.detach().numpy(), rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(out["y"], ty.detach().numpy(), rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(out["dh"][:, 0], th.grad.numpy(), rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(out["dx"], tx.grad.numpy(), rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(out["dw1"][:, 0], t1.grad.numpy(), rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(out["dw2"][:, 0], t2.grad.numpy(), rtol=1e-11, atol=1e-13)


@pytest.mark.parametrize("tanh", [False, True])
def test_finite_differences_routed(tanh):
    """Central differences of L = <dY, combine(FFN(dispatch(x)), gate)> with the
    routing (idx, gate, slot) frozen, against the oracle's backward."""
    flags = oracle.FLAG_GELU_TANH if tanh else 0
    rng = np.random.default_rng(21)
    T, N, E, k, d, f = 2, 10, 3, 2, 4, 6
    C = 4  # 2*10/3 = 6.7 -> capacity 4 forces drops
    lg = rng.standard_normal((T, N, E))
    idx, gate, slot, load = oracle.route(lg, k, C)
    assert np.any(slot < 0)
    x = rng.standard_normal((T, N, d))
    w1 = rng.standard_normal((T, E, d, f)) / np.sqrt(d)
    w2 = rng.standard_normal((T, E, f, d)) / np.sqrt(f)
    dy = rng.standard_normal((T, N, d))

    def loss(x_, w1_, w2_):
        xe = oracle.dispatch(x_, None, idx, slot, E, C)
        _, _, ye = oracle.expert_fwd(xe, w1_, w2_, load, flags)
        return float((oracle.combine(ye, gate, idx, slot, N) * dy).sum())

    xe = oracle.dispatch(x, None, idx, slot, E, C)
    h, a, ye = oracle.expert_fwd(xe, w1, w2, load, flags)
    dye = oracle.dispatch(dy, gate, idx, slot, E, C)
    _, dxe, dw1, dw2 = oracle.expert_bwd(xe, h, a, w1, w2, dye, load, flags)
    dx = oracle.combine(dxe, None, idx, slot, N)

    eps = 1e-6
    for name, arr, grad in (("x", x, dx), ("w1", w1, dw1), ("w2", w2, dw2)):
        fd = np.zeros_like(arr)
        it = np.nditer(arr, flags=["multi_index"])
        for _ in it:
            i = it.multi_index
            p, m = arr.copy(), arr.copy()
            p[i] += eps
            m[i] -= eps
            args_p = {"x": (p, w1, w2), "w1": (x, p, w2), "w2": (x, w1, p)}[name]
            args_m = {"x": (m, w1, w2), "w1": (x, m, w2), "w2": (x, w1, m)}[name]
            fd[i] = (loss(*args_p) - loss(*args_m)) / (2 * eps)
        err = np.max(np.abs(fd - grad)) / np.max(np.abs(grad))
        assert err < 1e-6, (name, err)
    # an expert that received no token has zero weight gradients
    empty = load.reshape(-1) == 0
    assert np.all(dw1.reshape(T * E, d, f)[empty] == 0)
