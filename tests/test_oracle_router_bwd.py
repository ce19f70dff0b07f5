"""Pins of the oracle's router backward (CPU only).

The router gradient is the derivative of L = <dY, y> through the gates with the
routing (chosen experts, slots) fixed: it is checked against torch float64
autograd of the whole routed layer written independently (gates as a softmax of
the selected logits, or the full softmax gathered, times the expert MLP outputs),
and against central finite differences of L in W_r, the bias and x that re-route
through the oracle itself (the perturbation is small enough that no choice or
slot changes, which the test asserts).
"""
import numpy as np
import pytest
import torch

import oracle


def _problem(seed, T=2, N=12, E=4, k=2, d=6, f=8, C=5):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((T, N, d))
    wr = rng.standard_normal((T, d, E)) / np.sqrt(d)
    b = rng.standard_normal((T, E)) * 0.5
    w1 = rng.standard_normal((T, E, d, f)) / np.sqrt(d)
    w2 = rng.standard_normal((T, E, f, d)) / np.sqrt(f)
    dy = rng.standard_normal((T, N, d))
    return x, wr, b, w1, w2, dy, k, C


def _oracle_grads(x, wr, b, w1, w2, dy, k, C, flags):
    T, N, d = x.shape
    E = wr.shape[2]
    out = oracle.step(x, wr, b, w1, w2, dy, k, C, flags)
    _, dl, dw, db, dxr = oracle.router_bwd(x, wr, out["logits"], out["idx"], out["gate"],
                                           out["slot"], dy, out["ye"], flags)
    return out, dl, dw, db, out["dx"] + dxr


def _torch_layer(x, wr, b, w1, w2, idx, slot, renorm, tanh):
    logits = torch.einsum("tnd,tde->tne", x, wr) + b[:, None, :]
    il = torch.as_tensor(idx, dtype=torch.int64)
    if renorm:
        gates = torch.softmax(torch.gather(logits, -1, il), dim=-1)
    else:
        gates = torch.gather(torch.softmax(logits, dim=-1), -1, il)
    T, N, k = idx.shape
    y = torch.zeros_like(x)
    rows = []
    for t in range(T):
        for n in range(N):
            acc = torch.zeros(x.shape[-1], dtype=x.dtype)
            for j in range(k):
                if slot[t, n, j] < 0:
                    continue
                e = int(idx[t, n, j])
                h = x[t, n] @ w1[t, e]
                a = torch.nn.functional.gelu(h, approximate="tanh" if tanh else "none")
                acc = acc + gates[t, n, j] * (a @ w2[t, e])
            rows.append(acc)
    return torch.stack(rows).reshape(x.shape), logits


@pytest.mark.parametrize("flags", [0, oracle.FLAG_NO_RENORM, oracle.FLAG_GELU_TANH])
def test_router_bwd_against_torch_autograd(flags):
    x, wr, b, w1, w2, dy, k, C = _problem(3 + flags)
    out, dl, dw, db, dx_total = _oracle_grads(x, wr, b, w1, w2, dy, k, C, flags)
    assert np.any(out["slot"] < 0)  # some choices are dropped
    tx, twr, tb = (torch.tensor(a, requires_grad=True) for a in (x, wr, b))
    y, logits = _torch_layer(tx, twr, tb, torch.tensor(w1), torch.tensor(w2), out["idx"],
                             out["slot"], not (flags & oracle.FLAG_NO_RENORM),
                             bool(flags & oracle.FLAG_GELU_TANH))
    logits.retain_grad()
    (y * torch.tensor(dy)).sum().backward()
    np.testing.assert_allclose(y.detach().numpy(), out["y"], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(dl, logits.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dw, twr.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(db, tb.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dx_total, tx.grad.numpy(), rtol=1e-10, atol=1e-12)


@pytest.mark.parametrize("flags", [0, oracle.FLAG_NO_RENORM])
def test_router_bwd_finite_differences(flags):
    x, wr, b, w1, w2, dy, k, C = _problem(11 + flags, T=1, N=8, E=3, d=4, f=5, C=4)
    out, dl, dw, db, dx_total = _oracle_grads(x, wr, b, w1, w2, dy, k, C, flags)
    idx0, slot0 = out["idx"], out["slot"]
    E = wr.shape[2]

    def loss(x_, wr_, b_):
        lg = oracle.router_logits(x_, wr_, b_)
        idx, gate, slot, load = oracle.route(lg, k, C, flags)
        assert np.array_equal(idx, idx0) and np.array_equal(slot, slot0)
        xe = oracle.dispatch(x_, None, idx, slot, E, C)
        _, _, ye = oracle.expert_fwd(xe, w1, w2, load, flags)
        return float((oracle.combine(ye, gate, idx, slot, x_.shape[1]) * dy).sum())

    eps = 1e-6
    for name, arr, grad in (("wr", wr, dw), ("b", b, db), ("x", x, dx_total)):
        fd = np.zeros_like(arr)
        it = np.nditer(arr, flags=["multi_index"])
        for _ in it:
            i = it.multi_index
            p, m = arr.copy(), arr.copy()
            p[i] += eps
            m[i] -= eps
            args_p = {"wr": (x, p, b), "b": (x, wr, p), "x": (p, wr, b)}[name]
            args_m = {"wr": (x, m, b), "b": (x, wr, m), "x": (m, wr, b)}[name]
            fd[i] = (loss(*args_p) - loss(*args_m)) / (2 * eps)
        err = np.max(np.abs(fd - grad)) / np.max(np.abs(grad))
        assert err < 1e-6, (name, err)


def test_router_bwd_dropped_choice_has_zero_gate_gradient():
    x, wr, b, w1, w2, dy, k, C = _problem(5, C=2)
    out, dl, dw, db, dx_total = _oracle_grads(x, wr, b, w1, w2, dy, k, C, 0)
    dgate, *_ = oracle.router_bwd(x, wr, out["logits"], out["idx"], out["gate"], out["slot"], dy,
                                  out["ye"], 0)
    assert np.all(dgate[out["slot"] < 0] == 0.0)
    # softmax over the selected logits: the gradient of every token's logits sums to 0
    np.testing.assert_allclose(dl.sum(-1), 0.0, atol=1e-12)
