"""Pins of the oracle's attention experts (CPU only).

The forward and backward of H-head softmax attention among each group's routed
tokens (the reading of Section 2.1's expertized attention, with the T^2 score
term of Section 3.2.1) are checked against
  * torch float64 autograd through torch.nn.functional.scaled_dot_product_attention,
    a separate implementation of the attention core that the oracle does not use,
    for the forward and for every gradient;
  * central finite differences of <dYe, Ye> in Xe and in each weight;
  * closed forms: one token (the softmax of one score is 1, so Ye = Xe W_v W_o);
    W_q = 0 (every score equal, so each head's output is the mean of its V rows);
    the token order (attention among the group's tokens is permutation
    equivariant); padding rows and empty groups (no effect, zero outputs).
"""
import numpy as np
import pytest
import torch

from oracle import attention as att


def _case(seed, G=3, C=9, d=16, H=2, dk=4, loads=(9, 5, 0)):
    rng = np.random.default_rng(seed)
    hd = H * dk
    xe = rng.standard_normal((G, C, d))
    wq, wk, wv = (rng.standard_normal((G, d, hd)) / np.sqrt(d) for _ in range(3))
    wo = rng.standard_normal((G, hd, d)) / np.sqrt(hd)
    dye = rng.standard_normal((G, C, d))
    load = np.array(loads[:G])
    for g in range(G):  # padding rows hold junk that must not matter
        xe[g, load[g]:] = 1e3
        dye[g, load[g]:] = -1e3
    return xe, wq, wk, wv, wo, dye, load, H


def _torch_ref(xe, wq, wk, wv, wo, dye, load, H):
    G, C, d = xe.shape
    out = {"ye": np.zeros_like(xe), "dxe": np.zeros_like(xe), "dwq": np.zeros_like(wq),
           "dwk": np.zeros_like(wk), "dwv": np.zeros_like(wv), "dwo": np.zeros_like(wo)}
    for g in range(G):
        L = int(load[g])
        if L == 0:
            continue
        x = torch.tensor(xe[g, :L], requires_grad=True)
        ws = [torch.tensor(w[g], requires_grad=True) for w in (wq, wk, wv, wo)]
        hd = ws[0].shape[1]
        dk = hd // H

        def heads(t):
            return t.reshape(L, H, dk).permute(1, 0, 2)  # [H, L, dk]
        q, k, v = heads(x @ ws[0]), heads(x @ ws[1]), heads(x @ ws[2])
        o = torch.nn.functional.scaled_dot_product_attention(q, k, v)
        y = o.permute(1, 0, 2).reshape(L, hd) @ ws[3]
        (y * torch.tensor(dye[g, :L])).sum().backward()
        out["ye"][g, :L] = y.detach().numpy()
        out["dxe"][g, :L] = x.grad.numpy()
        for n, w in zip(("dwq", "dwk", "dwv", "dwo"), ws):
            out[n][g] = w.grad.numpy()
    return out


@pytest.mark.parametrize("seed", range(6))
def test_against_torch_autograd(seed):
    c = _case(seed)
    fw = att.attention_expert_fwd(*c[:5], c[6], c[7])
    bw = att.attention_expert_bwd(*c)
    ref = _torch_ref(*c)
    np.testing.assert_allclose(fw["ye"], ref["ye"], rtol=1e-10, atol=1e-12)
    for n in ("dxe", "dwq", "dwk", "dwv", "dwo"):
        np.testing.assert_allclose(bw[n], ref[n], rtol=1e-9, atol=1e-11, err_msg=n)


def test_finite_differences():
    xe, wq, wk, wv, wo, dye, load, H = _case(11, G=1, C=6, d=8, H=2, dk=3, loads=(6,))
    bw = att.attention_expert_bwd(xe, wq, wk, wv, wo, dye, load, H)

    def f(xe_, wq_, wk_, wv_, wo_):
        return float((att.attention_expert_fwd(xe_, wq_, wk_, wv_, wo_, load, H)["ye"] * dye).sum())
    rng = np.random.default_rng(0)
    args = [xe, wq, wk, wv, wo]
    for i, name in enumerate(("dxe", "dwq", "dwk", "dwv", "dwo")):
        for _ in range(6):
            idx = tuple(rng.integers(0, s) for s in args[i].shape)
            h = 1e-6
            up = [a.copy() for a in args]
            dn = [a.copy() for a in args]
            up[i][idx] += h
            dn[i][idx] -= h
            num = (f(*up) - f(*dn)) / (2 * h)
            assert abs(num - bw[name][idx]) < 1e-6 * max(1.0, abs(num)), (name, idx)


def test_one_token_is_the_value_path():
    xe, wq, wk, wv, wo, dye, load, H = _case(3, G=1, loads=(1,))
    fw = att.attention_expert_fwd(xe, wq, wk, wv, wo, load, H)
    np.testing.assert_allclose(fw["ye"][0, 0], xe[0, 0] @ wv[0] @ wo[0], rtol=1e-12)
    assert np.all(fw["p"][0, :, 0, 0] == 1.0)


def test_zero_queries_average_the_values():
    xe, wq, wk, wv, wo, dye, load, H = _case(4, G=1, loads=(7,))
    wq = np.zeros_like(wq)
    fw = att.attention_expert_fwd(xe, wq, wk, wv, wo, load, H)
    v = xe[0, :7] @ wv[0]
    np.testing.assert_allclose(fw["o"][0, :7], np.broadcast_to(v.mean(axis=0), (7, v.shape[1])),
                               rtol=1e-12, atol=1e-14)


def test_permutation_equivariance_padding_and_empty_groups():
    xe, wq, wk, wv, wo, dye, load, H = _case(5)
    fw = att.attention_expert_fwd(xe, wq, wk, wv, wo, load, H)
    perm = np.random.default_rng(1).permutation(5)
    xp = xe.copy()
    xp[1, :5] = xe[1, perm]
    fp = att.attention_expert_fwd(xp, wq, wk, wv, wo, load, H)
    np.testing.assert_allclose(fp["ye"][1, :5], fw["ye"][1, perm], rtol=1e-12, atol=1e-13)
    assert np.all(fw["ye"][1, 5:] == 0) and np.all(fw["ye"][2] == 0)
    bw = att.attention_expert_bwd(xe, wq, wk, wv, wo, dye, load, H)
    assert np.all(bw["dwq"][2] == 0) and np.all(bw["dxe"][2] == 0) and np.all(bw["dxe"][1, 5:] == 0)
    # junk in padding rows changes nothing
    xj = xe.copy()
    xj[1, 5:] = -7.0
    assert np.array_equal(att.attention_expert_fwd(xj, wq, wk, wv, wo, load, H)["ye"], fw["ye"])


def test_stored_o_enters_only_through_d_and_dwo():
    """The backward handed the forward's O: the exact O reproduces the default
    (rowsum(dO_h * O_h) = rowsum(dP_h * P_h) when O_h = P_h V_h); an O moved
    orthogonally to dO in every head row leaves D, hence dXe and dW_q,k,v, as
    they were and moves dW_o by (the move)^T dYe; a move along dO shifts each
    row's dS by -P_ij r_i, with r_i the change of D_i."""
    xe, wq, wk, wv, wo, dye, load, H = _case(6)
    fw = att.attention_expert_fwd(xe, wq, wk, wv, wo, load, H)
    base = att.attention_expert_bwd(xe, wq, wk, wv, wo, dye, load, H)
    same = att.attention_expert_bwd(xe, wq, wk, wv, wo, dye, load, H, o=fw["o"])
    for n in base:
        np.testing.assert_allclose(same[n], base[n], rtol=1e-10, atol=1e-12)
    G, C, d = xe.shape
    hd = wq.shape[-1]
    dk = hd // H
    rng = np.random.default_rng(11)
    do = np.einsum("gcd,ghd->gch", dye, wo)
    delta = np.zeros((G, C, hd))
    for g in range(G):
        L = int(load[g])
        for h in range(H):
            c = slice(h * dk, (h + 1) * dk)
            r = rng.standard_normal((L, dk))
            u = do[g, :L, c]
            delta[g, :L, c] = r - (r * u).sum(1, keepdims=True) / (u * u).sum(1, keepdims=True) * u
    orth = att.attention_expert_bwd(xe, wq, wk, wv, wo, dye, load, H, o=fw["o"] + delta)
    for n in ("dxe", "dwq", "dwk", "dwv"):
        np.testing.assert_allclose(orth[n], base[n], rtol=1e-10, atol=1e-12)
    rows = (np.arange(C)[None, :] < load[:, None])[..., None]
    np.testing.assert_allclose(orth["dwo"] - base["dwo"], np.einsum("gch,gcd->ghd", delta, dye * rows),
                               rtol=1e-10, atol=1e-12)
    # along dO: D_i of head h grows by r_i = 0.1 |dO_i,h|^2, so dQ_h moves by -diag(r) P_h K_h / sqrt(d_k)
    along = att.attention_expert_bwd(xe, wq, wk, wv, wo, dye, load, H, o=fw["o"] + 0.1 * do * rows)
    np.testing.assert_allclose(along["dwv"], base["dwv"], rtol=1e-10, atol=1e-12)
    want = base["dwq"].copy()
    for g in range(G):
        L = int(load[g])
        if L == 0:
            continue
        x = xe[g, :L]
        q, k = x @ wq[g], x @ wk[g]
        dq = np.zeros((L, hd))
        for h in range(H):
            c = slice(h * dk, (h + 1) * dk)
            r = 0.1 * (do[g, :L, c] ** 2).sum(1, keepdims=True)
            dq[:, c] = -(r * fw["p"][g, h, :L, :L]) @ k[:, c] / np.sqrt(dk)
        want[g] += x.T @ dq
    np.testing.assert_allclose(along["dwq"], want, rtol=1e-9, atol=1e-11)
