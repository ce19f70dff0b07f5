"""Oracle of the attention-expert variant -- TEST INFRASTRUCTURE, NOT PRODUCT CODE.

Only the test suite, the smoke check and the benchmark's CPU-baseline leg may
import this module.  It shares no code with the CUDA library.

Section 2.1 says V-MoE turns the ViT's self-attention as well as its MLP into
expertized blocks with routed tokens, and Section 3.2.1's memory estimator gives
an attention expert with T tokens and key width d_k buffers of order T d_k (the
Q / K / V projections) and T^2 (the attention scores).  The paper gives no
further detail.  The readings taken here:

  * an attention expert e of task t owns W_q, W_k, W_v [d, H d_k] and
    W_o [H d_k, d]; its input is the block of tokens dispatched to it,
    Xe[t,e] rows [0, L) with L = load[t,e] (the same routing, capacity and
    dispatch as the FFN experts);
  * it runs H-head softmax attention among those L tokens only -- tokens of
    other experts and padding rows are neither queries nor keys:
        Q = Xe W_q, K = Xe W_k, V = Xe W_v                       [L, H d_k]
        S_h = Q_h K_h^T / sqrt(d_k),  P_h = softmax over the L keys  [L, L]
        O_h = P_h V_h,  O = [O_1 .. O_H],  Ye = O W_o             [L, d]
    and the combine gate-weights Ye back to token order as for the FFN;
  * no biases, no masking within the L tokens, the softmax with its row
    maximum subtracted;
  * the backward holds routing and gates fixed (as for the FFN experts): the
    gradient of <dYe, Ye> with respect to Xe and the four weights.

float64 throughout; numpy matmul is the only library primitive.
"""
from __future__ import annotations

import numpy as np


def _f64(a):
    return np.asarray(a, dtype=np.float64)


def attention_expert_fwd(xe, wq, wk, wv, wo, load, heads):
    """Forward of every (task, expert) group.

    xe [G, C, d]; wq, wk, wv [G, d, H*dk]; wo [G, H*dk, d]; load [G] (or [T, E]).
    Returns dict of Q, K, V, O [G, C, H*dk], P [G, H, C, C] and ye [G, C, d];
    rows (and for P, columns) at or past a group's load are zero."""
    xe, wq, wk, wv, wo = map(_f64, (xe, wq, wk, wv, wo))
    G, C, d = xe.reshape(-1, xe.shape[-2], xe.shape[-1]).shape
    xe = xe.reshape(G, C, d)
    wq, wk, wv = (w.reshape(G, d, -1) for w in (wq, wk, wv))
    hd = wq.shape[-1]
    wo = wo.reshape(G, hd, d)
    dk = hd // heads
    ld = np.asarray(load).reshape(-1)
    out = {k: np.zeros((G, C, hd)) for k in ("q", "k", "v", "o")}
    out["p"] = np.zeros((G, heads, C, C))
    out["ye"] = np.zeros((G, C, d))
    scale = 1.0 / np.sqrt(dk)
    for g in range(G):
        L = int(min(max(ld[g], 0), C))
        if L == 0:
            continue
        x = xe[g, :L]
        q, k, v = x @ wq[g], x @ wk[g], x @ wv[g]
        o = np.zeros((L, hd))
        for h in range(heads):
            c = slice(h * dk, (h + 1) * dk)
            s = (q[:, c] @ k[:, c].T) * scale
            s = s - s.max(axis=1, keepdims=True)
            e = np.exp(s)
            p = e / e.sum(axis=1, keepdims=True)
            o[:, c] = p @ v[:, c]
            out["p"][g, h, :L, :L] = p
        out["q"][g, :L], out["k"][g, :L], out["v"][g, :L], out["o"][g, :L] = q, k, v, o
        out["ye"][g, :L] = o @ wo[g]
    return out


def attention_expert_bwd(xe, wq, wk, wv, wo, dye, load, heads, o=None):
    """Backward of every group: gradients of sum_g <dye[g], ye[g]> (valid rows).

    Returns dict dxe [G, C, d] (rows past the load zero), dwq, dwk, dwv [G, d, H*dk],
    dwo [G, H*dk, d] (zero for an empty group).  Chain rule, step by step:
        dO = dYe W_o^T,  dW_o = O^T dYe
        per head: dV_h = P_h^T dO_h,  dP_h = dO_h V_h^T,
                  dS_h = P_h * (dP_h - D_h),  D_h = rowsum(dP_h * P_h),
                  dQ_h = dS_h K_h / sqrt(d_k),  dK_h = dS_h^T Q_h / sqrt(d_k)
        dXe = dQ W_q^T + dK W_k^T + dV W_v^T,
        dW_q = Xe^T dQ,  dW_k = Xe^T dK,  dW_v = Xe^T dV.

    o [G, C, H*dk], optional: the forward's O as stored by whoever ran the
    forward, for a backward handed that O rather than recomputing it.  It then
    stands in for O in dW_o and in D_h = rowsum(dO_h * O_h), which equals
    rowsum(dP_h * P_h) when O_h = P_h V_h exactly (row i: sum_j P_ij dO_i.V_j)."""
    fw = attention_expert_fwd(xe, wq, wk, wv, wo, load, heads)
    xe, wq, wk, wv, wo, dye = map(_f64, (xe, wq, wk, wv, wo, dye))
    G, C, d = fw["ye"].shape
    xe = xe.reshape(G, C, d)
    dye = dye.reshape(G, C, d)
    wq, wk, wv = (w.reshape(G, d, -1) for w in (wq, wk, wv))
    hd = wq.shape[-1]
    wo = wo.reshape(G, hd, d)
    dk = hd // heads
    ld = np.asarray(load).reshape(-1)
    scale = 1.0 / np.sqrt(dk)
    o_given = None if o is None else _f64(o).reshape(G, C, hd)
    res = {"dxe": np.zeros((G, C, d)), "dwq": np.zeros((G, d, hd)), "dwk": np.zeros((G, d, hd)),
           "dwv": np.zeros((G, d, hd)), "dwo": np.zeros((G, hd, d))}
    for g in range(G):
        L = int(min(max(ld[g], 0), C))
        if L == 0:
            continue
        x, dy = xe[g, :L], dye[g, :L]
        q, k, v, og = (fw[n][g, :L] for n in ("q", "k", "v", "o"))
        if o_given is not None:
            og = o_given[g, :L]
        do = dy @ wo[g].T
        res["dwo"][g] = og.T @ dy
        dq, dkk, dv = np.zeros((L, hd)), np.zeros((L, hd)), np.zeros((L, hd))
        for h in range(heads):
            c = slice(h * dk, (h + 1) * dk)
            p = fw["p"][g, h, :L, :L]
            dv[:, c] = p.T @ do[:, c]
            dp = do[:, c] @ v[:, c].T
            if o_given is None:
                dd = (dp * p).sum(axis=1, keepdims=True)
            else:
                dd = (do[:, c] * og[:, c]).sum(axis=1, keepdims=True)
            ds = p * (dp - dd)
            dq[:, c] = (ds @ k[:, c]) * scale
            dkk[:, c] = (ds.T @ q[:, c]) * scale
        res["dxe"][g, :L] = dq @ wq[g].T + dkk @ wk[g].T + dv @ wv[g].T
        res["dwq"][g] = x.T @ dq
        res["dwk"][g] = x.T @ dkk
        res["dwv"][g] = x.T @ dv
    return res
