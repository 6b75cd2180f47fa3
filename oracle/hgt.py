"""CPU oracle of the attention variant of the layer (Heterogeneous Graph Transformer).  TEST
INFRASTRUCTURE ONLY.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg import this module; the
product path never calls it and shares no code with it.  Plain numpy in fp64, written edge by edge.

What is computed (Section 3.2, Eq. 6-11), for one layer over the typed graph, with S heads of
width d_h = d / S:

* Key, query, value ... K(i) = h_i W_K[tau(i)] + b_K[tau(i)], likewise Q and V (one linear map of
                        each kind per node type; head s takes columns s d_h .. (s + 1) d_h).
* Eq. 6 ............... Att-head^s(i, e, j) = (K^s(i) W_att[r, s] . Q^s(j)) * mu[r] / sqrt(d_h),
                        r = phi(e), W_att[r, s] a d_h x d_h matrix per relation and head.
* Eq. 7 ............... Msg-head^s(i, e, j) = V^s(i) W_msg[r, s].
* Eq. 8 ............... alpha^s(i, e, j) = softmax over all edges e into j (every relation) of the
                        head-s scores.
* Eq. 9-10 ............ h~_j = concat over heads of sum_e alpha^s(e) Msg-head^s(e); 0 for a node with
                        no in-edge.
* Eq. 11 .............. h'_j = sigma(h~_j W_agg[tau(j)] + b_agg[tau(j)]) + h_j, then (optionally)
                        LayerNorm per node type, as in the mean-aggregation layer.
* hgt_backward ........ the chain rule of all of it, step by step.

Readings where the paper is silent or ambiguous (listed again in the design notes):
  K, Q and V are separate linear maps with bias per node type (the paper writes Linear^s for both
  K and Q; the transformer it cites uses three maps); W_att and W_msg are per relation and head;
  mu is one learnable scalar per relation (each relation fixes its endpoint types, so the
  meta-relation triplet is the relation); the softmax runs over every in-edge of j across all
  relations (Eq. 8's N(j)); the aggregation (+) sums the weighted messages; sigma = ReLU; the
  residual needs d_in = d_out; LayerNorm after the residual (population variance, eps 1e-5).
  store="bf16": the tensors the bf16 kernels store -- K, V, Q, the relation-scaled queries
  Q'_r(j) = Q(j) blockdiag(W_att[r])^T mu[r] / sqrt(d_h), the per-relation weighted sums
  S_r(j) = sum over the r-edges into j of alpha V(i), and U without its bias -- are rounded to bf16; weights and
  products of weights are not; all other arithmetic stays fp64.  The GPU tests compare with the
  plain definition (store="f64"); this mode serves to study the effect of those roundings.
"""
from __future__ import annotations

import numpy as np

from .hg_oracle import act_fwd, act_grad, node_type, round_bf16, valid_edges

F64 = np.float64


def blockdiag(W: np.ndarray) -> np.ndarray:
    """S blocks of d_h x d_h -> the d x d block-diagonal matrix."""
    S, dh, _ = W.shape
    out = np.zeros((S * dh, S * dh), F64)
    for s in range(S):
        out[s * dh:(s + 1) * dh, s * dh:(s + 1) * dh] = W[s]
    return out


def _typed_linear(H, types, W, b):
    out = np.empty((H.shape[0], W.shape[2]), F64)
    for t in range(W.shape[0]):
        m = types == t
        out[m] = H[m] @ W[t] + b[t]
    return out


def hgt_forward(src, dst, rel, type_offsets, rels, params: dict, H, heads: int, act: str = "relu",
                layernorm: bool = True, ln_eps: float = 1e-5, store: str = "f64") -> tuple:
    """One layer.  params: W_K, W_Q, W_V (T x d x d), b_K, b_Q, b_V (T x d), W_att, W_msg
    (R x S x d_h x d_h), mu (R), W_agg (T x d x d), b_agg (T x d), ln_gamma, ln_beta (T x d).
    Returns (H_out, cache)."""
    P = {k: np.asarray(v, F64) for k, v in params.items()}
    H = np.asarray(H, F64)
    rnd = round_bf16 if store == "bf16" else (lambda x: x)
    N, d = H.shape
    S = heads
    dh = d // S
    offs = np.asarray(type_offsets, np.int64)
    types = node_type(np.arange(N), offs)
    ok = valid_edges(src, dst, rel, offs, rels)
    src = np.asarray(src, np.int64)[ok]
    dst = np.asarray(dst, np.int64)[ok]
    rel = np.asarray(rel, np.int64)[ok]
    E = src.shape[0]
    K = rnd(_typed_linear(H, types, P["W_K"], P["b_K"]))
    V = rnd(_typed_linear(H, types, P["W_V"], P["b_V"]))
    Q = rnd(_typed_linear(H, types, P["W_Q"], P["b_Q"]))
    scale = P["mu"] / np.sqrt(dh)
    # Eq. 6 through the relation-scaled query of each (relation, target): score = K . Q'
    R = len(rels)
    Qp = np.zeros((R, N, d), F64)
    for r in range(R):
        Qp[r] = rnd(Q @ blockdiag(P["W_att"][r]).T * scale[r])
    score = np.zeros((E, S), F64)
    for s in range(S):
        cols = slice(s * dh, (s + 1) * dh)
        score[:, s] = (K[src, cols] * Qp[rel, dst][:, cols]).sum(axis=1)
    # Eq. 8: softmax over every in-edge of the target, per head
    mx = np.full((N, S), -np.inf)
    np.maximum.at(mx, dst, score)
    ex = np.exp(score - mx[dst])
    den = np.zeros((N, S), F64)
    np.add.at(den, dst, ex)
    alpha = ex / den[dst]
    # Eq. 7, 9, 10 through the per-relation sums S_r(j) = sum alpha V(i), then W_msg
    Ssum = np.zeros((R, N, d), F64)
    for s in range(S):
        cols = slice(s * dh, (s + 1) * dh)
        contrib = alpha[:, s:s + 1] * V[src, cols]
        acc = np.zeros((R, N, dh), F64)
        np.add.at(acc, (rel, dst), contrib)
        Ssum[:, :, cols] = acc
    Ssum = rnd(Ssum)
    U = np.zeros((N, d), F64)
    for t in range(len(offs) - 1):
        lo, hi = int(offs[t]), int(offs[t + 1])
        u = np.zeros((hi - lo, d), F64)
        for r, (_, tt) in enumerate(rels):
            if tt == t:
                Vr = blockdiag(P["W_msg"][r]) @ P["W_agg"][t]
                u += Ssum[r, lo:hi] @ Vr
        U[lo:hi] = rnd(u) + P["b_agg"][t]  # stored without its bias, as the kernels do
    Y = act_fwd(U, act) + H
    out = Y
    mean = rstd = None
    if layernorm:
        mean = Y.mean(axis=1, keepdims=True)
        var = ((Y - mean) ** 2).mean(axis=1, keepdims=True)
        rstd = 1.0 / np.sqrt(var + ln_eps)
        out = (Y - mean) * rstd * P["ln_gamma"][types] + P["ln_beta"][types]
    cache = dict(src=src, dst=dst, rel=rel, types=types, K=K, V=V, Q=Q, Qp=Qp, score=score, alpha=alpha,
                 Ssum=Ssum, U=U, Y=Y, mean=mean, rstd=rstd, scale=scale)
    return out, cache


def hgt_backward(src, dst, rel, type_offsets, rels, params: dict, H, dOut, heads: int, act: str = "relu",
                 layernorm: bool = True, ln_eps: float = 1e-5, store: str = "f64") -> tuple:
    """Gradients of <dOut, H_out> for one layer: (dH, grads) with grads keyed like params."""
    P = {k: np.asarray(v, F64) for k, v in params.items()}
    H = np.asarray(H, F64)
    _, c = hgt_forward(src, dst, rel, type_offsets, rels, params, H, heads, act, layernorm, ln_eps, store)
    N, d = H.shape
    S = heads
    dh = d // S
    offs = np.asarray(type_offsets, np.int64)
    types, src, dst, rel = c["types"], c["src"], c["dst"], c["rel"]
    R = len(rels)
    g = {k: np.zeros_like(v) for k, v in P.items()}
    dY = np.asarray(dOut, F64)
    if layernorm:
        xhat = (c["Y"] - c["mean"]) * c["rstd"]
        g["ln_gamma"] = np.zeros_like(P["ln_gamma"])
        g["ln_beta"] = np.zeros_like(P["ln_beta"])
        np.add.at(g["ln_gamma"], types, dY * xhat)
        np.add.at(g["ln_beta"], types, dY)
        gx = dY * P["ln_gamma"][types]
        dY = c["rstd"] * (gx - gx.mean(axis=1, keepdims=True) - xhat * (gx * xhat).mean(axis=1, keepdims=True))
    dH = dY.copy()  # residual of Eq. 11
    dU = dY * act_grad(c["U"], act)
    # U = h~ W_agg + b with h~ = sum_r S_r blockdiag(W_msg[r])
    dS = np.zeros((R, N, d), F64)
    for t in range(len(offs) - 1):
        lo, hi = int(offs[t]), int(offs[t + 1])
        g["b_agg"][t] = dU[lo:hi].sum(axis=0)
        ht = np.zeros((hi - lo, d), F64)
        for r, (_, tt) in enumerate(rels):
            if tt == t:
                B = blockdiag(P["W_msg"][r])
                ht += c["Ssum"][r, lo:hi] @ B
                dht_r = dU[lo:hi] @ P["W_agg"][t].T           # gradient of h~ (rows of type t)
                dS[r, lo:hi] = dht_r @ B.T
                GB = c["Ssum"][r, lo:hi].T @ dht_r             # gradient of blockdiag(W_msg[r])
                for s in range(S):
                    cols = slice(s * dh, (s + 1) * dh)
                    g["W_msg"][r, s] = GB[cols, cols]
        g["W_agg"][t] = ht.T @ dU[lo:hi]
    # S_r(j) = sum over r-edges into j of alpha V(i): per edge and head
    alpha, K, V, Qp = c["alpha"], c["K"], c["V"], c["Qp"]
    E = src.shape[0]
    dalpha = np.zeros((E, S), F64)
    dV = np.zeros((N, d), F64)
    for s in range(S):
        cols = slice(s * dh, (s + 1) * dh)
        dSe = dS[rel, dst][:, cols]
        dalpha[:, s] = (dSe * V[src, cols]).sum(axis=1)
        np.add.at(dV[:, cols], src, alpha[:, s:s + 1] * dSe)
    # softmax over the in-edges of each target
    tot = np.zeros((N, S), F64)
    np.add.at(tot, dst, alpha * dalpha)
    dscore = alpha * (dalpha - tot[dst])
    # score = K(i) . Q'_r(j) per head
    dK = np.zeros((N, d), F64)
    dQp = np.zeros((R, N, d), F64)
    for s in range(S):
        cols = slice(s * dh, (s + 1) * dh)
        np.add.at(dK[:, cols], src, dscore[:, s:s + 1] * Qp[rel, dst][:, cols])
        acc = np.zeros((R, N, dh), F64)
        np.add.at(acc, (rel, dst), dscore[:, s:s + 1] * K[src, cols])
        dQp[:, :, cols] = acc
    # Q'_r = Q blockdiag(W_att[r])^T mu[r] / sqrt(d_h)
    Q = c["Q"]
    dQ = np.zeros((N, d), F64)
    for r in range(R):
        B = blockdiag(P["W_att"][r])
        dQ += dQp[r] @ B * c["scale"][r]
        G = dQp[r].T @ Q  # d x d: gradient of (blockdiag(W_att[r])^T scale) is its transpose
        for s in range(S):
            cols = slice(s * dh, (s + 1) * dh)
            g["W_att"][r, s] = G[cols, cols] * c["scale"][r]
        g["mu"][r] = (G * B).sum() / np.sqrt(dh)
    # the three typed linear maps
    for name, dZ in (("K", dK), ("Q", dQ), ("V", dV)):
        W = P["W_" + name]
        for t in range(W.shape[0]):
            m = types == t
            g["W_" + name][t] = H[m].T @ dZ[m]
            g["b_" + name][t] = dZ[m].sum(axis=0)
            dH[m] += dZ[m] @ W[t].T
    return dH, g
