"""CPU oracle of the temporal module.  TEST INFRASTRUCTURE ONLY.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg import this module; the
product path never calls it and shares no code with it.  Plain numpy in fp64.

What is computed (Section 3.2, "Temporal Graph Learning", Eq. 12-13), per node, from its spatial
embedding x = h^t (the last layer's output at the current snapshot) and its context
C = [H^{t-w}; ...; H^{t-1}] (the node's final states at the w previous snapshots, rows c_1 .. c_w):

* context_attention  Eq. 12: u_k = tanh(c_k W_a) (W_a = Q^T, so the k-th column of Q C^T is u_k),
                     e_k = r . u_k, a = softmax_k(e), and the weighted history
                     H~^{t-1} = sum_k a_k c_k.
* gru_cell ......... Eq. 13: H^t = GRU(x, H~^{t-1}) with the gates
                       r = sigmoid(x W_ir + b_ir + h W_hr + b_hr)
                       z = sigmoid(x W_iz + b_iz + h W_hz + b_hz)
                       n = tanh(x W_in + b_in + r * (h W_hn + b_hn))
                       H^t = (1 - z) * n + z * h          (h = H~^{t-1})
* temporal_backward  the chain rule of both, step by step.

Readings where the paper is silent or ambiguous (listed again in the design notes):
  Q multiplies the context from the left in Eq. 12 (Q C^T with the states as rows of C); it is
  stored transposed, W_a = Q^T (d x d, input x output), so u_k = tanh(c_k W_a);
  the GRU is the common cell with the reset gate applied to (h W_hn + b_hn); its weights are stored
  as W_i = [W_ir | W_iz | W_in] and W_h = [W_hr | W_hz | W_hn] (d x 3d each, input x output) with
  biases b_i, b_h (3d each);
  the context rows are earlier snapshots' outputs, held fixed during the step (no gradient flows
  into them: truncated backpropagation through time);
  w = 3 (Section 4.1); a node with fewer than w earlier states is not distinguished (the context
  holds w rows for every node, zero rows where a state does not exist).
  store="bf16": the weighted history H~ is rounded to bf16 before the GRU (the tensor that the
  GRU's matrix product reads), so both sides take the gates' decisions from the same inputs; all
  other arithmetic stays fp64.
"""
from __future__ import annotations

import numpy as np

from .hg_oracle import round_bf16

F64 = np.float64


def sigmoid(x) -> np.ndarray:
    x = np.asarray(x, F64)
    e = np.exp(-np.abs(x))
    return np.where(x >= 0.0, 1.0 / (1.0 + e), e / (1.0 + e))


def softmax_rows(e: np.ndarray) -> np.ndarray:
    """Softmax over the last axis (max subtracted first)."""
    m = e.max(axis=-1, keepdims=True)
    p = np.exp(e - m)
    return p / p.sum(axis=-1, keepdims=True)


def context_attention(C, Wa, rvec) -> tuple:
    """Eq. 12 for every node.  C: (w, n, d) context rows; returns (U (w, n, d), e (n, w),
    a (n, w), Ht (n, d))."""
    C = np.asarray(C, F64)
    U = np.tanh(C @ np.asarray(Wa, F64))
    e = np.einsum("knd,d->nk", U, np.asarray(rvec, F64))
    a = softmax_rows(e)
    Ht = np.einsum("nk,knd->nd", a, C)
    return U, e, a, Ht


def gru_cell(x, h, p: dict) -> dict:
    """Eq. 13 (gates as in the module docstring).  x, h: (n, d)."""
    x = np.asarray(x, F64)
    h = np.asarray(h, F64)
    d = x.shape[1]
    gi = x @ np.asarray(p["W_i"], F64) + np.asarray(p["b_i"], F64)
    gh = h @ np.asarray(p["W_h"], F64) + np.asarray(p["b_h"], F64)
    r = sigmoid(gi[:, :d] + gh[:, :d])
    z = sigmoid(gi[:, d:2 * d] + gh[:, d:2 * d])
    hn = gh[:, 2 * d:]
    n = np.tanh(gi[:, 2 * d:] + r * hn)
    out = (1.0 - z) * n + z * h
    return {"r": r, "z": z, "n": n, "hn": hn, "out": out}


def temporal_forward(X, C, p: dict, store: str = "f64") -> dict:
    """H^t from the spatial embeddings X (n, d) and the context C (w, n, d).  p: Wa, r (attention),
    W_i, W_h, b_i, b_h (GRU)."""
    U, e, a, Ht = context_attention(C, p["Wa"], p["r"])
    if store == "bf16":
        Ht = round_bf16(Ht)
    g = gru_cell(X, Ht, p)
    return {"U": U, "e": e, "a": a, "Ht": Ht, **g}


def temporal_backward(X, C, p: dict, dOut, store: str = "f64") -> dict:
    """Gradients of <dOut, H^t> with respect to X and every parameter (the context is fixed)."""
    X = np.asarray(X, F64)
    C = np.asarray(C, F64)
    dOut = np.asarray(dOut, F64)
    f = temporal_forward(X, C, p, store)
    d = X.shape[1]
    r, z, n, hn, h = f["r"], f["z"], f["n"], f["hn"], f["Ht"]
    # H^t = (1 - z) n + z h
    dn = dOut * (1.0 - z)
    dz = dOut * (h - n)
    dh = dOut * z
    # n = tanh(gi_n + r hn)
    dpre_n = dn * (1.0 - n * n)
    dr = dpre_n * hn
    dhn = dpre_n * r
    dpre_r = dr * r * (1.0 - r)
    dpre_z = dz * z * (1.0 - z)
    dgi = np.concatenate([dpre_r, dpre_z, dpre_n], axis=1)  # gradient of x W_i + b_i
    dgh = np.concatenate([dpre_r, dpre_z, dhn], axis=1)     # gradient of h W_h + b_h
    W_i = np.asarray(p["W_i"], F64)
    W_h = np.asarray(p["W_h"], F64)
    out = {"dX": dgi @ W_i.T, "dW_i": X.T @ dgi, "db_i": dgi.sum(axis=0), "dW_h": h.T @ dgh,
           "db_h": dgh.sum(axis=0)}
    dh = dh + dgh @ W_h.T  # total gradient of the weighted history H~
    # H~ = sum_k a_k c_k, a = softmax(e), e_k = r . u_k, u_k = tanh(c_k W_a)
    U, a = f["U"], f["a"]
    da = np.einsum("nd,knd->nk", dh, C)
    de = a * (da - (a * da).sum(axis=1, keepdims=True))
    rvec = np.asarray(p["r"], F64)
    out["dr"] = np.einsum("nk,knd->d", de, U)
    dU = de.T[:, :, None] * rvec[None, None, :]      # (w, n, d)
    dpreU = dU * (1.0 - U * U)
    out["dWa"] = np.einsum("knd,kne->de", C, dpreU)
    out["out"] = f["out"]
    assert out["dX"].shape == (X.shape[0], d)
    return out
