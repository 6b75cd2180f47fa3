"""CPU oracle of the prediction head and the joint objective.  TEST INFRASTRUCTURE ONLY.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg import this module; the
product path never calls it and shares no code with it.  Plain numpy in fp64.

What is computed (Section 3.4, Eq. 18-20 and the MeanAgg / MLP / loss steps of Algorithm 1):

* final_embedding .. MeanAgg: the final embedding of a node is the mean of its replicas.  A row of
                     this subgraph's output H that also lives in a second view (row idx_b[k] of
                     H_rep for row idx_a[k] of H) becomes (H[idx_a[k]] + H_rep[idx_b[k]]) / 2;
                     every other row is H itself.
* mlp_forward ...... Eq. 18: z = W_2 sigma(W_1 h + b_1) + b_2 per labelled row, sigma = ReLU,
                     hidden width d, one output logit.
* bce_terms ........ Eq. 19 per row with the predicted probability p = 1 / (1 + exp(-z)):
                     -[y log p + (1 - y) log(1 - p)], written with log p = -softplus(-z) and
                     log(1 - p) = -softplus(z), which is the same quantity without overflow.
* head_loss ........ L_BCE = mean of the terms over the labelled rows; Eq. 20:
                     L_total = L_BCE + lambda_CCA L_CCA.
* head_backward .... the chain rule of head_loss, step by step: dz = (p - y) / N_m, then through
                     the MLP, then MeanAgg splits a replicated row's gradient in halves.

Readings where the paper is silent or ambiguous (listed again in the design notes):
  the MLP output is a logit and the probability of Eq. 19 is its logistic sigmoid; sigma of
  Eq. 18 is ReLU and the hidden width equals d; W_1 is stored d x d (input x hidden) and applied
  as h W_1 to a row h, W_2 is a vector of d entries;
  MeanAgg averages the replicas present in the step (this subgraph's row and, for an overlap
  node, the second view's row); a detached second view receives no gradient;
  N_m is the number of labelled rows handed to the head; labels may be fractional (y in [0, 1]);
  store="bf16": the averaged rows are rounded to bf16 (round to nearest even), as the bf16 kernel
  stores them for the weight gradient; all other arithmetic stays fp64.  (The kernel's
  pre-activation uses the unrounded mean of the two stored rows; the GPU tests compare with the
  plain definition, store="f64".)
"""
from __future__ import annotations

import numpy as np

from .hg_oracle import round_bf16

F64 = np.float64


def final_embedding(H, idx_a, H_rep, idx_b, store: str = "f64") -> np.ndarray:
    """MeanAgg of Algorithm 1 over the two replicas of the overlap rows (fp64, all rows of H)."""
    Hf = np.array(H, F64, copy=True)
    idx_a = np.asarray(idx_a, np.int64)
    if idx_a.size:
        m = 0.5 * (np.asarray(H, F64)[idx_a] + np.asarray(H_rep, F64)[np.asarray(idx_b, np.int64)])
        Hf[idx_a] = round_bf16(m) if store == "bf16" else m
    return Hf


def mlp_forward(Hrows, W1, b1, w2, b2) -> tuple:
    """Eq. 18 on a block of rows: A = Hrows W_1 + b_1, R = ReLU(A), z = R w_2 + b_2.
    Returns (A, R, z)."""
    A = np.asarray(Hrows, F64) @ np.asarray(W1, F64) + np.asarray(b1, F64)
    R = np.where(A > 0.0, A, 0.0)
    z = R @ np.asarray(w2, F64).reshape(-1) + float(np.asarray(b2, F64).reshape(-1)[0])
    return A, R, z


def softplus(x) -> np.ndarray:
    """log(1 + exp(x)) evaluated as max(x, 0) + log1p(exp(-|x|))."""
    x = np.asarray(x, F64)
    return np.maximum(x, 0.0) + np.log1p(np.exp(-np.abs(x)))


def bce_terms(z, y) -> np.ndarray:
    """Per-row binary cross-entropy of Eq. 19 for logit z and label y:
    y * softplus(-z) + (1 - y) * softplus(z) = -[y log p + (1 - y) log(1 - p)], p = sigmoid(z)."""
    z = np.asarray(z, F64)
    y = np.asarray(y, F64)
    return y * softplus(-z) + (1.0 - y) * softplus(z)


def sigmoid(z) -> np.ndarray:
    z = np.asarray(z, F64)
    e = np.exp(-np.abs(z))
    return np.where(z >= 0.0, 1.0 / (1.0 + e), e / (1.0 + e))


def head_loss(H, idx_a, H_rep, idx_b, lab_idx, lab_y, params: dict, cca_loss: float | None = None,
              lambda_cca: float = 0.1, store: str = "f64") -> dict:
    """L_BCE over the labelled rows (Eq. 18-19 on the MeanAgg embedding) and L_total (Eq. 20).
    params: W1 (d x d), b1 (d), w2 (d), b2 (1).  cca_loss None: L_total = L_BCE."""
    Hf = final_embedding(H, idx_a, H_rep, idx_b, store)
    lab_idx = np.asarray(lab_idx, np.int64)
    _, _, z = mlp_forward(Hf[lab_idx], params["W1"], params["b1"], params["w2"], params["b2"])
    n = lab_idx.shape[0]
    bce = float(bce_terms(z, lab_y).sum() / n) if n else 0.0
    total = bce + (lambda_cca * float(cca_loss) if cca_loss is not None else 0.0)
    return {"total": total, "bce": bce, "logits": z}


def head_backward(H, idx_a, H_rep, idx_b, lab_idx, lab_y, params: dict, dloss: float = 1.0,
                  store: str = "f64") -> dict:
    """Gradient of dloss * L_BCE with respect to W1, b1, w2, b2 and to the rows of H and H_rep
    (full-shape arrays, non-zero only on labelled rows and their replicas)."""
    Hf = final_embedding(H, idx_a, H_rep, idx_b, store)
    lab_idx = np.asarray(lab_idx, np.int64)
    n = lab_idx.shape[0]
    d = Hf.shape[1]
    W1 = np.asarray(params["W1"], F64)
    w2 = np.asarray(params["w2"], F64).reshape(-1)
    Hl = Hf[lab_idx]
    A, R, z = mlp_forward(Hl, W1, params["b1"], w2, params["b2"])
    # dL/dz of the mean BCE: (sigmoid(z) - y) / N_m
    dz = dloss * (sigmoid(z) - np.asarray(lab_y, F64)) / max(n, 1)
    dR = np.outer(dz, w2)
    dA = np.where(A > 0.0, dR, 0.0)
    out = {
        "dW1": Hl.T @ dA,
        "db1": dA.sum(axis=0),
        "dw2": R.T @ dz,
        "db2": np.array([dz.sum()]),
    }
    dHl = dA @ W1.T  # gradient at the final embedding of each labelled row
    dHf = np.zeros((Hf.shape[0], d), F64)
    dHf[lab_idx] = dHl
    # MeanAgg: a replicated row passes half of its gradient to each replica
    dH = dHf.copy()
    dH_rep = np.zeros(np.shape(H_rep), F64) if H_rep is not None else None
    idx_a = np.asarray(idx_a, np.int64)
    if idx_a.size:
        idx_b = np.asarray(idx_b, np.int64)
        dH[idx_a] = 0.5 * dHf[idx_a]
        dH_rep[idx_b] = 0.5 * dHf[idx_a]
    out["dH"] = dH
    out["dH_rep"] = dH_rep
    out["logits"] = z
    return out
