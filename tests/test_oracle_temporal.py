"""Pins of the oracle's temporal module (Eq. 12-13): context attention over the last w states and
the GRU cell.

torch's own GRUCell (a library routine with the same gate convention) pins the cell and, through
autograd, every gradient; the attention is rebuilt with torch.softmax.  Central finite differences
pin the gradient again.  Closed forms: w = 1 (a = 1), r = 0 (uniform weights: the mean of the
context), a saturated update gate (H^t = the weighted history, or = the candidate n), zero weights
(H^t = h / 2).  Planted mistakes must fail.
"""
import numpy as np
import pytest
import torch

from oracle import temporal as OT


def problem(seed, n=40, d=6, w=3, scale=1.0):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((n, d))
    C = rng.standard_normal((w, n, d))
    p = {"Wa": scale * rng.standard_normal((d, d)) / np.sqrt(d), "r": rng.standard_normal(d),
         "W_i": rng.standard_normal((d, 3 * d)) / np.sqrt(d), "W_h": rng.standard_normal((d, 3 * d)) / np.sqrt(d),
         "b_i": 0.2 * rng.standard_normal(3 * d), "b_h": 0.2 * rng.standard_normal(3 * d)}
    return X, C, p


def torch_temporal(X, C, p, dOut):
    d = X.shape[1]
    T = {k: torch.tensor(v, requires_grad=True) for k, v in p.items()}
    Xt = torch.tensor(X, requires_grad=True)
    Ct = torch.tensor(C)  # the context is fixed
    U = torch.tanh(Ct @ T["Wa"])
    e = (U * T["r"]).sum(-1).T  # (n, w)
    a = torch.softmax(e, dim=1)
    Ht = (a.T[:, :, None] * Ct).sum(0)
    cell = torch.nn.GRUCell(d, d).double()
    with torch.no_grad():
        cell.weight_ih.copy_(T["W_i"].T)
        cell.weight_hh.copy_(T["W_h"].T)
        cell.bias_ih.copy_(T["b_i"])
        cell.bias_hh.copy_(T["b_h"])
    out = cell(Xt, Ht)
    (out * torch.tensor(dOut)).sum().backward()
    g = {"dX": Xt.grad.numpy(), "dWa": T["Wa"].grad.numpy(), "dr": T["r"].grad.numpy(),
         "dW_i": cell.weight_ih.grad.numpy().T, "dW_h": cell.weight_hh.grad.numpy().T,
         "db_i": cell.bias_ih.grad.numpy(), "db_h": cell.bias_hh.grad.numpy()}
    # the cell's own parameters carry their gradients; the attention ones flow through Ht
    return out.detach().numpy(), g


@pytest.mark.parametrize("seed,w", [(0, 3), (1, 1), (2, 5)])
def test_matches_torch_gru_cell_and_autograd(seed, w):
    X, C, p = problem(seed, w=w)
    dOut = np.random.default_rng(seed + 50).standard_normal(X.shape)
    want_out, want = torch_temporal(X, C, p, dOut)
    f = OT.temporal_forward(X, C, p)
    assert np.allclose(f["out"], want_out, rtol=0, atol=1e-13)
    g = OT.temporal_backward(X, C, p, dOut)
    for k, v in want.items():
        assert np.allclose(g[k], v, rtol=1e-11, atol=1e-13), k


def test_finite_differences():
    X, C, p = problem(3, n=12, d=4)
    dOut = np.random.default_rng(4).standard_normal(X.shape)
    g = OT.temporal_backward(X, C, p, dOut)
    h = 1e-6
    rng = np.random.default_rng(5)

    def L(X_, p_):
        return float((OT.temporal_forward(X_, C, p_)["out"] * dOut).sum())

    for name in ("Wa", "r", "W_i", "W_h", "b_i", "b_h"):
        for _ in range(4):
            j = tuple(int(rng.integers(0, s)) for s in p[name].shape)
            hi = {k: v.copy() for k, v in p.items()}
            lo = {k: v.copy() for k, v in p.items()}
            hi[name][j] += h
            lo[name][j] -= h
            fd = (L(X, hi) - L(X, lo)) / (2 * h)
            assert abs(fd - g["d" + name][j]) < 1e-7 * max(1.0, abs(fd)), (name, j)
    for _ in range(6):
        j = (int(rng.integers(0, X.shape[0])), int(rng.integers(0, X.shape[1])))
        hi, lo = X.copy(), X.copy()
        hi[j] += h
        lo[j] -= h
        fd = (L(hi, p) - L(lo, p)) / (2 * h)
        assert abs(fd - g["dX"][j]) < 1e-7 * max(1.0, abs(fd))


def test_closed_forms():
    X, C, p = problem(6)
    d = X.shape[1]
    # w = 1: the only weight is 1 and the history is the one context row
    _, _, a, Ht = OT.context_attention(C[:1], p["Wa"], p["r"])
    assert np.all(a == 1.0) and np.array_equal(Ht, C[0])
    # r = 0: uniform weights, the history is the mean of the context
    _, _, a, Ht = OT.context_attention(C, p["Wa"], np.zeros(d))
    assert np.allclose(a, 1.0 / 3.0, rtol=0, atol=1e-15) and np.allclose(Ht, C.mean(axis=0), rtol=0, atol=1e-14)
    # update gate saturated at 1 (b_iz = +80): H^t = the weighted history; at 0: H^t = n
    q = {k: v.copy() for k, v in p.items()}
    q["b_i"][d:2 * d] = 80.0
    f = OT.temporal_forward(X, C, q)
    assert np.allclose(f["out"], f["Ht"], rtol=0, atol=1e-15)
    q["b_i"][d:2 * d] = -80.0
    f = OT.temporal_forward(X, C, q)
    assert np.allclose(f["out"], f["n"], rtol=0, atol=1e-15)
    # zero GRU weights and biases: r = z = 1/2, n = 0, so H^t = h / 2
    q = dict(p, W_i=np.zeros((d, 3 * d)), W_h=np.zeros((d, 3 * d)), b_i=np.zeros(3 * d), b_h=np.zeros(3 * d))
    f = OT.temporal_forward(X, C, q)
    assert np.allclose(f["out"], 0.5 * f["Ht"], rtol=0, atol=1e-15)


def test_bf16_storage_rounds_the_history():
    from hgsynth import bf16_round
    X, C, p = problem(7)
    f = OT.temporal_forward(X, C, p, store="bf16")
    exact = OT.context_attention(C, p["Wa"], p["r"])[3]
    assert np.array_equal(f["Ht"], bf16_round(exact).astype(np.float64))


def test_planted_mistakes_are_caught(monkeypatch):
    X, C, p = problem(8)
    dOut = np.random.default_rng(9).standard_normal(X.shape)
    want_out, want = torch_temporal(X, C, p, dOut)

    def caught():
        f = OT.temporal_forward(X, C, p)
        g = OT.temporal_backward(X, C, p, dOut)
        return not np.allclose(f["out"], want_out, atol=1e-9) or any(
            not np.allclose(g[k], v, rtol=1e-8, atol=1e-10) for k, v in want.items())

    good_soft, good_sig = OT.softmax_rows, OT.sigmoid
    # softmax over the nodes instead of over the w states
    monkeypatch.setattr(OT, "softmax_rows", lambda e: good_soft(e.T).T)
    assert caught()
    monkeypatch.setattr(OT, "softmax_rows", good_soft)
    # a gate with the wrong sign
    monkeypatch.setattr(OT, "sigmoid", lambda x: good_sig(-np.asarray(x)))
    assert caught()
    monkeypatch.setattr(OT, "sigmoid", good_sig)
    # reset gate applied to h before its product with W_hn
    good_cell = OT.gru_cell

    def cell_wrong(x, h, q):
        out = good_cell(x, h, q)
        d = x.shape[1]
        gi = x @ q["W_i"] + q["b_i"]
        n = np.tanh(gi[:, 2 * d:] + (out["r"] * h) @ q["W_h"][:, 2 * d:] + q["b_h"][2 * d:])
        return dict(out, n=n, out=(1 - out["z"]) * n + out["z"] * h)

    monkeypatch.setattr(OT, "gru_cell", cell_wrong)
    assert caught()
    monkeypatch.setattr(OT, "gru_cell", good_cell)
    assert not caught()
