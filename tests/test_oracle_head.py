"""Pins of the oracle's prediction head and joint objective (Eq. 18-20, MeanAgg of Algorithm 1).

Closed forms: zero weights give L_BCE = log 2 and dL/db2 = 1/2 - mean(y); a head whose output does
not depend on the row gives the two-class cross-entropy of one logit (log(4/3) and log 4 at
z = log 3).  Eq. 19 in its probability form, and torch's binary cross-entropy, pin the stable
form.  torch autograd (fp64) on an independent dense formulation pins the loss and every
gradient; central finite differences pin it again.  MeanAgg special cases (identical replicas, no
replica, the halves of a replicated row's gradient summing to the unsplit gradient), the joint
objective, order invariance, bf16 storage of the averaged rows, and planted mistakes.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from oracle import head as OH


def problem(seed, N=120, d=6, n_rep=30, n_lab=40, rows_rep=90, frac_y=False):
    rng = np.random.default_rng(seed)
    H = rng.standard_normal((N, d))
    H_rep = rng.standard_normal((rows_rep, d))
    idx_a = np.sort(rng.choice(N, n_rep, replace=False))
    idx_b = rng.choice(rows_rep, n_rep, replace=False)
    lab = np.sort(rng.choice(N, n_lab, replace=False))
    y = rng.random(n_lab) if frac_y else (rng.random(n_lab) < 0.3).astype(np.float64)
    p = {"W1": rng.standard_normal((d, d)) / math.sqrt(d), "b1": 0.3 * rng.standard_normal(d),
         "w2": rng.standard_normal(d) / math.sqrt(d), "b2": np.array([0.2])}
    return H, idx_a, H_rep, idx_b, lab, y, p


def torch_head(H, idx_a, H_rep, idx_b, lab, y, p):
    """Dense fp64 formulation with torch ops and torch's BCE-with-logits; returns the loss and the
    autograd gradients."""
    t = {k: torch.tensor(np.asarray(v, np.float64), requires_grad=True) for k, v in p.items()}
    Ht = torch.tensor(H, requires_grad=True)
    Rt = torch.tensor(H_rep, requires_grad=True)
    ia = torch.tensor(np.asarray(idx_a, np.int64))
    ib = torch.tensor(np.asarray(idx_b, np.int64))
    mask = torch.zeros(H.shape[0], 1, dtype=torch.float64)
    mask[ia] = 1.0
    other = torch.zeros_like(Ht).index_put((ia,), Rt[ib])  # the second replica, on its rows
    Hf = Ht * (1 - mask) + 0.5 * (Ht + other) * mask
    x = Hf[torch.tensor(np.asarray(lab, np.int64))]
    z = torch.relu(x @ t["W1"] + t["b1"]) @ t["w2"] + t["b2"]
    loss = torch.nn.functional.binary_cross_entropy_with_logits(z, torch.tensor(np.asarray(y, np.float64)))
    loss.backward()
    g = {"d" + k: v.grad.numpy() for k, v in t.items()}
    g["dH"], g["dH_rep"] = Ht.grad.numpy(), Rt.grad.numpy()
    return float(loss.detach()), z.detach().numpy(), g


def test_zero_weights_give_log2():
    H, ia, Hr, ib, lab, y, p = problem(0)
    zero = {k: np.zeros_like(v) for k, v in p.items()}
    out = OH.head_loss(H, ia, Hr, ib, lab, y, zero)
    assert abs(out["bce"] - math.log(2.0)) < 1e-15
    g = OH.head_backward(H, ia, Hr, ib, lab, y, zero)
    assert abs(g["db2"][0] - (0.5 - y.mean())) < 1e-15
    for k in ("dW1", "db1", "dw2", "dH", "dH_rep"):
        assert np.abs(g[k]).max() == 0.0, k


@pytest.mark.parametrize("label,want", [(1.0, math.log(4.0 / 3.0)), (0.0, math.log(4.0))])
def test_row_independent_logit_closed_form(label, want):
    # W1 = 0: every row has the hidden layer relu(b1), so z = relu(b1) . w2 + b2 for all rows
    H, ia, Hr, ib, lab, _, p = problem(1)
    d = H.shape[1]
    q = {"W1": np.zeros((d, d)), "b1": np.r_[1.0, -2.0, np.zeros(d - 2)], "w2": np.r_[0.5, 7.0, np.zeros(d - 2)],
         "b2": np.array([math.log(3.0) - 0.5])}
    y = np.full(len(lab), label)
    out = OH.head_loss(H, ia, Hr, ib, lab, y, q)
    assert np.allclose(out["logits"], math.log(3.0), rtol=0, atol=1e-15)
    assert abs(out["bce"] - want) < 1e-14
    # p = 3/4, so dL/db2 = (3/4 - y); dL/dw2 = (3/4 - y) relu(b1)
    g = OH.head_backward(H, ia, Hr, ib, lab, y, q)
    assert abs(g["db2"][0] - (0.75 - label)) < 1e-14
    assert np.allclose(g["dw2"], (0.75 - label) * np.maximum(q["b1"], 0), atol=1e-14)


def test_bce_matches_probability_form():
    rng = np.random.default_rng(2)
    z = rng.uniform(-12, 12, 500)
    y = rng.random(500)
    p = 1.0 / (1.0 + np.exp(-z))
    direct = -(y * np.log(p) + (1 - y) * np.log(1 - p))
    assert np.allclose(OH.bce_terms(z, y), direct, rtol=1e-9, atol=1e-12)
    lib = torch.nn.functional.binary_cross_entropy(torch.tensor(p), torch.tensor(y), reduction="none").numpy()
    assert np.allclose(OH.bce_terms(z, y), lib, rtol=1e-9, atol=1e-12)
    # far tails stay finite: z = +-800 gives 0 and 800
    assert OH.bce_terms(np.array([800.0]), np.array([1.0]))[0] == 0.0
    assert OH.bce_terms(np.array([-800.0]), np.array([1.0]))[0] == 800.0


@pytest.mark.parametrize("seed,frac", [(3, False), (4, True), (5, False)])
def test_loss_and_gradients_match_torch_autograd(seed, frac):
    H, ia, Hr, ib, lab, y, p = problem(seed, frac_y=frac)
    loss, z, g = torch_head(H, ia, Hr, ib, lab, y, p)
    out = OH.head_loss(H, ia, Hr, ib, lab, y, p)
    assert abs(out["bce"] - loss) < 1e-13
    assert np.allclose(out["logits"], z, rtol=0, atol=1e-13)
    mine = OH.head_backward(H, ia, Hr, ib, lab, y, p)
    for k in ("dW1", "db1", "dw2", "db2", "dH", "dH_rep"):
        assert np.allclose(mine[k], np.asarray(g[k]).reshape(mine[k].shape), rtol=1e-11, atol=1e-14), k


def test_finite_differences():
    H, ia, Hr, ib, lab, y, p = problem(6, N=40, d=4, n_rep=10, n_lab=15, rows_rep=30)
    g = OH.head_backward(H, ia, Hr, ib, lab, y, p, dloss=1.0)
    h = 1e-6
    rng = np.random.default_rng(7)

    def loss_with(**kw):
        args = dict(H=H, H_rep=Hr, p=p)
        args.update(kw)
        return OH.head_loss(args["H"], ia, args["H_rep"], ib, lab, y, args["p"])["bce"]

    for name in ("W1", "b1", "w2", "b2"):
        for _ in range(4):
            j = tuple(rng.integers(0, s) for s in p[name].shape)
            hi, lo = {k: v.copy() for k, v in p.items()}, {k: v.copy() for k, v in p.items()}
            hi[name][j] += h
            lo[name][j] -= h
            fd = (loss_with(p=hi) - loss_with(p=lo)) / (2 * h)
            assert abs(fd - g["d" + name][j]) < 1e-7 * max(1.0, abs(fd)), (name, j)
    for key, arr, rows in (("dH", H, lab), ("dH_rep", Hr, ib)):
        for r in rows[:5]:
            c = int(rng.integers(0, arr.shape[1]))
            hi, lo = arr.copy(), arr.copy()
            hi[r, c] += h
            lo[r, c] -= h
            kw_hi = {"H" if key == "dH" else "H_rep": hi}
            kw_lo = {"H" if key == "dH" else "H_rep": lo}
            fd = (loss_with(**kw_hi) - loss_with(**kw_lo)) / (2 * h)
            assert abs(fd - g[key][r, c]) < 1e-7 * max(1.0, abs(fd)), (key, r, c)


def test_meanagg_special_cases():
    H, ia, Hr, ib, lab, y, p = problem(8)
    # no replica: H unchanged, all the gradient stays in H
    assert np.array_equal(OH.final_embedding(H, ia[:0], Hr, ib[:0]), H)
    # identical replicas: the mean is the row itself
    same = Hr.copy()
    same[ib] = H[ia]
    assert np.allclose(OH.final_embedding(H, ia, same, ib), H, rtol=0, atol=1e-15)
    # the halves of a replicated row's gradient add up to the gradient without replicas
    g_rep = OH.head_backward(H, ia, same, ib, lab, y, p)
    g_one = OH.head_backward(H, ia[:0], same, ib[:0], lab, y, p)
    total = g_rep["dH"].copy()
    total[ia] += g_rep["dH_rep"][ib]
    assert np.allclose(total, g_one["dH"], rtol=0, atol=1e-15)
    assert np.array_equal(g_rep["dW1"], g_one["dW1"])
    # unlabelled rows and their replicas get no gradient
    unl = np.setdiff1d(np.arange(H.shape[0]), lab)
    assert np.abs(g_rep["dH"][unl]).max() == 0.0


def test_joint_objective():
    H, ia, Hr, ib, lab, y, p = problem(9, n_rep=40)
    L_cca = oracle.align_forward(H, ia, Hr, ib, lambda_n=2e-4, eps=1e-8)[0]
    out = OH.head_loss(H, ia, Hr, ib, lab, y, p, cca_loss=L_cca, lambda_cca=0.1)
    assert out["total"] == out["bce"] + 0.1 * L_cca
    assert OH.head_loss(H, ia, Hr, ib, lab, y, p)["total"] == out["bce"]


def test_order_invariance_and_dloss_scaling():
    H, ia, Hr, ib, lab, y, p = problem(10)
    perm = np.random.default_rng(11).permutation(len(lab))
    a = OH.head_backward(H, ia, Hr, ib, lab, y, p, dloss=1.0)
    b = OH.head_backward(H, ia, Hr, ib, lab[perm], y[perm], p, dloss=1.0)
    c = OH.head_backward(H, ia, Hr, ib, lab, y, p, dloss=-2.5)
    for k in ("dW1", "db1", "dw2", "db2", "dH", "dH_rep"):
        assert np.allclose(a[k], b[k], rtol=1e-12, atol=1e-16), k
        assert np.allclose(c[k], -2.5 * a[k], rtol=1e-13, atol=1e-16), k


def test_bf16_storage_of_averaged_rows():
    from hgsynth import bf16_round
    H, ia, Hr, ib, lab, y, p = problem(12)
    H, Hr = bf16_round(H).astype(np.float64), bf16_round(Hr).astype(np.float64)
    Hf = OH.final_embedding(H, ia, Hr, ib, store="bf16")
    others = np.setdiff1d(np.arange(H.shape[0]), ia)
    assert np.array_equal(Hf[others], H[others])
    exact = 0.5 * (H[ia] + Hr[ib])
    assert np.array_equal(Hf[ia], bf16_round(exact).astype(np.float64))
    assert np.abs(Hf[ia] - exact).max() <= np.abs(exact).max() * 2.0 ** -8


def test_planted_mistakes_are_caught(monkeypatch):
    H, ia, Hr, ib, lab, y, p = problem(13)
    loss, _, g = torch_head(H, ia, Hr, ib, lab, y, p)

    def caught():
        mine = OH.head_backward(H, ia, Hr, ib, lab, y, p)
        out = OH.head_loss(H, ia, Hr, ib, lab, y, p)
        return abs(out["bce"] - loss) > 1e-9 or any(
            not np.allclose(mine[k], np.asarray(g[k]).reshape(mine[k].shape), rtol=1e-9, atol=1e-12)
            for k in ("dW1", "db1", "dw2", "db2", "dH", "dH_rep"))

    good_fe, good_sig, good_sp = OH.final_embedding, OH.sigmoid, OH.softplus
    # MeanAgg that sums instead of averaging
    monkeypatch.setattr(OH, "final_embedding", lambda H_, a, R, b, store="f64": good_fe(H_, a, R, b, store) + (
        np.isin(np.arange(H_.shape[0]), a)[:, None] * good_fe(H_, a, R, b, store)))
    assert caught()
    monkeypatch.setattr(OH, "final_embedding", good_fe)
    # a sign error in dz
    monkeypatch.setattr(OH, "sigmoid", lambda z: 1.0 - good_sig(z))
    assert caught()
    monkeypatch.setattr(OH, "sigmoid", good_sig)
    # softplus missing its log1p term
    monkeypatch.setattr(OH, "softplus", lambda x: np.maximum(np.asarray(x, np.float64), 0.0))
    assert caught()
    monkeypatch.setattr(OH, "softplus", good_sp)
    assert not caught()
