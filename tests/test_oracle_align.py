"""Pins of the oracle's alignment loss (Eq. 14-17) and its gradient (CPU only).

With eps = 0 and the population standard deviation, the standardised columns have unit norm, so
Z^T Z is the Pearson correlation matrix: L_inv = sum_k 2 (1 - rho_k(a, b)) and L_dec = sum over
both views of sum_{k != l} rho_kl^2.  numpy.corrcoef supplies rho independently.  Special cases:
d = 1, identical views, centred orthonormal columns (QR), invariance to per-column affine maps,
hand-derived values, torch autograd and finite differences for the gradient, planted mistakes.
"""
import json
import os

import numpy as np
import pytest
import torch

import oracle
from oracle import hg_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def views(seed, n=200, d=5, N=260):
    rng = np.random.default_rng(seed)
    Ha = rng.standard_normal((N, d)) * rng.uniform(0.5, 3, d) + rng.uniform(-2, 2, d)
    Hb = 0.6 * Ha + 0.8 * rng.standard_normal((N, d))
    idx_a = np.sort(rng.choice(N, n, replace=False))
    idx_b = rng.permutation(idx_a)
    Hb = Hb[rng.permutation(N)]
    return Ha, idx_a, Hb, idx_b


def closed_form(A, B, lam):
    d = A.shape[1]
    c = np.corrcoef(np.concatenate([A, B], axis=1), rowvar=False)
    rho_ab = np.diag(c[:d, d:])
    ca, cb = c[:d, :d], c[d:, d:]
    off = ~np.eye(d, dtype=bool)
    l_inv = float(np.sum(2 * (1 - rho_ab)))
    l_dec = float(np.sum(ca[off] ** 2) + np.sum(cb[off] ** 2))
    return l_inv + lam * l_dec, l_inv, l_dec


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_loss_matches_pearson_closed_form(seed):
    Ha, ia, Hb, ib = views(seed)
    got = oracle.align_forward(Ha, ia, Hb, ib, lambda_n=2e-4, eps=0.0)
    want = closed_form(Ha[ia], Hb[ib], 2e-4)
    assert np.allclose(got, want, rtol=1e-12, atol=1e-12)


def test_d1_and_identical_views():
    Ha, ia, Hb, ib = views(4, d=1)
    L, l_inv, l_dec = oracle.align_forward(Ha, ia, Hb, ib, eps=0.0)
    rho = np.corrcoef(Ha[ia, 0], Hb[ib, 0])[0, 1]
    assert np.isclose(l_inv, 2 * (1 - rho), rtol=1e-12) and abs(l_dec) < 1e-20
    Ha, ia, _, _ = views(5)
    L, l_inv, _ = oracle.align_forward(Ha, ia, Ha, ia, eps=0.0)
    assert abs(l_inv) < 1e-24
    dA, dB = oracle.align_backward(Ha, ia, Ha, ia, lambda_n=0.0, eps=0.0)
    assert np.abs(dA).max() < 1e-12 and np.abs(dB).max() < 1e-12


def test_orthonormal_columns_have_no_decorrelation_loss():
    rng = np.random.default_rng(6)
    n, d = 64, 6
    X = rng.standard_normal((n, d))
    X -= X.mean(axis=0)
    Q, _ = np.linalg.qr(X)  # centred, orthonormal columns
    Q -= Q.mean(axis=0)
    idx = np.arange(n)
    _, _, l_dec = oracle.align_forward(Q, idx, Q, idx, eps=0.0)
    assert abs(l_dec) < 1e-20


def test_invariant_to_column_affine_maps():
    Ha, ia, Hb, ib = views(7)
    rng = np.random.default_rng(8)
    a, c = rng.uniform(0.2, 5, Ha.shape[1]), rng.uniform(-3, 3, Ha.shape[1])
    L0 = oracle.align_forward(Ha, ia, Hb, ib, eps=0.0)
    L1 = oracle.align_forward(Ha * a + c, ia, Hb, ib, eps=0.0)
    assert np.allclose(L0, L1, rtol=1e-10)


def test_golden_hand_example():
    gd = json.load(open(os.path.join(GOLDEN, "cca_tiny.json")))
    A, B = np.array(gd["A"], float), np.array(gd["B"], float)
    idx = np.arange(A.shape[0])
    L, l_inv, l_dec = oracle.align_forward(A, idx, B, idx, gd["lambda_n"], gd["eps"])
    assert np.isclose(l_inv, gd["L_inv"], rtol=1e-13) and np.isclose(l_dec, gd["L_dec"], rtol=1e-13)
    assert np.isclose(L, gd["L"], rtol=1e-13)


def torch_loss(Ha, ia, Hb, ib, lam, eps):
    A = torch.tensor(Ha, requires_grad=True)
    B = torch.tensor(Hb, requires_grad=True)

    def z(X):
        n = X.shape[0]
        return (X - X.mean(0)) / (torch.sqrt(X.var(0, unbiased=False) + eps) * np.sqrt(n))

    Za, Zb = z(A[torch.tensor(ia)]), z(B[torch.tensor(ib)])
    I = torch.eye(Ha.shape[1], dtype=torch.float64)
    L = ((Za - Zb) ** 2).sum() + lam * (((Za.T @ Za - I) ** 2).sum() + ((Zb.T @ Zb - I) ** 2).sum())
    return L, A, B


@pytest.mark.parametrize("eps", [0.0, 1e-3])
def test_gradient_matches_torch_autograd(eps):
    Ha, ia, Hb, ib = views(9, n=50, d=4, N=70)
    lam, dloss = 0.05, 0.1
    L, A, B = torch_loss(Ha, ia, Hb, ib, lam, eps)
    assert np.isclose(L.item(), oracle.align_forward(Ha, ia, Hb, ib, lam, eps)[0], rtol=1e-12)
    (dloss * L).backward()
    dA, dB = oracle.align_backward(Ha, ia, Hb, ib, lam, eps, dloss)
    assert np.allclose(dA, A.grad.numpy(), rtol=0, atol=1e-12)
    assert np.allclose(dB, B.grad.numpy(), rtol=0, atol=1e-12)


def test_gradient_finite_differences():
    Ha, ia, Hb, ib = views(10, n=30, d=3, N=40)
    lam, eps = 0.3, 1e-4
    dA, dB = oracle.align_backward(Ha, ia, Hb, ib, lam, eps)
    rng = np.random.default_rng(11)
    h = 1e-6
    for which in "ab":
        V = rng.standard_normal(Ha.shape)
        if which == "a":
            fd = (oracle.align_forward(Ha + h * V, ia, Hb, ib, lam, eps)[0]
                  - oracle.align_forward(Ha - h * V, ia, Hb, ib, lam, eps)[0]) / (2 * h)
            an = float((dA * V).sum())
        else:
            fd = (oracle.align_forward(Ha, ia, Hb + h * V, ib, lam, eps)[0]
                  - oracle.align_forward(Ha, ia, Hb - h * V, ib, lam, eps)[0]) / (2 * h)
            an = float((dB * V).sum())
        assert abs(fd - an) <= 1e-6 * max(1.0, abs(an))


# ---------------------------------------------------------------------------------------------
# planted mistakes
# ---------------------------------------------------------------------------------------------
def test_planted_sample_std_is_caught(monkeypatch):
    def standardise_sample_std(X, eps):
        n = X.shape[0]
        mu = X.mean(axis=0)
        s = np.sqrt(((X - mu) ** 2).sum(axis=0) / (n - 1) + eps)
        return (X - mu) / (s * np.sqrt(n)), mu, s

    monkeypatch.setattr(O, "standardise", standardise_sample_std)
    Ha, ia, Hb, ib = views(0)
    got = O.align_forward(Ha, ia, Hb, ib, lambda_n=2e-4, eps=0.0)
    want = closed_form(Ha[ia], Hb[ib], 2e-4)
    assert abs(got[0] - want[0]) > 1e-3 * abs(want[0])


def test_planted_gradient_sign_is_caught():
    Ha, ia, Hb, ib = views(9, n=50, d=4, N=70)
    lam = 0.05
    L, A, B = torch_loss(Ha, ia, Hb, ib, lam, 0.0)
    L.backward()
    # a copy of the backward that forgets the minus sign of the invariance term for view b
    Za, _, _ = O.standardise(Hb[ib] * 0 + Ha[ia], 0.0)
    Zb, _, _ = O.standardise(Hb[ib], 0.0)
    Gb = 2.0 * (Za - Zb) + 4.0 * lam * Zb @ (Zb.T @ Zb - np.eye(4))
    dB = np.zeros_like(Hb)
    dB[ib] = O._standardise_backward(Hb[ib], Gb, 0.0)
    assert np.abs(dB - B.grad.numpy()).max() > 1e-3
