"""Pins of the oracle's layer forward / backward (CPU only).

* dense normalised adjacency built with Python loops, multiplied with numpy (aggregation);
* a dense torch fp64 formulation with torch's own layer_norm and autograd (forward and every
  gradient), an independent library path;
* central finite differences in fp64;
* invariants: rows of the mean operator sum to one, permutation equivariance within node
  types, star graph, single edge, W_r = 0;
* hand-derived values (tests/golden/layer_tiny.json);
* planted mistakes in copies of oracle functions must be caught by these pins.
"""
import json
import os

import numpy as np
import pytest
import torch

import oracle
from oracle import hg_oracle as O
from hgsynth import RELATIONS

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def small_graph(seed, n_user=24, n_risk=9, num_rels=5, num_edges=300, d=6):
    rng = np.random.default_rng(seed)
    rels = RELATIONS[:num_rels]
    offs = np.array([0, n_user, n_user + n_risk], np.int64)
    size = (n_user, n_risk)
    r = rng.integers(0, num_rels, num_edges)
    # skewed sources and destinations so that some rows are empty and some are hubs
    pick = lambda n: int(min(n - 1, rng.zipf(1.6) - 1))  # noqa: E731
    src = np.array([offs[rels[k][0]] + pick(size[rels[k][0]]) for k in r], np.int64)
    dst = np.array([offs[rels[k][1]] + pick(size[rels[k][1]]) for k in r], np.int64)
    H = rng.standard_normal((int(offs[-1]), d))
    a = np.sqrt(6.0 / (2 * d))
    params = dict(W_rel=rng.uniform(-a, a, (num_rels, d, d)), W_agg=rng.uniform(-a, a, (2, d, d)),
                  b_agg=0.3 * rng.standard_normal((2, d)), ln_gamma=1 + 0.2 * rng.standard_normal((2, d)),
                  ln_beta=0.2 * rng.standard_normal((2, d)))
    return src, dst, r, offs, rels, H, params


def dense_mean_matrix(src, dst, rel, offs, rels, r):
    """Normalised adjacency D_r^-1 A_r (n_t x N), built edge by edge with Python loops."""
    tt = rels[r][1]
    n_t = int(offs[tt + 1] - offs[tt])
    A = np.zeros((n_t, int(offs[-1])))
    for s, t, k in zip(src.tolist(), dst.tolist(), rel.tolist()):
        if k == r:
            A[t - offs[tt], s] += 1.0
    deg = A.sum(axis=1, keepdims=True)
    return np.divide(A, deg, out=np.zeros_like(A), where=deg > 0)


def torch_layer(src, dst, rel, offs, rels, params, H, act="relu", layernorm=True, eps=1e-5):
    """Dense torch formulation of one layer; returns (out, leaves) with requires_grad leaves."""
    P = {k: torch.tensor(v, dtype=torch.float64, requires_grad=True) for k, v in params.items()}
    Ht = torch.tensor(H, dtype=torch.float64, requires_grad=True)
    outs = []
    for t in range(len(offs) - 1):
        lo, hi = int(offs[t]), int(offs[t + 1])
        Z = torch.zeros(hi - lo, H.shape[1], dtype=torch.float64)
        for r, (_, tt) in enumerate(rels):
            if tt == t:
                A = torch.tensor(dense_mean_matrix(src, dst, rel, offs, rels, r))
                Z = Z + (A @ Ht) @ P["W_rel"][r]
        U = Z @ P["W_agg"][t] + P["b_agg"][t]
        if act == "relu":
            a = torch.relu(U)
        elif act == "gelu_tanh":
            a = torch.nn.functional.gelu(U, approximate="tanh")
        else:
            a = U
        Y = a + Ht[lo:hi]
        if layernorm:
            Y = torch.nn.functional.layer_norm(Y, (H.shape[1],), P["ln_gamma"][t], P["ln_beta"][t], eps)
        outs.append(Y)
    return torch.cat(outs), P, Ht


# ---------------------------------------------------------------------------------------------
def test_aggregation_matches_dense_matrix():
    src, dst, rel, offs, rels, H, _ = small_graph(0)
    csr = oracle.build_csr(src, dst, rel, offs, rels)
    for r in range(len(rels)):
        M = oracle.mean_aggregate(csr[r], H)
        assert np.allclose(M, dense_mean_matrix(src, dst, rel, offs, rels, r) @ H, rtol=0, atol=1e-12)


def test_aggregation_rows_sum_to_one():
    src, dst, rel, offs, rels, H, _ = small_graph(1)
    csr = oracle.build_csr(src, dst, rel, offs, rels)
    ones = np.ones_like(H)
    for r in range(len(rels)):
        M = oracle.mean_aggregate(csr[r], ones)
        deg = csr[r]["deg"]
        assert np.all(M[deg > 0] == 1.0) and np.all(M[deg == 0] == 0.0)


def test_star_and_single_edge():
    offs = np.array([0, 6, 7], np.int64)
    rels = RELATIONS[:2]
    H = np.arange(7 * 3, dtype=np.float64).reshape(7, 3)
    # star: users 0..5 all point to risk node 6 (relation 1 = user -> risk)
    src = np.arange(6)
    dst = np.full(6, 6)
    rel = np.ones(6, np.int64)
    csr = oracle.build_csr(src, dst, rel, offs, rels)
    assert np.allclose(oracle.mean_aggregate(csr[1], H)[0], H[:6].mean(axis=0))
    # single edge user 2 -> user 4 (relation 0): identity copy into row 4, zeros elsewhere
    csr = oracle.build_csr(np.array([2]), np.array([4]), np.array([0]), offs, rels)
    M = oracle.mean_aggregate(csr[0], H)
    assert np.array_equal(M[4], H[2]) and np.all(np.delete(M, 4, axis=0) == 0)


@pytest.mark.parametrize("layernorm", [True, False])
def test_permutation_equivariance_within_types(layernorm):
    src, dst, rel, offs, rels, H, params = small_graph(2)
    n = int(offs[-1])
    rng = np.random.default_rng(9)
    perm = np.concatenate([rng.permutation(int(offs[t + 1] - offs[t])) + offs[t] for t in range(2)])
    inv = np.empty(n, np.int64)
    inv[perm] = np.arange(n)  # node i is renamed inv[i]
    csr = oracle.build_csr(src, dst, rel, offs, rels)
    out, _ = oracle.layer_forward(csr, offs, rels, params, H, layernorm=layernorm)
    csr_p = oracle.build_csr(inv[src], inv[dst], rel, offs, rels)
    out_p, _ = oracle.layer_forward(csr_p, offs, rels, params, H[perm], layernorm=layernorm)
    assert np.allclose(out_p, out[perm], rtol=0, atol=1e-12)


@pytest.mark.parametrize("act", ["relu", "gelu_tanh", "none"])
@pytest.mark.parametrize("layernorm", [True, False])
def test_forward_and_backward_match_torch_autograd(act, layernorm):
    src, dst, rel, offs, rels, H, params = small_graph(3)
    csr = oracle.build_csr(src, dst, rel, offs, rels)
    out, _ = oracle.layer_forward(csr, offs, rels, params, H, act, layernorm)
    ref, P, Ht = torch_layer(src, dst, rel, offs, rels, params, H, act, layernorm)
    assert np.allclose(out, ref.detach().numpy(), rtol=0, atol=1e-12)
    dout = np.random.default_rng(4).standard_normal(out.shape)
    (ref * torch.tensor(dout)).sum().backward()
    dH, g = oracle.layer_backward(csr, offs, rels, params, H, dout, act, layernorm)
    assert np.allclose(dH, Ht.grad.numpy(), rtol=0, atol=1e-11)
    for k in ("W_rel", "W_agg", "b_agg") + (("ln_gamma", "ln_beta") if layernorm else ()):
        assert np.allclose(g[k], P[k].grad.numpy(), rtol=0, atol=1e-11), k


def test_backward_finite_differences():
    src, dst, rel, offs, rels, H, params = small_graph(5, n_user=10, n_risk=4, num_edges=80, d=4)
    csr = oracle.build_csr(src, dst, rel, offs, rels)
    rng = np.random.default_rng(6)
    dout = rng.standard_normal(H.shape)
    f = lambda p, h: float((oracle.layer_forward(csr, offs, rels, p, h, "gelu_tanh")[0] * dout).sum())  # noqa: E731
    dH, g = oracle.layer_backward(csr, offs, rels, params, H, dout, "gelu_tanh")
    h = 1e-6
    for k in list(params) + ["H"]:
        base = H if k == "H" else params[k]
        v = rng.standard_normal(base.shape)
        plus = dict(params)
        minus = dict(params)
        if k == "H":
            fd = (f(params, H + h * v) - f(params, H - h * v)) / (2 * h)
            an = float((dH * v).sum())
        else:
            plus[k] = base + h * v
            minus[k] = base - h * v
            fd = (f(plus, H) - f(minus, H)) / (2 * h)
            an = float((g[k] * v).sum())
        assert abs(fd - an) <= 1e-6 * max(1.0, abs(an)), (k, fd, an)


def test_zero_relation_weights_give_bias_path():
    src, dst, rel, offs, rels, H, params = small_graph(7)
    p = dict(params)
    p["W_rel"] = np.zeros_like(p["W_rel"])
    csr = oracle.build_csr(src, dst, rel, offs, rels)
    out, _ = oracle.layer_forward(csr, offs, rels, p, H, layernorm=False)
    ty = O.node_type(np.arange(H.shape[0]), offs)
    assert np.allclose(out, np.maximum(p["b_agg"][ty], 0) + H, rtol=0, atol=1e-15)


def test_golden_tiny_layer():
    gd = json.load(open(os.path.join(GOLDEN, "layer_tiny.json")))
    offs = np.array(gd["type_offsets"])
    rels = tuple(tuple(r) for r in gd["rels"])
    src, dst, rel = (np.array(gd[k]) for k in ("src", "dst", "rel"))
    H = np.array(gd["H"], float)
    params = dict(W_rel=np.array(gd["W_rel"], float), W_agg=np.array(gd["W_agg"], float),
                  b_agg=np.array(gd["b_agg"], float), ln_gamma=np.ones((2, 2)), ln_beta=np.zeros((2, 2)))
    csr = oracle.build_csr(src, dst, rel, offs, rels)
    for r in range(3):
        assert np.array_equal(oracle.mean_aggregate(csr[r], H), np.array(gd[f"M_r{r}"], float))
    out, _ = oracle.layer_forward(csr, offs, rels, params, H, "relu", layernorm=False)
    assert np.array_equal(out, np.array(gd["H_out_no_ln"], float))
    out, _ = oracle.layer_forward(csr, offs, rels, params, H, "relu", layernorm=True, ln_eps=gd["ln_eps"])
    for row, half in zip(out, gd["H_out_ln_half_gaps"]):
        x = half / np.sqrt(half * half + gd["ln_eps"])
        assert np.allclose(row, [-x, x], rtol=0, atol=1e-15)


def test_sampled_rows_match_full():
    src, dst, rel, offs, rels, H, params = small_graph(8)
    csr = oracle.build_csr(src, dst, rel, offs, rels)
    out, _ = oracle.layer_forward(csr, offs, rels, params, H)
    rows = np.array([0, 3, 5, 23, 24, 30, 32])
    got, _ = oracle.layer_forward_rows(src, dst, rel, offs, rels, params, H, rows)
    assert np.allclose(got, out[rows], rtol=0, atol=1e-12)
    # backward with an upstream gradient that lives on a row subset S
    rng = np.random.default_rng(1)
    S = np.array([1, 3, 4, 10, 24, 27, 31])
    dout = np.zeros_like(H)
    dout[S] = rng.standard_normal((len(S), H.shape[1]))
    dH, g = oracle.layer_backward(csr, offs, rels, params, H, dout)
    q = np.arange(H.shape[0])
    dq, gs = oracle.layer_backward_rows(src, dst, rel, offs, rels, params, H, S, dout[S], q)
    assert np.allclose(dq, dH, rtol=0, atol=1e-12)
    for k in g:
        assert np.allclose(gs[k], g[k], rtol=0, atol=1e-12), k


# ---------------------------------------------------------------------------------------------
# planted mistakes: a copy of the oracle with one plausible error must fail a pin above
# ---------------------------------------------------------------------------------------------
def _agg_sum_instead_of_mean(csr_r, H):
    deg = csr_r["deg"]
    S = np.zeros((deg.shape[0], H.shape[1]))
    np.add.at(S, np.repeat(np.arange(deg.shape[0]), deg), H[csr_r["col"]])
    return S


def test_planted_sum_instead_of_mean_is_caught(monkeypatch):
    src, dst, rel, offs, rels, H, _ = small_graph(1)
    csr = oracle.build_csr(src, dst, rel, offs, rels)
    monkeypatch.setattr(O, "mean_aggregate", _agg_sum_instead_of_mean)
    errs = [np.abs(O.mean_aggregate(csr[r], H) - dense_mean_matrix(src, dst, rel, offs, rels, r) @ H).max()
            for r in range(len(rels))]
    assert max(errs) > 1e-3


@pytest.mark.parametrize("mistake", ["no_residual", "transposed_w_rel", "wrong_ln_grad"])
def test_planted_layer_mistakes_are_caught(mistake):
    src, dst, rel, offs, rels, H, params = small_graph(3)
    csr = oracle.build_csr(src, dst, rel, offs, rels)
    if mistake == "no_residual":
        # the update of Eq. 11 without its "+ h^(l-1)" term
        ref, _, _ = torch_layer(src, dst, rel, offs, rels, params, H, layernorm=False)
        out = O.layer_forward(csr, offs, rels, params, H, layernorm=False)[0] - H
        assert np.abs(out - ref.detach().numpy()).max() > 1e-3
        return
    ref, P, Ht = torch_layer(src, dst, rel, offs, rels, params, H)
    if mistake == "transposed_w_rel":
        p2 = dict(params)
        p2["W_rel"] = np.transpose(params["W_rel"], (0, 2, 1))
        out, _ = O.layer_forward(csr, offs, rels, p2, H)
        assert np.abs(out - ref.detach().numpy()).max() > 1e-3
    else:
        dout = np.random.default_rng(4).standard_normal(H.shape)
        (ref * torch.tensor(dout)).sum().backward()
        p2 = dict(params)
        p2["ln_gamma"] = np.ones_like(params["ln_gamma"])  # gain forgotten in dX_hat = dout * gamma
        dH, _ = O.layer_backward(csr, offs, rels, p2, H, dout)
        assert np.abs(dH - Ht.grad.numpy()).max() > 1e-3


# ---------------------------------------------------------------------------------------------
# bf16 storage mode: the oracle's rounding and its use at the two storage points
# ---------------------------------------------------------------------------------------------
def test_round_bf16_matches_torch():
    rng = np.random.default_rng(21)
    x = np.concatenate([rng.standard_normal(100_000) * 10.0 ** rng.integers(-30, 30, 100_000),
                        [0.0, -0.0, 1.0, 1.00390625, 1.01171875, 3.0e38, -1e-38]])
    want = torch.tensor(x, dtype=torch.float64).to(torch.float32).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(O.round_bf16(x), want)


def test_bf16_store_mode_matches_torch_with_bf16_casts():
    """store='bf16' = the dense torch formulation with M_r and Z W_agg (U without its bias) cast
    through torch.bfloat16."""
    src, dst, rel, offs, rels, H, params = small_graph(13, d=8)
    csr = oracle.build_csr(src, dst, rel, offs, rels)
    out, _ = oracle.layer_forward(csr, offs, rels, params, H, store="bf16")
    P = {k: torch.tensor(v, dtype=torch.float64) for k, v in params.items()}
    Ht = torch.tensor(H)
    bf = lambda t: t.to(torch.float32).to(torch.bfloat16).to(torch.float64)  # noqa: E731
    outs = []
    for t in range(2):
        lo, hi = int(offs[t]), int(offs[t + 1])
        Z = torch.zeros(hi - lo, H.shape[1], dtype=torch.float64)
        for r, (_, tt) in enumerate(rels):
            if tt == t:
                A = torch.tensor(dense_mean_matrix(src, dst, rel, offs, rels, r))
                Z = Z + bf(A @ Ht) @ P["W_rel"][r]
        U = bf(Z @ P["W_agg"][t]) + P["b_agg"][t]
        Y = torch.relu(U) + Ht[lo:hi]
        outs.append(torch.nn.functional.layer_norm(Y, (H.shape[1],), P["ln_gamma"][t], P["ln_beta"][t], 1e-5))
    assert np.allclose(out, torch.cat(outs).numpy(), rtol=0, atol=1e-12)
    # and the two modes differ (the rounding is really applied)
    out64, _ = oracle.layer_forward(csr, offs, rels, params, H)
    assert np.abs(out - out64).max() > 1e-6
