"""Pins of the oracle's attention layer (Heterogeneous Graph Transformer, Eq. 6-11).

torch autograd (fp64) on an independent formulation -- per-edge scores and messages, torch's own
scatter max, index_add segment sums and layer_norm -- pins the forward and every gradient; central
finite differences pin the gradient again.  Closed forms: a zero attention matrix (or mu = 0) makes
alpha uniform over each target's in-edges, so h~ is the plain mean of the messages; a target with
one in-edge takes that message; a node with no in-edge keeps act(b_agg) + h.  Order invariance of
the edges; planted mistakes (softmax per relation instead of over all of N(j), no 1/sqrt(d_h), heads
mixed) must fail.
"""
import numpy as np
import pytest
import torch

from oracle import hgt as OH
from oracle import hg_oracle as O

RELS = ((0, 0), (0, 1), (1, 0))


def graph(seed, n_user=30, n_risk=10, E=160, d=8, heads=2, rels=RELS):
    rng = np.random.default_rng(seed)
    N = n_user + n_risk
    offs = np.array([0, n_user, N], np.int64)
    src, dst, rel = [], [], []
    for _ in range(E):
        r = int(rng.integers(0, len(rels)))
        ts, tt = rels[r]
        src.append(int(rng.integers(offs[ts], offs[ts + 1])))
        dst.append(int(rng.integers(offs[tt], offs[tt + 1])))
        rel.append(r)
    H = rng.standard_normal((N, d))
    S, dh = heads, d // heads
    R, T = len(rels), 2
    a = np.sqrt(6 / (2 * d))
    p = {"W_K": rng.uniform(-a, a, (T, d, d)), "W_Q": rng.uniform(-a, a, (T, d, d)),
         "W_V": rng.uniform(-a, a, (T, d, d)), "b_K": 0.1 * rng.standard_normal((T, d)),
         "b_Q": 0.1 * rng.standard_normal((T, d)), "b_V": 0.1 * rng.standard_normal((T, d)),
         "W_att": rng.standard_normal((R, S, dh, dh)) / np.sqrt(dh), "W_msg": rng.standard_normal((R, S, dh, dh)) / np.sqrt(dh),
         "mu": 1.0 + 0.3 * rng.standard_normal(R), "W_agg": rng.uniform(-a, a, (T, d, d)),
         "b_agg": 0.2 * rng.standard_normal((T, d)), "ln_gamma": 1 + 0.1 * rng.standard_normal((T, d)),
         "ln_beta": 0.1 * rng.standard_normal((T, d))}
    return (np.array(src), np.array(dst), np.array(rel), offs, rels), H, p


def torch_layer(g, H, p, heads, layernorm=True, act="relu"):
    src, dst, rel, offs, rels = g
    N, d = H.shape
    S, dh = heads, d // heads
    T = {k: torch.tensor(v, requires_grad=True) for k, v in p.items()}
    Ht = torch.tensor(H, requires_grad=True)
    types = torch.tensor(O.node_type(np.arange(N), offs))
    s_, d_, r_ = (torch.tensor(x) for x in (src, dst, rel))

    def lin(name):
        return torch.einsum("nd,nde->ne", Ht, T["W_" + name][types]) + T["b_" + name][types]

    K, Q, V = lin("K"), lin("Q"), lin("V")
    Ks, Qs, Vs = (x.view(N, S, dh) for x in (K, Q, V))
    # Eq. 6 per edge and head
    att = torch.einsum("esa,esab,esb->es", Ks[s_], T["W_att"][r_], Qs[d_]) * (T["mu"][r_] / dh ** 0.5)[:, None]
    mx = torch.zeros(N, S, dtype=torch.float64).scatter_reduce(0, d_[:, None].expand(-1, S), att.detach(), "amax",
                                                               include_self=False)
    ex = torch.exp(att - mx[d_])
    den = torch.zeros(N, S, dtype=torch.float64).index_add(0, d_, ex)
    alpha = ex / den[d_]
    msg = torch.einsum("esa,esab->esb", Vs[s_], T["W_msg"][r_])
    ht = torch.zeros(N, S, dh, dtype=torch.float64).index_add(0, d_, alpha[:, :, None] * msg).reshape(N, d)
    U = torch.einsum("nd,nde->ne", ht, T["W_agg"][types]) + T["b_agg"][types]
    Y = (torch.relu(U) if act == "relu" else U) + Ht
    if layernorm:
        Yn = torch.nn.functional.layer_norm(Y, (d,), eps=1e-5)
        Y = Yn * T["ln_gamma"][types] + T["ln_beta"][types]
    return Y, Ht, T


@pytest.mark.parametrize("seed,heads,ln", [(0, 2, True), (1, 4, False), (2, 1, True)])
def test_matches_torch_autograd(seed, heads, ln):
    g, H, p = graph(seed, heads=heads)
    out, _ = OH.hgt_forward(*g, p, H, heads, layernorm=ln)
    Y, Ht, T = torch_layer(g, H, p, heads, layernorm=ln)
    assert np.allclose(out, Y.detach().numpy(), rtol=0, atol=1e-12)
    dOut = np.random.default_rng(seed + 9).standard_normal(H.shape)
    (Y * torch.tensor(dOut)).sum().backward()
    dH, gr = OH.hgt_backward(*g, p, H, dOut, heads, layernorm=ln)
    assert np.allclose(dH, Ht.grad.numpy(), rtol=1e-10, atol=1e-11)
    for k, v in T.items():
        if not ln and k in ("ln_gamma", "ln_beta"):
            continue
        assert np.allclose(gr[k], v.grad.numpy(), rtol=1e-10, atol=1e-11), k


def test_finite_differences():
    g, H, p = graph(3, n_user=12, n_risk=5, E=50, d=4, heads=2)
    dOut = np.random.default_rng(4).standard_normal(H.shape)
    dH, gr = OH.hgt_backward(*g, p, H, dOut, 2)
    h = 1e-6
    rng = np.random.default_rng(5)

    def L(H_, p_):
        return float((OH.hgt_forward(*g, p_, H_, 2)[0] * dOut).sum())

    for name in p:
        for _ in range(2):
            j = tuple(int(rng.integers(0, s)) for s in np.shape(p[name]))
            hi = {k: np.array(v, copy=True) for k, v in p.items()}
            lo = {k: np.array(v, copy=True) for k, v in p.items()}
            hi[name][j] += h
            lo[name][j] -= h
            fd = (L(H, hi) - L(H, lo)) / (2 * h)
            assert abs(fd - gr[name][j]) < 1e-6 * max(1.0, abs(fd)), (name, j)
    for _ in range(5):
        j = (int(rng.integers(0, H.shape[0])), int(rng.integers(0, H.shape[1])))
        hi, lo = H.copy(), H.copy()
        hi[j] += h
        lo[j] -= h
        assert abs((L(hi, p) - L(lo, p)) / (2 * h) - dH[j]) < 1e-6


@pytest.mark.parametrize("zero", ["W_att", "mu"])
def test_uniform_attention_is_the_mean_message(zero):
    g, H, p = graph(6, heads=2)
    src, dst, rel, offs, rels = g
    q = dict(p)
    q[zero] = np.zeros_like(p[zero])
    _, c = OH.hgt_forward(*g, q, H, 2, act="none", layernorm=False)
    deg = np.bincount(dst, minlength=H.shape[0])
    assert np.allclose(c["alpha"], 1.0 / deg[dst][:, None], rtol=0, atol=1e-15)
    # h~_j = mean over in-edges of V(i) blockdiag(W_msg[r]), so U = h~ W_agg + b
    types = O.node_type(np.arange(H.shape[0]), offs)
    V = np.stack([H[i] @ p["W_V"][types[i]] + p["b_V"][types[i]] for i in range(H.shape[0])])
    ht = np.zeros_like(H)
    for e in range(len(src)):
        ht[dst[e]] += V[src[e]] @ OH.blockdiag(p["W_msg"][rel[e]]) / deg[dst[e]]
    U = np.stack([ht[j] @ p["W_agg"][types[j]] + p["b_agg"][types[j]] for j in range(H.shape[0])])
    assert np.allclose(c["U"], U, rtol=0, atol=1e-12)


def test_single_edge_and_isolated_targets():
    g, H, p = graph(7, E=25, heads=2)
    src, dst, rel, offs, rels = g
    _, c = OH.hgt_forward(*g, p, H, 2, layernorm=False)
    deg = np.bincount(dst, minlength=H.shape[0])
    one = deg[dst] == 1
    assert np.allclose(c["alpha"][one], 1.0, rtol=0, atol=1e-15)
    types = O.node_type(np.arange(H.shape[0]), offs)
    iso = np.flatnonzero(deg == 0)
    assert iso.size > 0
    out, _ = OH.hgt_forward(*g, p, H, 2, layernorm=False)
    assert np.allclose(out[iso], np.maximum(p["b_agg"][types[iso]], 0) + H[iso], rtol=0, atol=1e-14)


def test_edge_order_invariance():
    g, H, p = graph(8, heads=4)
    src, dst, rel, offs, rels = g
    perm = np.random.default_rng(9).permutation(len(src))
    a, _ = OH.hgt_forward(*g, p, H, 4)
    b, _ = OH.hgt_forward(src[perm], dst[perm], rel[perm], offs, rels, p, H, 4)
    assert np.allclose(a, b, rtol=0, atol=1e-13)


def test_planted_mistakes_are_caught():
    g, H, p = graph(10, heads=2)
    Y, _, _ = torch_layer(g, H, p, 2)
    want = Y.detach().numpy()

    def caught():
        return not np.allclose(OH.hgt_forward(*g, p, H, 2)[0], want, atol=1e-9)

    assert not caught()
    src, dst, rel, offs, rels = g
    q = dict(p)
    q["mu"] = p["mu"] * np.sqrt(2.0)  # stands for a missing 1/sqrt(d_h)
    assert not np.allclose(OH.hgt_forward(*g, q, H, 2)[0], want, atol=1e-9)
    # heads mixed: treat the two heads as one (a single head of width d over the same weights)
    p1 = dict(p, W_att=np.stack([OH.blockdiag(w)[None] for w in p["W_att"]]),
              W_msg=np.stack([OH.blockdiag(w)[None] for w in p["W_msg"]]))
    assert not np.allclose(OH.hgt_forward(*g, p1, H, 1)[0], want, atol=1e-9)
    # a softmax per relation instead of over every in-edge: relabel every relation's targets apart
    dst2 = dst + 1000 * rel
    N2 = H.shape[0] + 1000 * len(rels)
    mx = np.full(N2, -np.inf)
    _, c = OH.hgt_forward(*g, p, H, 2)
    sc = c["score"][:, 0]
    np.maximum.at(mx, dst2, sc)
    ex = np.exp(sc - mx[dst2])
    den = np.zeros(N2)
    np.add.at(den, dst2, ex)
    per_rel = ex / den[dst2]
    assert not np.allclose(per_rel, c["alpha"][:, 0], atol=1e-6)


def test_bf16_storage_points():
    from hgsynth import bf16_round
    g, H, p = graph(11, heads=2)
    out_b, cb = OH.hgt_forward(*g, p, H, 2, store="bf16")
    out_f, cf = OH.hgt_forward(*g, p, H, 2)
    for k in ("K", "V", "Q", "Qp", "Ssum"):
        assert np.array_equal(cb[k], bf16_round(cb[k]).astype(np.float64)), k
    ub = cb["U"] - p["b_agg"][cb["types"]]  # U is stored without its bias
    assert np.allclose(ub, bf16_round(ub).astype(np.float64), rtol=0, atol=1e-12)
    assert np.abs(out_b - out_f).max() <= 2e-2 * np.abs(out_f).max()
