"""Pin of the oracle's whole step (layers forward, alignment, layers backward) against one torch
autograd graph of the same dense formulation (CPU only)."""
import numpy as np
import torch

import oracle
from tests.test_oracle_align import torch_loss  # noqa: F401  (same loss formula, autograd)
from tests.test_oracle_layer import small_graph, torch_layer


def two_stacks():
    """The small two-layer problem, its oracle inputs, and the dense torch formulation of both
    stacks (sharing the weights) up to their outputs."""
    src, dst, rel, offs, rels, X, p0 = small_graph(11, d=5)
    _, _, _, _, _, _, p1 = small_graph(12, d=5)
    rng = np.random.default_rng(13)
    Xb = X + 0.1 * rng.standard_normal(X.shape)
    dtop = rng.standard_normal(X.shape)
    idx = np.sort(rng.choice(X.shape[0], 12, replace=False))
    graph = dict(src=src, dst=dst, rel=rel, type_offsets=offs, rels=rels)
    h1a, P0, Xa_t = torch_layer(src, dst, rel, offs, rels, p0, X)
    h1b, P0b, Xb_t = torch_layer(src, dst, rel, offs, rels, p0, Xb)
    outs = []
    for h1 in (h1a, h1b):
        # second layer on a torch input: rebuild the dense formulation with h1 as input
        Ht = h1
        parts = []
        P1 = {k: torch.tensor(v, dtype=torch.float64) for k, v in p1.items()}
        for t in range(2):
            lo, hi = int(offs[t]), int(offs[t + 1])
            Z = torch.zeros(hi - lo, X.shape[1], dtype=torch.float64)
            for r, (_, tt) in enumerate(rels):
                if tt == t:
                    from tests.test_oracle_layer import dense_mean_matrix
                    A = torch.tensor(dense_mean_matrix(src, dst, rel, offs, rels, r))
                    Z = Z + (A @ Ht) @ P1["W_rel"][r]
            U = Z @ P1["W_agg"][t] + P1["b_agg"][t]
            Y = torch.relu(U) + Ht[lo:hi]
            parts.append(torch.nn.functional.layer_norm(Y, (X.shape[1],), P1["ln_gamma"][t], P1["ln_beta"][t], 1e-5))
        outs.append(torch.cat(parts))
    return graph, X, Xb, dtop, idx, [p0, p1], outs, (P0, P0b, Xa_t, Xb_t)


def test_step_matches_torch_autograd():
    graph, X, Xb, dtop, idx, params, outs, (P0, P0b, Xa_t, Xb_t) = two_stacks()
    res = oracle.step(graph, X, params, dtop, {"idx": idx, "X_b": Xb}, lambda_n=2e-4, var_eps=1e-8, dloss=0.1)
    # torch: two stacks sharing weights, loss = <H_a, dtop> + 0.1 * L_CCA(H_a[idx], H_b[idx])
    Ha, Hb = outs
    ii = torch.tensor(idx)

    def z(M):
        n = M.shape[0]
        return (M - M.mean(0)) / (torch.sqrt(M.var(0, unbiased=False) + 1e-8) * np.sqrt(n))

    Za, Zb = z(Ha[ii]), z(Hb[ii])
    I = torch.eye(X.shape[1], dtype=torch.float64)
    L = ((Za - Zb) ** 2).sum() + 2e-4 * (((Za.T @ Za - I) ** 2).sum() + ((Zb.T @ Zb - I) ** 2).sum())
    total = (Ha * torch.tensor(dtop)).sum() + 0.1 * L
    total.backward()
    assert np.isclose(res["loss"][0], L.item(), rtol=1e-12)
    assert np.allclose(res["H"][-1], Ha.detach().numpy(), atol=1e-12)
    assert np.allclose(res["dX"], Xa_t.grad.numpy(), atol=1e-10)
    assert np.allclose(res["dX_b"], Xb_t.grad.numpy(), atol=1e-10)
    # layer-0 weights are shared by both stacks in torch; the oracle reports each stack's share
    for k in ("W_rel", "W_agg", "b_agg", "ln_gamma", "ln_beta"):
        both = res["grads"][0][k] + res["grads_b"][0][k]
        assert np.allclose(both, P0[k].grad.numpy() + P0b[k].grad.numpy(), atol=1e-10), k


def test_step_with_head_matches_torch_autograd():
    """The joint objective of Eq. 20: L_BCE of the head on the MeanAgg of both stacks' outputs
    (Eq. 18-19) plus 0.1 * L_CCA, through both stacks."""
    graph, X, Xb, _, idx, params, outs, (P0, P0b, Xa_t, Xb_t) = two_stacks()
    rng = np.random.default_rng(21)
    d = X.shape[1]
    hp = {"W1": rng.standard_normal((d, d)) / np.sqrt(d), "b1": 0.2 * rng.standard_normal(d),
          "w2": rng.standard_normal(d), "b2": np.array([-0.4])}
    lab = np.sort(np.concatenate([idx[:5], rng.choice(np.setdiff1d(np.arange(X.shape[0]), idx), 9, replace=False)]))
    y = (rng.random(len(lab)) < 0.4).astype(np.float64)
    res = oracle.step(graph, X, params, None, {"idx": idx, "X_b": Xb}, lambda_n=2e-4, var_eps=1e-8, dloss=0.1,
                      head={"params": hp, "lab_idx": lab, "lab_y": y})
    Ha, Hb = outs
    ii = torch.tensor(idx)
    mask = torch.zeros(Ha.shape[0], 1, dtype=torch.float64)
    mask[ii] = 1.0
    other = torch.zeros_like(Ha).index_put((ii,), Hb[ii])
    Hf = Ha * (1 - mask) + 0.5 * (Ha + other) * mask
    T = {k: torch.tensor(v, requires_grad=True) for k, v in hp.items()}
    zl = torch.relu(Hf[torch.tensor(lab)] @ T["W1"] + T["b1"]) @ T["w2"] + T["b2"]
    bce = torch.nn.functional.binary_cross_entropy_with_logits(zl, torch.tensor(y))

    def z(M):
        n = M.shape[0]
        return (M - M.mean(0)) / (torch.sqrt(M.var(0, unbiased=False) + 1e-8) * np.sqrt(n))

    Za, Zb = z(Ha[ii]), z(Hb[ii])
    I = torch.eye(d, dtype=torch.float64)
    L = ((Za - Zb) ** 2).sum() + 2e-4 * (((Za.T @ Za - I) ** 2).sum() + ((Zb.T @ Zb - I) ** 2).sum())
    total = bce + 0.1 * L
    total.backward()
    assert np.isclose(res["head_loss"][0], total.item(), rtol=1e-12)
    assert np.isclose(res["head_loss"][1], bce.item(), rtol=1e-12)
    assert np.allclose(res["dX"], Xa_t.grad.numpy(), atol=1e-10)
    assert np.allclose(res["dX_b"], Xb_t.grad.numpy(), atol=1e-10)
    for k in ("W1", "b1", "w2", "b2"):
        assert np.allclose(res["head_grads"]["d" + k], T[k].grad.numpy(), atol=1e-12), k
    for k in ("W_rel", "W_agg", "b_agg", "ln_gamma", "ln_beta"):
        both = res["grads"][0][k] + res["grads_b"][0][k]
        assert np.allclose(both, P0[k].grad.numpy() + P0b[k].grad.numpy(), atol=1e-10), k
