"""CPU oracle of the hot path.  TEST INFRASTRUCTURE ONLY.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg import this module; the
product path (the C-ABI library and its Python binding) never calls it, and it shares no code
with that path.  Everything is plain numpy in fp64; the inputs are the seeded arrays of `hgsynth`
(bf16 inputs arrive as fp32 values that are exactly representable in bf16).

What is computed, and the reading of the paper each function follows:

* build_csr ........ the relation-typed adjacency of the snapshot (Section 2.2: node types tau,
                     relations phi, meta-relation triplets), restricted to the subgraph
                     (Eq. 5 and the induced subgraph of Algorithm 1), laid out per relation by
                     destination (CSR) and by source (CSC).  Within a row the neighbours keep the
                     input edge order (ascending edge id).  Invalid edges (ids out of range, relation
                     out of range, endpoint types that do not match the relation) are dropped.
* layer_forward .... one heterogeneous message-passing layer: per relation r the message of
                     Eq. 7 with one matrix W_r per relation, the aggregation of Eq. 10 with the
                     mean as the operator (+) and the per-relation means summed into the target,
                     then the update of Eq. 11 (Linear_agg per target type, activation, residual),
                     optionally followed by LayerNorm per target type.
* layer_backward ... the chain rule of layer_forward, written out step by step.
* align_forward .... the consistency-alignment loss of Eq. 14-17 on the overlap rows.
* align_backward ... its gradient with respect to both views' rows.
* overlap_intersect  the overlap batch B of Section 3.3 as pairs of local rows, ascending by
                     global id (B is the intersection of the two overlapping node sets of Eq. 5).

Readings where the paper is silent or ambiguous (listed again in the design notes):
  mean aggregation per relation, no attention (the GraphSAGE-style backbone of Table 6);
  relations into one type are summed; a row with no in-edge of relation r gets M_r = 0;
  activation = ReLU (GELU with the tanh form as an option); the residual needs d_in = d_out;
  LayerNorm after the residual add, population variance, eps 1e-5, gain/shift per node type;
  alignment standardisation uses the population standard deviation with eps added to the
  variance; both loss terms are plain sums (squared Frobenius norms); lambda_n = 2e-4.

Storage precision of intermediates (store="bf16").  For bf16 workloads the kernels store the
relation means M_r in bf16 and the pre-activation without its bias, Z W_agg, in bf16 (the
activation and its derivative are taken at that stored value plus the bias); weights, and
products of weights, are never rounded.  The ReLU mask
is an integer decision made by floating point, and the paper fixes no precision; where a
pre-activation lies within a rounding of zero either mask is a valid outcome.  store="bf16"
rounds M_r and U to bf16 (round to nearest, ties to even; its own rounding routine) and keeps
every other operation, including all gradients, in fp64, so that a test on inputs with such
near-zero pre-activations can compare row by row with the decisions the kernel takes.
store="f64" (default) is the plain definition, the yardstick of every other comparison.

Functions that no independent pin covers are marked "parity unpinned" in their docstring; every
function here has pins in tests/test_oracle_*.py.
"""
from __future__ import annotations

import numpy as np

F64 = np.float64
GELU_K = float(np.sqrt(2.0 / np.pi))


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round to the nearest bfloat16 (ties to even) via fp32: keep the top 16 bits of the fp32
    pattern after adding 0x7FFF plus the lowest kept bit.  Returns fp64 values."""
    f = np.ascontiguousarray(np.asarray(x, np.float64).astype(np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000).astype(np.uint32)
    return r.view(np.float32).astype(np.float64).reshape(f.shape)


def _stored(x: np.ndarray, store: str) -> np.ndarray:
    if store == "f64":
        return x
    if store == "bf16":
        return round_bf16(x)
    raise ValueError(store)


# ----------------------------------------------------------------------------------------------
# graph layout
# ----------------------------------------------------------------------------------------------
def node_type(ids: np.ndarray, type_offsets: np.ndarray) -> np.ndarray:
    return np.searchsorted(np.asarray(type_offsets), ids, side="right") - 1


def valid_edges(src, dst, rel, type_offsets, rels) -> np.ndarray:
    """Mask of edges whose ids are in range and whose endpoint types match their relation."""
    src = np.asarray(src, np.int64)
    dst = np.asarray(dst, np.int64)
    rel = np.asarray(rel, np.int64)
    n = int(type_offsets[-1])
    ok = (rel >= 0) & (rel < len(rels)) & (src >= 0) & (src < n) & (dst >= 0) & (dst < n)
    rs = np.array([r[0] for r in rels] + [-1], np.int64)
    rt = np.array([r[1] for r in rels] + [-1], np.int64)
    rr = np.where(ok, rel, len(rels))
    ok &= node_type(np.where(ok, src, 0), type_offsets) == rs[rr]
    ok &= node_type(np.where(ok, dst, 0), type_offsets) == rt[rr]
    return ok


def build_csr(src, dst, rel, type_offsets, rels) -> list:
    """Per relation r: CSR by destination (row_ptr over the n_t destination rows, col = source node
    id, eid) and CSC by source (csc_ptr over the n_s source rows, csc_col = destination node id,
    csc_eid, csc_coef = fp32 1/deg_r(destination)).  Row order: local id within the type.  Within a
    CSR row the in-edges ascend by (source id, edge id), within a CSC row the out-edges by
    (destination id, edge id), so the parallel edges of a node pair are adjacent."""
    src = np.asarray(src, np.int64)
    dst = np.asarray(dst, np.int64)
    rel = np.asarray(rel, np.int64)
    offs = np.asarray(type_offsets, np.int64)
    ok = valid_edges(src, dst, rel, offs, rels)
    out = []
    for r, (ts, tt) in enumerate(rels):
        n_s = int(offs[ts + 1] - offs[ts])
        n_t = int(offs[tt + 1] - offs[tt])
        eids = np.flatnonzero(ok & (rel == r))  # ascending edge id
        dl = dst[eids] - offs[tt]
        sl = src[eids] - offs[ts]
        by_dst = eids[np.argsort(dl * n_s + sl, kind="stable")]  # (destination, source, edge id)
        deg = np.bincount(dl, minlength=n_t)
        row_ptr = np.concatenate([[0], np.cumsum(deg)]).astype(np.int64)
        by_src = eids[np.argsort(sl * n_t + dl, kind="stable")]  # (source, destination, edge id)
        odeg = np.bincount(sl, minlength=n_s)
        csc_ptr = np.concatenate([[0], np.cumsum(odeg)]).astype(np.int64)
        coef = np.float32(1.0) / deg[dst[by_src] - offs[tt]].astype(np.float32)
        out.append(dict(row_ptr=row_ptr, col=src[by_dst], eid=by_dst, deg=deg,
                        csc_ptr=csc_ptr, csc_col=dst[by_src], csc_eid=by_src, csc_coef=coef))
    return out


def node_order(csr: list, type_offsets, rels, node_type: int, tile_rows: int = 128) -> tuple:
    """The order in which the tensor-core forward projection visits the nodes of one type (a layout
    of the kernels, not of the paper): the relation mask of local node j has bit k set when the k-th
    relation into the type (ascending relation id) has an in-edge at j; perm lists the local ids by
    ascending (mask, id); tile_mask[q] is the OR of the masks at positions tile_rows q onwards."""
    offs = np.asarray(type_offsets, np.int64)
    n = int(offs[node_type + 1] - offs[node_type])
    mask = np.zeros(n, np.int64)
    k = 0
    for r, (_, tt) in enumerate(rels):
        if tt != node_type:
            continue
        mask |= (csr[r]["deg"] > 0).astype(np.int64) << k
        k += 1
    perm = np.argsort(mask, kind="stable")
    tiles = -(-n // tile_rows)
    tile_mask = np.zeros(tiles, np.int64)
    for q in range(tiles):
        tile_mask[q] = np.bitwise_or.reduce(mask[perm[q * tile_rows:(q + 1) * tile_rows]])
    return perm, tile_mask


# ----------------------------------------------------------------------------------------------
# layer
# ----------------------------------------------------------------------------------------------
def act_fwd(u: np.ndarray, act: str) -> np.ndarray:
    if act == "relu":
        return np.maximum(u, 0.0)
    if act == "gelu_tanh":
        return 0.5 * u * (1.0 + np.tanh(GELU_K * (u + 0.044715 * u ** 3)))
    if act == "none":
        return u
    raise ValueError(act)


def act_grad(u: np.ndarray, act: str) -> np.ndarray:
    if act == "relu":
        return (u > 0).astype(F64)
    if act == "gelu_tanh":
        t = np.tanh(GELU_K * (u + 0.044715 * u ** 3))
        return 0.5 * (1.0 + t) + 0.5 * u * (1.0 - t * t) * GELU_K * (1.0 + 3 * 0.044715 * u * u)
    if act == "none":
        return np.ones_like(u)
    raise ValueError(act)


def mean_aggregate(csr_r: dict, H: np.ndarray) -> np.ndarray:
    """M_r[j] = (1/deg_r(j)) * sum over in-edges (i -> j) of relation r of H[i]; 0 if deg_r(j) = 0.
    Eq. 10 with (+) = mean over the neighbours of relation r (messages of Eq. 7 before W_r)."""
    deg = csr_r["deg"]
    n_t = deg.shape[0]
    rows = np.repeat(np.arange(n_t), deg)
    S = np.zeros((n_t, H.shape[1]), F64)
    np.add.at(S, rows, np.asarray(H, F64)[csr_r["col"]])
    return np.where(deg[:, None] > 0, S / np.maximum(deg, 1)[:, None], 0.0)


def _p64(params: dict) -> dict:
    return {k: np.asarray(v, F64) for k, v in params.items()}


def layer_forward(csr: list, type_offsets, rels, params: dict, H, act: str = "relu",
                  layernorm: bool = True, ln_eps: float = 1e-5, store: str = "f64") -> tuple:
    """H_out[j] = LN_tau(act(Z[j] W_agg[tau] + b[tau]) + H[j]),  Z[j] = sum_{r: t_r = tau} M_r[j] W_r.
    Eq. 7 (one W_r per relation), Eq. 10 (mean), Eq. 11 (update + residual), LayerNorm optional.
    Returns (H_out, cache) with the intermediates per type."""
    p = _p64(params)
    H = np.asarray(H, F64)
    offs = np.asarray(type_offsets, np.int64)
    out = np.empty_like(H)
    cache = {"M": {}, "types": {}}
    for t in range(len(offs) - 1):
        lo, hi = int(offs[t]), int(offs[t + 1])
        Z = np.zeros((hi - lo, H.shape[1]), F64)
        for r, (_, tt) in enumerate(rels):
            if tt != t:
                continue
            M = _stored(mean_aggregate(csr[r], H), store)
            cache["M"][r] = M
            Z += M @ p["W_rel"][r]
        U = _stored(Z @ p["W_agg"][t], store) + p["b_agg"][t]  # U is stored without its bias
        Y = act_fwd(U, act) + H[lo:hi]
        c = {"Z": Z, "U": U, "Y": Y}
        if layernorm:
            mu = Y.mean(axis=1, keepdims=True)
            var = ((Y - mu) ** 2).mean(axis=1, keepdims=True)
            rstd = 1.0 / np.sqrt(var + ln_eps)
            Xh = (Y - mu) * rstd
            out[lo:hi] = Xh * p["ln_gamma"][t] + p["ln_beta"][t]
            c.update(mu=mu[:, 0], rstd=rstd[:, 0], Xh=Xh)
        else:
            out[lo:hi] = Y
        cache["types"][t] = c
    return out, cache


def layer_backward(csr: list, type_offsets, rels, params: dict, H, dH_out, act: str = "relu",
                   layernorm: bool = True, ln_eps: float = 1e-5, store: str = "f64") -> tuple:
    """Gradients of layer_forward: returns (dH_in, grads) with grads = dict(W_rel, W_agg, b_agg,
    ln_gamma, ln_beta).  dH_in = residual path + transpose of the mean aggregation."""
    p = _p64(params)
    H = np.asarray(H, F64)
    dH_out = np.asarray(dH_out, F64)
    offs = np.asarray(type_offsets, np.int64)
    _, cache = layer_forward(csr, type_offsets, rels, params, H, act, layernorm, ln_eps, store)
    d = H.shape[1]
    R, T = len(rels), len(offs) - 1
    g = dict(W_rel=np.zeros((R, d, d)), W_agg=np.zeros((T, d, d)), b_agg=np.zeros((T, d)),
             ln_gamma=np.zeros((T, d)), ln_beta=np.zeros((T, d)))
    dH_in = np.zeros_like(H)
    for t in range(T):
        lo, hi = int(offs[t]), int(offs[t + 1])
        c = cache["types"][t]
        dout = dH_out[lo:hi]
        if layernorm:
            Xh, rstd = c["Xh"], c["rstd"][:, None]
            g["ln_gamma"][t] = (dout * Xh).sum(axis=0)
            g["ln_beta"][t] = dout.sum(axis=0)
            dXh = dout * p["ln_gamma"][t]
            dY = rstd * (dXh - dXh.mean(axis=1, keepdims=True) - Xh * (dXh * Xh).mean(axis=1, keepdims=True))
        else:
            dY = dout
        dH_in[lo:hi] += dY  # residual of Eq. 11
        dU = dY * act_grad(c["U"], act)
        g["b_agg"][t] = dU.sum(axis=0)
        g["W_agg"][t] = c["Z"].T @ dU
        dZ = dU @ p["W_agg"][t].T
        for r, (_, tt) in enumerate(rels):
            if tt != t:
                continue
            M = cache["M"][r]
            g["W_rel"][r] = M.T @ dZ
            dM = dZ @ p["W_rel"][r].T
            deg = csr[r]["deg"]
            rows = np.repeat(np.arange(hi - lo), deg)
            # edge (i -> j) of relation r carries dM[j] / deg_r(j) back to its source i
            np.add.at(dH_in, csr[r]["col"], dM[rows] / deg[rows][:, None])
    return dH_in, g


# ----------------------------------------------------------------------------------------------
# sampled forms for full-size checks: the same definitions, evaluated only where asked
# ----------------------------------------------------------------------------------------------
def _row_aggregates(src, dst, rel, valid, rows_sorted, H, R, chunk=1 << 20):
    """For sorted node ids `rows_sorted`: S[k, r] = sum of H[src] over valid in-edges of relation r
    into rows_sorted[k], and deg[k, r] their count."""
    n = rows_sorted.shape[0]
    d = H.shape[1]
    S = np.zeros((n, R, d), F64)
    deg = np.zeros((n, R), np.int64)
    pos = np.searchsorted(rows_sorted, dst)
    pos_c = np.minimum(pos, n - 1)
    hit = valid & (rows_sorted[pos_c] == dst)
    e = np.flatnonzero(hit)
    np.add.at(deg, (pos_c[e], rel[e]), 1)
    for s in range(0, e.shape[0], chunk):
        ec = e[s:s + chunk]
        np.add.at(S, (pos_c[ec], rel[ec]), np.asarray(H[src[ec]], F64))
    return S, deg


def layer_forward_rows(src, dst, rel, type_offsets, rels, params, H, rows, act="relu",
                       layernorm=True, ln_eps=1e-5, store="f64") -> tuple:
    """layer_forward evaluated only at node ids `rows` (sorted, unique), straight from the COO list.
    Returns (H_out[rows], cache) with per-row M (n x R x d), Z, U, deg, Xh, rstd."""
    src = np.asarray(src, np.int64)
    dst = np.asarray(dst, np.int64)
    rel = np.asarray(rel, np.int64)
    p = _p64(params)
    rows = np.asarray(rows, np.int64)
    valid = valid_edges(src, dst, rel, type_offsets, rels)
    R = len(rels)
    S, deg = _row_aggregates(src, dst, rel, valid, rows, H, R)
    M = _stored(np.where(deg[:, :, None] > 0, S / np.maximum(deg, 1)[:, :, None], 0.0), store)
    ty = node_type(rows, type_offsets)
    d = H.shape[1]
    Z = np.zeros((rows.shape[0], d), F64)
    rt = np.array([r[1] for r in rels])
    for r in range(R):
        m = ty == rt[r]
        Z[m] += M[m, r] @ p["W_rel"][r]
    U = _stored(np.einsum("nk,nkj->nj", Z, p["W_agg"][ty]), store) + p["b_agg"][ty]
    Y = act_fwd(U, act) + np.asarray(H, F64)[rows]
    cache = dict(M=M, Z=Z, U=U, Y=Y, deg=deg, ty=ty)
    if layernorm:
        mu = Y.mean(axis=1, keepdims=True)
        var = ((Y - mu) ** 2).mean(axis=1, keepdims=True)
        rstd = 1.0 / np.sqrt(var + ln_eps)
        Xh = (Y - mu) * rstd
        cache.update(Xh=Xh, rstd=rstd[:, 0])
        return Xh * p["ln_gamma"][ty] + p["ln_beta"][ty], cache
    return Y, cache


def layer_backward_rows(src, dst, rel, type_offsets, rels, params, H, S_rows, dH_S, query_rows,
                        act="relu", layernorm=True, ln_eps=1e-5, store="f64") -> tuple:
    """layer_backward for an upstream gradient that is zero except on the sorted node ids S_rows
    (values dH_S).  Returns (dH_in[query_rows], grads); the weight gradients are complete because
    only rows in S_rows contribute to them."""
    src = np.asarray(src, np.int64)
    dst = np.asarray(dst, np.int64)
    rel = np.asarray(rel, np.int64)
    p = _p64(params)
    S_rows = np.asarray(S_rows, np.int64)
    query_rows = np.asarray(query_rows, np.int64)
    _, c = layer_forward_rows(src, dst, rel, type_offsets, rels, params, H, S_rows, act, layernorm, ln_eps, store)
    ty = c["ty"]
    dout = np.asarray(dH_S, F64)
    d = dout.shape[1]
    R, T = len(rels), len(type_offsets) - 1
    g = dict(W_rel=np.zeros((R, d, d)), W_agg=np.zeros((T, d, d)), b_agg=np.zeros((T, d)),
             ln_gamma=np.zeros((T, d)), ln_beta=np.zeros((T, d)))
    if layernorm:
        Xh, rstd = c["Xh"], c["rstd"][:, None]
        for t in range(T):
            m = ty == t
            g["ln_gamma"][t] = (dout[m] * Xh[m]).sum(axis=0)
            g["ln_beta"][t] = dout[m].sum(axis=0)
        dXh = dout * p["ln_gamma"][ty]
        dY = rstd * (dXh - dXh.mean(axis=1, keepdims=True) - Xh * (dXh * Xh).mean(axis=1, keepdims=True))
    else:
        dY = dout
    dU = dY * act_grad(c["U"], act)
    dZ = np.einsum("nj,nkj->nk", dU, p["W_agg"][ty])
    rt = np.array([r[1] for r in rels])
    dMs = np.zeros((S_rows.shape[0], R, d), F64)  # dM_r[j] / deg_r(j)
    for t in range(T):
        m = ty == t
        g["b_agg"][t] = dU[m].sum(axis=0)
        g["W_agg"][t] = c["Z"][m].T @ dU[m]
    for r in range(R):
        m = ty == rt[r]
        g["W_rel"][r] = c["M"][m, r].T @ dZ[m]
        dM = dZ[m] @ p["W_rel"][r].T
        degm = c["deg"][m, r]
        dMs[m, r] = np.where(degm[:, None] > 0, dM / np.maximum(degm, 1)[:, None], 0.0)
    # dH_in at the query rows: residual part (if the row is in S) + edges (i -> j in S) carrying dMs[j, r]
    out = np.zeros((query_rows.shape[0], d), F64)
    k = np.searchsorted(S_rows, query_rows)
    kc = np.minimum(k, S_rows.shape[0] - 1)
    ins = S_rows[kc] == query_rows
    out[ins] += dY[kc[ins]]
    valid = valid_edges(src, dst, rel, type_offsets, rels)
    qpos = np.searchsorted(query_rows, src)
    qc = np.minimum(qpos, query_rows.shape[0] - 1)
    spos = np.searchsorted(S_rows, dst)
    sc = np.minimum(spos, S_rows.shape[0] - 1)
    e = np.flatnonzero(valid & (query_rows[qc] == src) & (S_rows[sc] == dst))
    np.add.at(out, qc[e], dMs[sc[e], rel[e]])
    return out, g


# ----------------------------------------------------------------------------------------------
# alignment (Eq. 14-17) and overlap
# ----------------------------------------------------------------------------------------------
def standardise(X: np.ndarray, eps: float) -> tuple:
    """Eq. 14: H_hat = (H - mu) / (sigma * sqrt(n)) per feature column, population sigma with eps
    added to the variance.  Returns (H_hat, mu, s) with s = sqrt(var + eps)."""
    n = X.shape[0]
    mu = X.mean(axis=0)
    var = ((X - mu) ** 2).mean(axis=0)
    s = np.sqrt(var + eps)
    return (X - mu) / (s * np.sqrt(n)), mu, s


def align_forward(Ha, idx_a, Hb, idx_b, lambda_n: float = 2e-4, eps: float = 1e-8) -> tuple:
    """L_CCA = ||Z_a - Z_b||_F^2 + lambda_n (||Z_a^T Z_a - I||_F^2 + ||Z_b^T Z_b - I||_F^2)
    (Eq. 15, 16, 17) on Z = standardised overlap rows (Eq. 14).  Returns (L, L_inv, L_dec)."""
    A = np.asarray(Ha, F64)[np.asarray(idx_a, np.int64)]
    B = np.asarray(Hb, F64)[np.asarray(idx_b, np.int64)]
    Za, _, _ = standardise(A, eps)
    Zb, _, _ = standardise(B, eps)
    I = np.eye(A.shape[1])
    l_inv = float(((Za - Zb) ** 2).sum())
    l_dec = float(((Za.T @ Za - I) ** 2).sum() + ((Zb.T @ Zb - I) ** 2).sum())
    return l_inv + lambda_n * l_dec, l_inv, l_dec


def _standardise_backward(X: np.ndarray, G: np.ndarray, eps: float) -> np.ndarray:
    """Gradient through Eq. 14: with x_hat = (h - mu)/s and g = dL/dx_hat = G / sqrt(n),
    dL/dh = (1/s) (g - mean(g) - x_hat * mean(g * x_hat)) per column (s depends on h through var)."""
    n = X.shape[0]
    mu = X.mean(axis=0)
    s = np.sqrt(((X - mu) ** 2).mean(axis=0) + eps)
    xh = (X - mu) / s
    g = G / np.sqrt(n)
    return (g - g.mean(axis=0) - xh * (g * xh).mean(axis=0)) / s


def align_backward(Ha, idx_a, Hb, idx_b, lambda_n: float = 2e-4, eps: float = 1e-8,
                   dloss: float = 1.0) -> tuple:
    """dL/dH_a and dL/dH_b (full-shape arrays, non-zero only on the overlap rows) for
    L = dloss * L_CCA.  dL/dZ_a = 2 (Z_a - Z_b) + 4 lambda_n Z_a (Z_a^T Z_a - I), likewise for b
    with the sign of the invariance term flipped."""
    idx_a = np.asarray(idx_a, np.int64)
    idx_b = np.asarray(idx_b, np.int64)
    A = np.asarray(Ha, F64)[idx_a]
    B = np.asarray(Hb, F64)[idx_b]
    Za, _, _ = standardise(A, eps)
    Zb, _, _ = standardise(B, eps)
    I = np.eye(A.shape[1])
    Ga = dloss * (2.0 * (Za - Zb) + 4.0 * lambda_n * Za @ (Za.T @ Za - I))
    Gb = dloss * (-2.0 * (Za - Zb) + 4.0 * lambda_n * Zb @ (Zb.T @ Zb - I))
    dHa = np.zeros(np.shape(Ha), F64)
    dHb = np.zeros(np.shape(Hb), F64)
    dHa[idx_a] = _standardise_backward(A, Ga, eps)
    dHb[idx_b] = _standardise_backward(B, Gb, eps)
    return dHa, dHb


def overlap_intersect(gid_a, gid_b) -> tuple:
    """Local rows (idx_a, idx_b) of the nodes present in both subgraphs, ascending by global id."""
    _, ia, ib = np.intersect1d(np.asarray(gid_a, np.int64), np.asarray(gid_b, np.int64),
                               assume_unique=True, return_indices=True)
    return ia.astype(np.int64), ib.astype(np.int64)


# ----------------------------------------------------------------------------------------------
# one whole step of the hot path (used for the CPU baseline and small end-to-end checks)
# ----------------------------------------------------------------------------------------------
def step(graph: dict, X, params: list, dH_top, view_b: dict, act="relu", layernorm=True,
         ln_eps=1e-5, lambda_n=2e-4, var_eps=1e-8, dloss=0.1, store="f64", head: dict | None = None,
         interface: str = "f64") -> dict:
    """CSR build -> L layers forward -> overlap rows -> alignment loss and gradient -> L layers
    backward (view_b None: no alignment term, as for the first subgraph of a sequence).
    interface="bf16": the tensors handed from layer to layer (each layer's output, and the gradient
    with respect to it) are rounded to bf16, the storage type of every tensor the layer interface
    exchanges for a bf16 workload; the layers' own arithmetic stays as `store` says (fp64 by
    default).  store="bf16" implies interface="bf16".  `view_b` is either {"H_b": bank rows, "gid_a", "gid_b"} (a detached neighbour view)
    or {"idx": overlap rows, "X_b": second input} (a second live stack on the same graph).
    The last layer's upstream gradient is dH_top plus the alignment gradient.  With `head`
    ({"params", "lab_idx", "lab_y"}) the head's gradient (MeanAgg, MLP, masked BCE; Eq. 18-19)
    replaces dH_top, the joint objective L_BCE + dloss * L_CCA (Eq. 20, dloss = lambda_CCA) is
    returned as res["head_loss"], and res["head_grads"] holds the head's parameter gradients."""
    offs, rels = graph["type_offsets"], graph["rels"]
    csr = build_csr(graph["src"], graph["dst"], graph["rel"], offs, rels)

    # layer outputs and gradients passed between layers are tensors of the storage type
    io = round_bf16 if (store == "bf16" or interface == "bf16") else (lambda x: x)

    def run_stack(H0):
        hs = [np.asarray(H0, F64)]
        for p in params:
            hs.append(io(layer_forward(csr, offs, rels, p, hs[-1], act, layernorm, ln_eps, store)[0]))
        return hs

    def back_stack(hs, dtop):
        grads = [None] * len(params)
        dh = io(dtop)
        for l in range(len(params) - 1, -1, -1):
            dh, grads[l] = layer_backward(csr, offs, rels, params[l], hs[l], dh, act, layernorm, ln_eps, store)
            dh = io(dh)
        return dh, grads

    hs = run_stack(X)
    from . import head as head_mod  # the head module builds on this one

    def head_terms(Htop, ia, Hb, ib, l_cca):
        hl = head_mod.head_loss(Htop, ia, Hb, ib, head["lab_idx"], head["lab_y"], head["params"], cca_loss=l_cca,
                                lambda_cca=dloss, store=store)
        hb = head_mod.head_backward(Htop, ia, Hb, ib, head["lab_idx"], head["lab_y"], head["params"], dloss=1.0,
                                    store=store)
        return (hl["total"], hl["bce"]), hb

    if view_b is None:  # first subgraph of a sequence: no alignment term
        res = dict(H=hs, loss=(0.0, 0.0, 0.0), idx_a=np.zeros(0, np.int64), idx_b=np.zeros(0, np.int64))
        dtop = np.asarray(dH_top, F64) if head is None else None
        if head is not None:
            none = np.zeros(0, np.int64)
            res["head_loss"], hb = head_terms(hs[-1], none, None, none, 0.0)
            res["head_grads"] = {k: hb[k] for k in ("dW1", "db1", "dw2", "db2")}
            dtop = hb["dH"]
        res["dX"], res["grads"] = back_stack(hs, dtop)
        return res
    if "H_b" in view_b:
        ia, ib = overlap_intersect(view_b["gid_a"], view_b["gid_b"])
        Hb = view_b["H_b"]
        hs_b = None
    else:
        ia = ib = np.asarray(view_b["idx"], np.int64)
        hs_b = run_stack(view_b["X_b"])
        Hb = hs_b[-1]
    loss = align_forward(hs[-1], ia, Hb, ib, lambda_n, var_eps)
    dA, dB = align_backward(hs[-1], ia, Hb, ib, lambda_n, var_eps, dloss)
    res = dict(H=hs, loss=loss, idx_a=ia, idx_b=ib)
    if head is None:
        dtop = np.asarray(dH_top, F64) + dA
    else:
        res["head_loss"], hb = head_terms(hs[-1], ia, Hb, ib, loss[0])
        res["head_grads"] = {k: hb[k] for k in ("dW1", "db1", "dw2", "db2")}
        dtop = hb["dH"] + dA
        dB = dB + hb["dH_rep"]
    dX, grads = back_stack(hs, dtop)
    res["dX"], res["grads"] = dX, grads
    if hs_b is not None:
        res["dX_b"], res["grads_b"] = back_stack(hs_b, dB)
        res["H_b"] = hs_b
    return res
