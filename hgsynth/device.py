"""The workload recipe of graphs.py drawn on a torch device, for the benchmark's full-size instances.

graphs.py (numpy) needs minutes for a 200M-edge graph and its feature table; the benchmark only
needs an instance of the same recipe, not the same numbers, so it draws them here with torch's
generator on the GPU in about a second.  The deterministic parts of the recipe are shared with
graphs.py (the rank-frequency out-degree sequence with its cap / floor and exact rounding, the
relation table, the layer / head weights, the ring's global-id ranges); the random draws (node
rank permutations, Zipf destinations, the global edge shuffle, features, overlap sets, global ids,
labels) follow the same distributions with torch's stream, so the values differ from graphs.py.
The oracle never reads these instances (its CPU baseline samples come from graphs.py).

Like graphs.py, this module holds none of the method's arithmetic.
"""
from __future__ import annotations

import functools

import numpy as np
import torch

from . import graphs as G

_MIX = (0x9E3779B1, 0x85EBCA77, 0xC2B2AE3D, 0x27D4EB2F)


def _gen(device, *key) -> torch.Generator:
    """A torch generator seeded from integer key parts (same roles as graphs.py's seed keys)."""
    h = 0x165667B1
    for i, k in enumerate(key):
        h = (h * 31 + (int(k) + 1) * _MIX[i % 4]) & 0x7FFFFFFFFFFFFFFF
    g = torch.Generator(device=device)
    g.manual_seed(h)
    return g


@functools.lru_cache(maxsize=64)
def _out_degrees_cached(n_src: int, e_r: int, s: float, cap, floor) -> np.ndarray:
    return G._out_degrees(n_src, e_r, s, cap, floor)


def _bf16_store(x: torch.Tensor, dtype: str) -> torch.Tensor:
    return x.to(torch.bfloat16) if dtype == "bf16" else x.to(torch.float32)


def make_graph(sp: G.GraphSpec, sub: int = 0, device="cuda") -> dict:
    """COO edges (int32 src, dst, rel tensors on `device`) with graphs.py's recipe: per relation the
    exact rank-frequency out-degree sequence over a random rank permutation of the source type,
    destinations i.i.d. Zipf(s) over a second permutation of the destination type, one global
    shuffle."""
    g = _gen(device, sp.seed, sub, 0)
    sizes = (sp.n_user, sp.n_risk)
    offs = (0, sp.n_user)
    src_perm = [torch.randperm(n, generator=g, device=device) for n in sizes]
    dst_perm = [torch.randperm(n, generator=g, device=device) for n in sizes]
    rels = sp.rels
    n_user_src = sum(1 for (s, _) in rels if s == 0)
    srcs, dsts, rs = [], [], []
    for r, (ts, tt) in enumerate(rels):
        e_r = sp.num_edges // sp.num_rels + (sp.num_edges % sp.num_rels if r == 0 else 0)
        floor = None
        if sp.hub_floor is not None and ts == 0:
            floor = (sp.hub_floor[0], -(-sp.hub_floor[1] // n_user_src))
        deg = torch.from_numpy(_out_degrees_cached(sizes[ts], e_r, sp.zipf_s, sp.out_cap, floor)).to(device)
        src = torch.repeat_interleave(src_perm[ts], deg, output_size=e_r) + offs[ts]
        w = torch.arange(1, sizes[tt] + 1, dtype=torch.float64, device=device) ** (-sp.zipf_s)
        cdf = torch.cumsum(w, 0)
        cdf /= cdf[-1].clone()
        u = torch.rand(e_r, dtype=torch.float64, generator=g, device=device)
        rank = torch.clamp(torch.searchsorted(cdf, u, right=True), max=sizes[tt] - 1)
        dst = dst_perm[tt][rank] + offs[tt]
        srcs.append(src.to(torch.int32))
        dsts.append(dst.to(torch.int32))
        rs.append(torch.full((e_r,), r, dtype=torch.int32, device=device))
        del w, cdf, u, rank
    src = torch.cat(srcs)
    dst = torch.cat(dsts)
    rel = torch.cat(rs)
    del srcs, dsts, rs
    order = torch.randperm(src.shape[0], generator=g, device=device)
    return {"src": src[order], "dst": dst[order], "rel": rel[order],
            "type_offsets": np.array([0, sp.n_user, sp.n_user + sp.n_risk], np.int64), "rels": tuple(rels)}


def make_features(sp: G.GraphSpec, sub: int = 0, device="cuda", key: int = 1, rows: int | None = None) -> torch.Tensor:
    """N(0,1) rows in the storage type (key 1: input features, 3: second view / bank, 4: upstream
    gradient, as in graphs.py)."""
    g = _gen(device, sp.seed + key, sub)
    n = sp.num_nodes if rows is None else rows
    return _bf16_store(torch.randn(n, sp.d, generator=g, device=device), sp.dtype)


def overlap_nodes(sp: G.GraphSpec, graph: dict, sub: int = 0, device="cuda") -> torch.Tensor:
    """Sorted local ids (int32) of the overlap set: uniform over all nodes, or over the long tail
    (total degree <= 2) when sp.overlap == "longtail"."""
    g = _gen(device, sp.seed + 2, sub)
    n = sp.num_nodes
    if sp.overlap == "uniform":
        chosen = torch.randperm(n, generator=g, device=device)[: sp.n_overlap]
    else:
        deg = torch.bincount(graph["src"], minlength=n) + torch.bincount(graph["dst"], minlength=n)
        cand = torch.nonzero(deg <= 2).flatten()
        if cand.shape[0] >= sp.n_overlap:
            chosen = cand[torch.randperm(cand.shape[0], generator=g, device=device)[: sp.n_overlap]]
        else:
            chosen = torch.argsort(deg, stable=True)[: sp.n_overlap]
    return torch.sort(chosen).values.to(torch.int32)


def global_ids(sp: G.GraphSpec, overlap_local: torch.Tensor, sub: int = 0, device="cuda"):
    """Ascending int64 global ids of this subgraph (gid_a) and of a neighbour of the same type sizes
    (gid_b) that shares exactly the overlap nodes; ids drawn from an ID_SPACE_SCALE times larger
    space per type, users below risk events."""
    g = _gen(device, sp.seed + 2, sub, 1)
    su, sr = G.ID_SPACE_SCALE * sp.n_user, G.ID_SPACE_SCALE * sp.n_risk

    def pick(space, count, base):
        return base + torch.sort(torch.randperm(space, generator=g, device=device)[:count]).values

    gid_a = torch.cat([pick(su, sp.n_user, 0), pick(sr, sp.n_risk, su)])
    shared = gid_a[overlap_local.long()]
    parts = []
    for base, space, n_t in ((0, su, sp.n_user), (su, sr, sp.n_risk)):
        mine = gid_a[(gid_a >= base) & (gid_a < base + space)] - base
        sh = shared[(shared >= base) & (shared < base + space)]
        used = torch.zeros(space, dtype=torch.bool, device=device)
        used[mine] = True
        free = torch.nonzero(~used).flatten()
        fresh = base + free[torch.randperm(free.shape[0], generator=g, device=device)[: n_t - sh.shape[0]]]
        parts.append(torch.sort(torch.cat([sh, fresh])).values)
    return gid_a, torch.cat(parts)


def make_labels(sp: G.GraphSpec, sub: int = 0, device="cuda"):
    """Labelled user rows (ascending int32) and 0/1 labels (fp32): each user labelled with
    probability LABELLED_FRACTION, each label positive with probability POSITIVE_RATE."""
    g = _gen(device, sp.seed + 5, sub)
    rows = torch.nonzero(torch.rand(sp.n_user, generator=g, device=device) < G.LABELLED_FRACTION).flatten()
    y = (torch.rand(rows.shape[0], generator=g, device=device) < G.POSITIVE_RATE).to(torch.float32)
    return rows.to(torch.int32), y


def make_workload(sp: G.GraphSpec, sub: int = 0, device="cuda", with_dH_top: bool = False) -> dict:
    """Every input of one step of the workload, on `device`: graph, X, layer weights (graphs.py's,
    deterministic), the second view (perturbed copy, or a neighbour's embeddings with both id
    lists), labels, and optionally a synthetic upstream gradient."""
    w = {"spec": sp, "graph": make_graph(sp, sub, device), "X": make_features(sp, sub, device, 1),
         "params": [G.make_layer_params(sp, l) for l in range(sp.layers)]}
    ov = overlap_nodes(sp, w["graph"], sub, device)
    w["overlap_local"] = ov
    if sp.view_b == "perturbed":
        w["X_b"] = _bf16_store(w["X"].float() + 0.1 * make_features(sp, sub, device, 3).float(), sp.dtype)
    else:
        w["H_b"] = make_features(sp, sub, device, 3)
        w["gid_a"], w["gid_b"] = global_ids(sp, ov, sub, device)
    w["lab_idx"], w["lab_y"] = make_labels(sp, sub, device)
    if with_dH_top:
        w["dH_top"] = make_features(sp, sub, device, 4)
    return w


def ring_features(sp: G.GraphSpec, device="cuda") -> torch.Tensor:
    """One feature row per global id of the whole ring (a node shared by two subgraphs has one row)."""
    last = G.ring_ids(sp, sp.num_subgraphs - 1)
    return make_features(sp, 0, device, 1, rows=int(last[-1]) + 1)


def make_ring_part(sp: G.GraphSpec, k: int, table: torch.Tensor, device="cuda") -> dict:
    """Subgraph k of the ring: its own edges (keyed by k), the global ids of graphs.py's ring_ids
    (consecutive subgraphs share n_overlap ids), feature rows looked up in the ring's table, labels."""
    gid = torch.from_numpy(G.ring_ids(sp, k)).to(device)
    lab, y = make_labels(sp, k, device)
    return {"graph": make_graph(sp, k, device), "gid": gid, "X": table[gid], "lab_idx": lab, "lab_y": y}
