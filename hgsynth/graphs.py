"""Graph, feature, weight and overlap-set generators (seeded, numpy only).

Recipe (stated once here, repeated in the design notes):

* Node types: 0 = user, 1 = risk event; local ids are contiguous per type, users first
  (type_offsets = [0, n_user, n_user + n_risk]).
* Relations: the first R entries of RELATIONS, (src type, dst type) each; forward relations and
  their inverses (Section 2.2).  Relation r receives floor(E / R) edges, r0 takes the remainder.
* Out-degree: rank-frequency Zipf.  The source node of rank k (ranks drawn by a seeded permutation
  of the source type, shared by every relation with that source type, so hubs are hubs in all of
  them) expects E_r * k^-s / sum_k k^-s edges; an optional cap is applied by water-filling, an
  optional floor on the top ranks likewise, then largest-remainder rounding makes the sum exact.
* Destinations: i.i.d. rank-frequency Zipf(s) over an independent permutation of the destination
  type, so in-degrees are power-law too and forward hubs exist.
* Edge order: one seeded global shuffle (the COO input is unordered).  Multi-edges and self-loops
  are kept.
* Features ~ N(0,1) fp32, rounded to nearest-even bf16 for bf16 workloads.  Weights: Xavier
  uniform U(+-sqrt(6 / (2d))), biases 0, LayerNorm gain 1 / shift 0 (or small random affine
  values for tests, so that bias and affine bugs cannot hide behind zeros).
* Overlap set: "longtail" draws uniformly among nodes of total degree <= 2 (their h-index is <= 2,
  the paper's threshold, because an h-index never exceeds the degree); "uniform" draws among all
  nodes.  Global ids are sorted random draws from an 8x larger id space, users below risk events,
  so local order equals global-id order.
* Labels: 11.7 % of the users of a subgraph are labelled (the paper leaves 88.3 % unlabelled),
  5 % of those positive (the paper gives no rate).  Head weights: Xavier uniform W1 (d x d) and
  w2 (d), zero biases.
* Seeds: graph = seed, features = seed+1, overlap = seed+2, second view / bank = seed+3,
  upstream gradient = seed+4, labels = seed+5, temporal context = seed+6, layer l weights =
  seed+100+l, head weights = seed+200, temporal weights = seed+300; subgraph k mixes k into each
  seed.
* Temporal context: the w = 3 earlier states of every node, N(0,1) rounded to the storage type.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

RELATIONS = ((0, 0), (0, 1), (1, 0), (0, 1), (1, 0), (0, 0))
ID_SPACE_SCALE = 8


@dataclasses.dataclass(frozen=True)
class GraphSpec:
    name: str
    n_user: int
    n_risk: int
    num_rels: int
    num_edges: int
    zipf_s: float
    d: int
    dtype: str  # "f32" or "bf16": storage type of features, weights and activations
    layers: int
    n_overlap: int
    overlap: str  # "uniform" | "longtail"
    view_b: str  # "perturbed": live second stack on X + 0.1 N(0,1); "bank": fixed N(0,1) rows of a neighbour subgraph
    seed: int = 0
    out_cap: int | None = None  # max out-degree of one node within one relation
    hub_floor: tuple | None = None  # (count, total): top `count` user sources get >= total out-edges over user-source relations
    num_subgraphs: int = 1

    @property
    def num_nodes(self) -> int:
        return self.n_user + self.n_risk

    @property
    def rels(self):
        return RELATIONS[: self.num_rels]


WORKLOADS = {
    # 10k nodes / 100k edges, fp32 d=64, two live views (the perturbed copy is the second view).
    "tiny-10k": GraphSpec("tiny-10k", 8_000, 2_000, 3, 100_000, 1.5, 64, "f32", 2, 1_000, "uniform", "perturbed"),
    # 1M nodes / 20M edges, bf16 d=128, 130,435 long-tail overlap nodes (15 % of an 869,565-node base partition).
    "sub-1m": GraphSpec("sub-1m", 900_000, 100_000, 5, 20_000_000, 1.3, 128, "bf16", 2, 130_435, "longtail", "bank"),
    # 10M nodes / 200M edges, top-100 user hubs with >= 500k out-edges, 3 layers.
    "big-10m": GraphSpec("big-10m", 9_000_000, 1_000_000, 6, 200_000_000, 1.2, 128, "bf16", 3, 1_000_000, "uniform",
                         "bank", hub_floor=(100, 500_000)),
    # 16 subgraphs of 2M nodes / 40M edges, 400k nodes shared by consecutive subgraphs.
    "ring16-2m": GraphSpec("ring16-2m", 1_800_000, 200_000, 4, 40_000_000, 1.3, 128, "bf16", 2, 400_000, "uniform",
                           "bank", num_subgraphs=16),
    # 5M nodes / 100M edges, Zipf s=1.05 capped at 2M out-edges, bf16 d=256.
    "tail-5m": GraphSpec("tail-5m", 4_500_000, 500_000, 3, 100_000_000, 1.05, 256, "bf16", 2, 500_000, "uniform",
                         "bank", out_cap=2_000_000),
}


def spec(name: str, **overrides) -> GraphSpec:
    """A named workload, optionally with fields replaced (smaller test variants of the same recipe)."""
    s = WORKLOADS[name]
    return dataclasses.replace(s, **overrides) if overrides else s


def bf16_round(x) -> np.ndarray:
    """Round fp32 values to the nearest bfloat16 (ties to even); returns fp32 holding those values."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000).astype(np.uint32)
    return r.view(np.float32).reshape(x.shape)


def _store(x: np.ndarray, dtype: str) -> np.ndarray:
    x = np.asarray(x, dtype=np.float32)
    return bf16_round(x) if dtype == "bf16" else np.ascontiguousarray(x)


def _rng(*key) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([int(k) for k in key]))


def _waterfill_cap(x: np.ndarray, cap: float) -> np.ndarray:
    x = x.copy()
    capped = np.zeros(x.shape, bool)
    for _ in range(64):
        over = x > cap
        if not over.any():
            break
        excess = float((x[over] - cap).sum())
        x[over] = cap
        capped |= over
        free = ~capped
        x[free] += excess * x[free] / x[free].sum()
    return x


def _floor_top(x: np.ndarray, count: int, floor: float) -> np.ndarray:
    x = x.copy()
    deficit = float(np.maximum(floor - x[:count], 0).sum())
    x[:count] = np.maximum(x[:count], floor)
    rest = x[count:]
    x[count:] = rest - deficit * rest / rest.sum()
    return x


def _round_to_total(x: np.ndarray, total: int) -> np.ndarray:
    base = np.floor(x).astype(np.int64)
    short = int(total - base.sum())
    if short > 0:
        frac = x - base
        order = np.argsort(-frac, kind="stable")[:short]
        base[order] += 1
    elif short < 0:  # only from floating error; take from the largest entries
        order = np.argsort(-x, kind="stable")[: -short]
        base[order] -= 1
    return base


def _out_degrees(n_src: int, e_r: int, s: float, cap, floor) -> np.ndarray:
    w = np.arange(1, n_src + 1, dtype=np.float64) ** (-s)
    x = e_r * w / w.sum()
    if floor is not None:
        x = _floor_top(x, floor[0], floor[1])
    if cap is not None:
        x = _waterfill_cap(x, float(cap))
    return _round_to_total(x, e_r)


def make_graph(sp: GraphSpec, sub: int = 0) -> dict:
    """COO edge list (src, dst, rel as int32 node / relation ids) plus type and relation tables."""
    rng = _rng(sp.seed, sub, 0)
    sizes = (sp.n_user, sp.n_risk)
    offs = (0, sp.n_user)
    src_perm = [rng.permutation(n).astype(np.int64) for n in sizes]
    dst_perm = [rng.permutation(n).astype(np.int64) for n in sizes]
    rels = sp.rels
    n_user_src = sum(1 for (s, _) in rels if s == 0)
    srcs, dsts, rs = [], [], []
    for r, (ts, tt) in enumerate(rels):
        e_r = sp.num_edges // sp.num_rels + (sp.num_edges % sp.num_rels if r == 0 else 0)
        floor = None
        if sp.hub_floor is not None and ts == 0:
            floor = (sp.hub_floor[0], math.ceil(sp.hub_floor[1] / n_user_src))
        deg = _out_degrees(sizes[ts], e_r, sp.zipf_s, sp.out_cap, floor)
        src = np.repeat(src_perm[ts], deg) + offs[ts]
        w = np.arange(1, sizes[tt] + 1, dtype=np.float64) ** (-sp.zipf_s)
        cdf = np.cumsum(w)
        cdf /= cdf[-1]
        rank = np.minimum(np.searchsorted(cdf, rng.random(e_r), side="right"), sizes[tt] - 1)
        dst = dst_perm[tt][rank] + offs[tt]
        srcs.append(src.astype(np.int32))
        dsts.append(dst.astype(np.int32))
        rs.append(np.full(e_r, r, np.int32))
    src = np.concatenate(srcs)
    dst = np.concatenate(dsts)
    rel = np.concatenate(rs)
    order = rng.permutation(src.shape[0])
    return {
        "src": src[order],
        "dst": dst[order],
        "rel": rel[order],
        "type_offsets": np.array([0, sp.n_user, sp.n_user + sp.n_risk], np.int64),
        "rels": tuple(rels),
    }


def degree_stats(g: dict) -> dict:
    n = int(g["type_offsets"][-1])
    out_deg = np.bincount(g["src"], minlength=n)
    in_deg = np.bincount(g["dst"], minlength=n)
    top = np.sort(out_deg)[::-1][:100]
    return {
        "max_out_degree": int(out_deg.max()),
        "max_in_degree": int(in_deg.max()),
        "frac_out_degree_le2": float((out_deg <= 2).mean()),
        "top100_min_out_degree": int(top.min()),
    }


def make_features(sp: GraphSpec, sub: int = 0) -> np.ndarray:
    rng = _rng(sp.seed + 1, sub)
    return _store(rng.standard_normal((sp.num_nodes, sp.d), dtype=np.float32), sp.dtype)


def make_layer_params(sp: GraphSpec, layer: int, random_affine: bool = False, bias_margin: float | None = None) -> dict:
    """Per-layer weights: W_rel[r] (d_in x d_out), W_agg[t], b_agg[t], ln_gamma[t], ln_beta[t].

    bias_margin: biases of +-margin per column (seeded signs), which keep pre-activations away from
    the activation's kink so that the ReLU decisions of two implementations cannot differ."""
    rng = _rng(sp.seed + 100 + layer)
    d = sp.d
    a = math.sqrt(6.0 / (2 * d))
    W_rel = rng.uniform(-a, a, size=(sp.num_rels, d, d)).astype(np.float32)
    W_agg = rng.uniform(-a, a, size=(2, d, d)).astype(np.float32)
    if random_affine:
        b = 0.1 * rng.standard_normal((2, d), dtype=np.float32)
        gamma = 1.0 + 0.1 * rng.standard_normal((2, d), dtype=np.float32)
        beta = 0.1 * rng.standard_normal((2, d), dtype=np.float32)
    else:
        b = np.zeros((2, d), np.float32)
        gamma = np.ones((2, d), np.float32)
        beta = np.zeros((2, d), np.float32)
    if bias_margin is not None:
        b = (bias_margin * rng.choice([-1.0, 1.0], size=(2, d))).astype(np.float32)
    return {k: _store(v, sp.dtype) for k, v in
            dict(W_rel=W_rel, W_agg=W_agg, b_agg=b, ln_gamma=gamma, ln_beta=beta).items()}


def overlap_nodes(sp: GraphSpec, g: dict, sub: int = 0) -> np.ndarray:
    """Sorted local ids of the overlap set B inside this subgraph."""
    rng = _rng(sp.seed + 2, sub)
    n = sp.num_nodes
    if sp.overlap == "uniform":
        chosen = rng.choice(n, sp.n_overlap, replace=False)
    else:
        deg = np.bincount(g["src"], minlength=n) + np.bincount(g["dst"], minlength=n)
        cand = np.flatnonzero(deg <= 2)
        if cand.shape[0] >= sp.n_overlap:
            chosen = rng.choice(cand, sp.n_overlap, replace=False)
        else:
            chosen = np.argsort(deg, kind="stable")[: sp.n_overlap]
    return np.sort(chosen).astype(np.int32)


def _sorted_ids(rng, space: int, count: int, base: int) -> np.ndarray:
    return base + np.sort(rng.choice(space, count, replace=False)).astype(np.int64)


def global_ids(sp: GraphSpec, overlap_local: np.ndarray, sub: int = 0):
    """Global ids of this subgraph (gid_a) and of a neighbour subgraph (gid_b) of the same type sizes,
    sharing exactly the overlap nodes.  Both lists are strictly ascending."""
    rng = _rng(sp.seed + 2, sub, 1)
    su, sr = ID_SPACE_SCALE * sp.n_user, ID_SPACE_SCALE * sp.n_risk
    gid_a = np.concatenate([_sorted_ids(rng, su, sp.n_user, 0), _sorted_ids(rng, sr, sp.n_risk, su)])
    shared = gid_a[overlap_local]
    parts = []
    for base, space, n_t in ((0, su, sp.n_user), (su, sr, sp.n_risk)):
        mine = gid_a[(gid_a >= base) & (gid_a < base + space)] - base
        sh = shared[(shared >= base) & (shared < base + space)]
        used = np.zeros(space, bool)
        used[mine] = True
        free = np.flatnonzero(~used)
        fresh = base + rng.choice(free, n_t - sh.shape[0], replace=False).astype(np.int64)
        parts.append(np.sort(np.concatenate([sh, fresh])))
    gid_b = np.concatenate(parts)
    return gid_a, gid_b


@dataclasses.dataclass
class Workload:
    spec: GraphSpec
    graph: dict
    X: np.ndarray
    params: list
    overlap_local: np.ndarray
    gid_a: np.ndarray | None
    gid_b: np.ndarray | None
    X_b: np.ndarray | None  # second view's input features ("perturbed")
    H_b: np.ndarray | None  # neighbour subgraph's embeddings ("bank")
    dH_top: np.ndarray  # upstream gradient of the last layer's output (stands in for the prediction head)


def make_workload(sp: GraphSpec, sub: int = 0, random_affine: bool = False, with_ids: bool = True,
                  bias_margin: float | None = None) -> Workload:
    g = make_graph(sp, sub)
    X = make_features(sp, sub)
    params = [make_layer_params(sp, l, random_affine, bias_margin) for l in range(sp.layers)]
    ov = overlap_nodes(sp, g, sub)
    rng3 = _rng(sp.seed + 3, sub)
    X_b = H_b = None
    gid_a = gid_b = None
    if sp.view_b == "perturbed":
        X_b = _store(X + 0.1 * rng3.standard_normal(X.shape, dtype=np.float32), sp.dtype)
    else:
        H_b = _store(rng3.standard_normal((sp.num_nodes, sp.d), dtype=np.float32), sp.dtype)
        if with_ids:
            gid_a, gid_b = global_ids(sp, ov, sub)
    rng4 = _rng(sp.seed + 4, sub)
    dH_top = _store(rng4.standard_normal((sp.num_nodes, sp.d), dtype=np.float32), sp.dtype)
    return Workload(sp, g, X, params, ov, gid_a, gid_b, X_b, H_b, dH_top)


# ------------------------------------------------------------------------------------------------
# ring of overlapping subgraphs: subgraph k shares its first n_overlap nodes (split between the
# types in proportion to their sizes) with subgraph k-1 and its last ones with subgraph k+1
# ------------------------------------------------------------------------------------------------
FEATURE_BLOCK = 1 << 16


def _global_features(sp: GraphSpec, gids: np.ndarray) -> np.ndarray:
    """Feature rows keyed by global id (blocks of 65,536 ids share one seeded draw), so a node
    shared by two subgraphs has the same row in both."""
    out = np.empty((gids.shape[0], sp.d), np.float32)
    blocks = gids // FEATURE_BLOCK
    for b in np.unique(blocks):
        sel = np.flatnonzero(blocks == b)
        rows = _rng(sp.seed + 1, int(b), 7).standard_normal((FEATURE_BLOCK, sp.d), dtype=np.float32)
        out[sel] = rows[gids[sel] - b * FEATURE_BLOCK]
    return _store(out, sp.dtype)


def ring_ids(sp: GraphSpec, k: int) -> np.ndarray:
    """Sorted global ids of subgraph k of the ring (users below risk events)."""
    ov_u = round(sp.n_overlap * sp.n_user / sp.num_nodes)
    ov_r = sp.n_overlap - ov_u
    span_u = sp.num_subgraphs * (sp.n_user - ov_u) + ov_u
    u = k * (sp.n_user - ov_u) + np.arange(sp.n_user, dtype=np.int64)
    r = span_u + k * (sp.n_risk - ov_r) + np.arange(sp.n_risk, dtype=np.int64)
    return np.concatenate([u, r])


@dataclasses.dataclass
class RingPart:
    k: int
    graph: dict
    X: np.ndarray
    gid: np.ndarray
    dH_top: np.ndarray


def make_ring_part(sp: GraphSpec, k: int) -> RingPart:
    """Subgraph k of the ring: its own edges (seeded by k), features of its global ids."""
    g = make_graph(sp, sub=k)
    gid = ring_ids(sp, k)
    X = _global_features(sp, gid)
    dH_top = _store(_rng(sp.seed + 4, k).standard_normal((sp.num_nodes, sp.d), dtype=np.float32), sp.dtype)
    return RingPart(k, g, X, gid, dH_top)


# ------------------------------------------------------------------------------------------------
# labels and prediction-head weights
# ------------------------------------------------------------------------------------------------
LABELLED_FRACTION = 0.117  # the paper's data leaves 88.3 % of users unlabelled (Section 4.1)
POSITIVE_RATE = 0.05  # not given by the paper; a rare positive class, as in fraud data


def make_labels(sp: GraphSpec, sub: int = 0, fraction: float = LABELLED_FRACTION,
                positive_rate: float = POSITIVE_RATE) -> tuple:
    """Labelled user rows of one subgraph, ascending (int32), and their 0/1 labels (fp32): each user
    is labelled with probability `fraction`, each label is 1 with probability `positive_rate`
    (seed+5)."""
    rng = _rng(sp.seed + 5, sub)
    rows = np.flatnonzero(rng.random(sp.n_user) < fraction).astype(np.int32)
    y = (rng.random(rows.shape[0]) < positive_rate).astype(np.float32)
    return rows, y


def make_head_params(sp: GraphSpec, random_bias: bool = False, bias_margin: float | None = None) -> dict:
    """Two-layer head: W1 (d x d, input x hidden), b1 (d), w2 (d), b2 (1).  Xavier uniform weights,
    zero biases, or small N(0, 0.1) biases for tests (seed+200).  bias_margin: b1 of +-margin per
    hidden unit (seeded signs), keeping the hidden pre-activations away from the ReLU's kink."""
    rng = _rng(sp.seed + 200)
    d = sp.d
    a1 = math.sqrt(6.0 / (2 * d))
    a2 = math.sqrt(6.0 / (d + 1))
    W1 = rng.uniform(-a1, a1, size=(d, d)).astype(np.float32)
    w2 = rng.uniform(-a2, a2, size=(d,)).astype(np.float32)
    if random_bias:
        b1 = 0.1 * rng.standard_normal(d, dtype=np.float32)
        b2 = 0.1 * rng.standard_normal(1, dtype=np.float32)
    else:
        b1 = np.zeros(d, np.float32)
        b2 = np.zeros(1, np.float32)
    if bias_margin is not None:
        b1 = (bias_margin * rng.choice([-1.0, 1.0], size=d)).astype(np.float32)
    return {k: _store(v, sp.dtype) for k, v in dict(W1=W1, b1=b1, w2=w2, b2=b2).items()}


# ------------------------------------------------------------------------------------------------
# temporal module: context states and weights
# ------------------------------------------------------------------------------------------------
TEMPORAL_WINDOW = 3  # w of Section 4.1


def make_context(sp: GraphSpec, w: int = TEMPORAL_WINDOW, sub: int = 0, rows: int | None = None) -> np.ndarray:
    """The w earlier states of every node (w x N x d), N(0,1) rounded to the storage type (seed+6);
    block k holds the states k + 1 snapshots back."""
    n = sp.num_nodes if rows is None else rows
    rng = _rng(sp.seed + 6, sub)
    return _store(rng.standard_normal((w, n, sp.d), dtype=np.float32), sp.dtype)


def make_temporal_params(sp: GraphSpec) -> dict:
    """Attention Wa (d x d) and r (d), GRU W_i, W_h (d x 3d) and b_i, b_h (3d) (seed+300): Xavier
    uniform Wa, r ~ N(0, 4/d), and the GRU's usual U(+-1/sqrt(d)) for its weights and biases."""
    rng = _rng(sp.seed + 300)
    d = sp.d
    a = math.sqrt(6.0 / (2 * d))
    k = 1.0 / math.sqrt(d)
    p = {"Wa": rng.uniform(-a, a, (d, d)), "r": 2.0 * rng.standard_normal(d) / math.sqrt(d),
         "W_i": rng.uniform(-k, k, (d, 3 * d)), "W_h": rng.uniform(-k, k, (d, 3 * d)),
         "b_i": rng.uniform(-k, k, 3 * d), "b_h": rng.uniform(-k, k, 3 * d)}
    return {key: _store(v.astype(np.float32), sp.dtype) for key, v in p.items()}


def make_hgt_params(sp: GraphSpec, heads: int, layer: int = 0, bias_margin: float | None = None) -> dict:
    """Attention layer weights (seed+400+layer): Xavier uniform W_K, W_Q, W_V, W_agg (T x d x d); W_att,
    W_msg (R x S x d_h x d_h) ~ N(0, 1/d_h); mu = 1 (fp32); small N(0, 0.1) biases and LayerNorm
    shifts, gains 1 + N(0, 0.1); bias_margin: b_agg of +-margin per column (seeded signs)."""
    rng = _rng(sp.seed + 400 + layer)
    d, R, T = sp.d, sp.num_rels, 2
    dh = d // heads
    a = math.sqrt(6.0 / (2 * d))
    p = {"W_K": rng.uniform(-a, a, (T, d, d)), "W_Q": rng.uniform(-a, a, (T, d, d)),
         "W_V": rng.uniform(-a, a, (T, d, d)),
         "b_K": 0.1 * rng.standard_normal((T, d)), "b_Q": 0.1 * rng.standard_normal((T, d)),
         "b_V": 0.1 * rng.standard_normal((T, d)),
         "W_att": rng.standard_normal((R, heads, dh, dh)) / math.sqrt(dh),
         "W_msg": rng.standard_normal((R, heads, dh, dh)) / math.sqrt(dh),
         "W_agg": rng.uniform(-a, a, (T, d, d)), "b_agg": 0.1 * rng.standard_normal((T, d)),
         "ln_gamma": 1.0 + 0.1 * rng.standard_normal((T, d)), "ln_beta": 0.1 * rng.standard_normal((T, d))}
    if bias_margin is not None:
        p["b_agg"] = bias_margin * rng.choice([-1.0, 1.0], size=(T, d))
    out = {k: _store(np.asarray(v, np.float32), sp.dtype) for k, v in p.items()}
    out["mu"] = np.ones(R, np.float32)
    return out
