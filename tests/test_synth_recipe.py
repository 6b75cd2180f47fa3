"""The seeded synthetic workloads have the shapes their recipe states (CPU).

The generator stands in for the paper's proprietary data set, so these checks pin the stand-in
itself: exact edge counts, the out-degree cap and hub floor of the large workloads, the long-tail
share of the 5M-node workload (65-75 % of the nodes with out-degree <= 2), typed endpoints,
determinism, and the overlap sets and global ids the alignment path relies on."""
import math

import numpy as np
import pytest

import hgsynth
from hgsynth.graphs import WORKLOADS, _out_degrees


def out_degree_by_rank(sp):
    """Per source type, the total out-degree of each rank over the relations leaving that type (ranks
    are shared by those relations), plus the largest per-relation degree and the edge total."""
    sizes = (sp.n_user, sp.n_risk)
    n_user_src = sum(1 for (s, _) in sp.rels if s == 0)
    tot = [np.zeros(n, np.int64) for n in sizes]
    per_rel_max, total = 0, 0
    for r, (ts, _) in enumerate(sp.rels):
        e_r = sp.num_edges // sp.num_rels + (sp.num_edges % sp.num_rels if r == 0 else 0)
        floor = None
        if sp.hub_floor is not None and ts == 0:
            floor = (sp.hub_floor[0], math.ceil(sp.hub_floor[1] / n_user_src))
        deg = _out_degrees(sizes[ts], e_r, sp.zipf_s, sp.out_cap, floor)
        assert deg.sum() == e_r and deg.min() >= 0
        if sp.out_cap is None and floor is None:  # the rank-frequency law: non-increasing in rank
            assert np.all(np.diff(deg) <= 0)
        per_rel_max = max(per_rel_max, int(deg.max()))
        tot[ts] += deg
        total += e_r
    return tot, per_rel_max, total


@pytest.mark.parametrize("name", sorted(WORKLOADS))
def test_edge_totals_and_degree_constraints(name):
    sp = WORKLOADS[name]
    tot, per_rel_max, total = out_degree_by_rank(sp)
    assert total == sp.num_edges
    if sp.out_cap is not None:
        assert per_rel_max <= sp.out_cap
    if sp.hub_floor is not None:
        count, floor = sp.hub_floor
        assert np.sort(tot[0])[::-1][:count].min() >= floor


def test_long_tail_workload_shape():
    # 5M nodes, Zipf s = 1.05 capped at 2M out-edges per relation: 65-75 % of the nodes have
    # out-degree <= 2, and the cap binds (the uncapped law would give the top node ~8.8M edges)
    sp = WORKLOADS["tail-5m"]
    tot, per_rel_max, _ = out_degree_by_rank(sp)
    allo = np.concatenate(tot)
    assert 0.65 <= float((allo <= 2).mean()) <= 0.75
    assert per_rel_max == sp.out_cap


def test_small_graph_structure_and_determinism():
    sp = hgsynth.spec("tiny-10k")
    g = hgsynth.make_graph(sp)
    offs = g["type_offsets"]
    assert len(g["src"]) == sp.num_edges and g["src"].dtype == np.int32
    typ = lambda v: (v >= offs[1]).astype(int)  # noqa: E731
    for r, (ts, tt) in enumerate(g["rels"]):
        m = g["rel"] == r
        assert np.all(typ(g["src"][m]) == ts) and np.all(typ(g["dst"][m]) == tt)
    assert np.all((g["src"] >= 0) & (g["src"] < offs[-1]) & (g["dst"] >= 0) & (g["dst"] < offs[-1]))
    # the COO list is shuffled, and multi-edges occur (they are kept and counted)
    assert not np.all(np.diff(g["rel"]) >= 0)
    key = (g["rel"].astype(np.int64) << 40) | (g["src"].astype(np.int64) << 20) | g["dst"]
    assert np.unique(key).shape[0] < key.shape[0]
    # power-law in-degrees: forward hubs exist
    indeg = np.bincount(g["dst"], minlength=int(offs[-1]))
    assert indeg.max() > 50 * indeg.mean()
    g2 = hgsynth.make_graph(sp)
    assert all(np.array_equal(g[k], g2[k]) for k in ("src", "dst", "rel"))
    g3 = hgsynth.make_graph(sp, sub=1)
    assert not np.array_equal(g["src"], g3["src"])


def test_long_tail_overlap_set_and_global_ids():
    sp = hgsynth.spec("sub-1m", n_user=9_000, n_risk=1_000, num_edges=200_000, n_overlap=1_304)
    w = hgsynth.make_workload(sp)
    g, ov = w.graph, w.overlap_local
    n = sp.num_nodes
    deg = np.bincount(g["src"], minlength=n) + np.bincount(g["dst"], minlength=n)
    assert ov.shape[0] == sp.n_overlap and np.all(np.diff(ov) > 0)
    assert np.all(deg[ov] <= 2)  # h-index <= degree <= 2: the paper's long-tail threshold
    a, b = w.gid_a, w.gid_b
    assert np.all(np.diff(a) > 0) and np.all(np.diff(b) > 0)
    assert np.array_equal(np.intersect1d(a, b), a[ov])
    # users below risk events in both id lists, so local order equals global-id order per type
    su = hgsynth.graphs.ID_SPACE_SCALE * sp.n_user
    assert np.all(a[: sp.n_user] < su) and np.all(a[sp.n_user:] >= su)
    assert np.all(b[: sp.n_user] < su) and np.all(b[sp.n_user:] >= su)


def test_features_and_weights_recipe():
    sp = hgsynth.spec("sub-1m", n_user=9_000, n_risk=1_000, num_edges=100_000, n_overlap=500)
    X = hgsynth.graphs.make_features(sp)
    assert X.shape == (sp.num_nodes, sp.d)
    # bf16 storage: the low 16 bits of every value are zero
    assert np.all((X.view(np.uint32) & 0xFFFF) == 0)
    assert abs(float(X.mean())) < 0.01 and abs(float(X.std()) - 1.0) < 0.01
    p = hgsynth.make_layer_params(sp, 0)
    a = math.sqrt(6.0 / (2 * sp.d))
    assert p["W_rel"].shape == (sp.num_rels, sp.d, sp.d) and p["W_agg"].shape == (2, sp.d, sp.d)
    assert np.abs(p["W_rel"]).max() <= a * (1 + 2 ** -8) and np.abs(p["W_agg"]).max() <= a * (1 + 2 ** -8)
    assert not p["b_agg"].any() and np.all(p["ln_gamma"] == 1) and not p["ln_beta"].any()


def test_ring_of_subgraphs_shares_exactly_the_overlap_with_the_next():
    # 16 subgraphs of 2M nodes; each shares 400k nodes (20 %) with the next and none with the one after
    sp = WORKLOADS["ring16-2m"]
    ids = [hgsynth.graphs.ring_ids(sp, k) for k in range(3)]
    for a in ids:
        assert a.shape[0] == sp.num_nodes and np.all(np.diff(a) > 0)
    assert np.intersect1d(ids[0], ids[1], assume_unique=True).shape[0] == sp.n_overlap
    assert np.intersect1d(ids[1], ids[2], assume_unique=True).shape[0] == sp.n_overlap
    assert np.intersect1d(ids[0], ids[2], assume_unique=True).shape[0] == 0
    # users below risk events, so local order is global-id order within each type
    last = hgsynth.graphs.ring_ids(sp, sp.num_subgraphs - 1)
    assert last[sp.n_user - 1] < ids[0][sp.n_user]


def test_ring_parts_carry_identical_rows_for_shared_nodes():
    sp = hgsynth.spec("ring16-2m", n_user=9_000, n_risk=1_000, num_edges=50_000, n_overlap=2_000, d=64)
    p0, p1 = hgsynth.graphs.make_ring_part(sp, 0), hgsynth.graphs.make_ring_part(sp, 1)
    shared, i0, i1 = np.intersect1d(p0.gid, p1.gid, return_indices=True)
    assert shared.shape[0] == sp.n_overlap
    assert np.array_equal(p0.X[i0], p1.X[i1])
    # independent edges per subgraph, and different rows for different nodes
    assert not np.array_equal(p0.graph["src"], p1.graph["src"])
    assert not np.array_equal(p0.X[: sp.n_overlap], p1.X[: sp.n_overlap])
