"""The benchmark's device-side generator (hgsynth.device) follows the recipe of hgsynth.graphs:
checked on the CPU (torch's CPU generator) on reduced instances of the workloads."""
import numpy as np
import torch

import hgsynth
from hgsynth import device as D
from hgsynth import graphs as G


def _np(t):
    return t.cpu().numpy()


def test_graph_recipe_edge_totals_degrees_and_types():
    sp = hgsynth.spec("big-10m", n_user=9_000, n_risk=1_000, num_edges=200_003, n_overlap=1_000,
                      hub_floor=(10, 2_000))
    g = D.make_graph(sp, device="cpu")
    src, dst, rel = _np(g["src"]), _np(g["dst"]), _np(g["rel"])
    offs = g["type_offsets"]
    assert len(src) == sp.num_edges and src.dtype == np.int32
    n_user_src = sum(1 for s, _ in sp.rels if s == 0)
    for r, (ts, tt) in enumerate(sp.rels):
        m = rel == r
        e_r = sp.num_edges // sp.num_rels + (sp.num_edges % sp.num_rels if r == 0 else 0)
        assert m.sum() == e_r
        assert np.all((src[m] >= offs[ts]) & (src[m] < offs[ts + 1]))
        assert np.all((dst[m] >= offs[tt]) & (dst[m] < offs[tt + 1]))
        floor = (sp.hub_floor[0], -(-sp.hub_floor[1] // n_user_src)) if ts == 0 else None
        want = np.sort(G._out_degrees(int(offs[ts + 1] - offs[ts]), e_r, sp.zipf_s, sp.out_cap, floor))
        got = np.sort(np.bincount(src[m] - offs[ts], minlength=int(offs[ts + 1] - offs[ts])))
        assert np.array_equal(got, want), r  # the same exact out-degree sequence as graphs.py
        # destinations: Zipf in-degrees, so the busiest destination is far above the mean
        indeg = np.bincount(dst[m] - offs[tt])
        assert indeg.max() > 20 * e_r / (offs[tt + 1] - offs[tt])
    # the input order is shuffled (not grouped by relation)
    assert (np.diff(rel) != 0).sum() > 1000
    g2 = D.make_graph(sp, device="cpu")
    assert torch.equal(g["src"], g2["src"]) and torch.equal(g["dst"], g2["dst"])  # seeded


def test_overlap_sets_ids_and_labels():
    sp = hgsynth.spec("sub-1m", n_user=18_000, n_risk=2_000, num_edges=300_000, n_overlap=2_609)
    w = D.make_workload(sp, device="cpu")
    g = w["graph"]
    n = sp.num_nodes
    ov = _np(w["overlap_local"])
    deg = np.bincount(_np(g["src"]), minlength=n) + np.bincount(_np(g["dst"]), minlength=n)
    assert len(ov) == sp.n_overlap and np.all(np.diff(ov) > 0) and np.all(deg[ov] <= 2)  # long tail
    ga, gb = _np(w["gid_a"]), _np(w["gid_b"])
    assert len(ga) == len(gb) == n and np.all(np.diff(ga) > 0) and np.all(np.diff(gb) > 0)
    common = np.intersect1d(ga, gb)
    assert np.array_equal(common, ga[ov])  # exactly the overlap nodes are shared
    assert np.all(ga[: sp.n_user] < G.ID_SPACE_SCALE * sp.n_user) and np.all(ga[sp.n_user:] >= G.ID_SPACE_SCALE * sp.n_user)
    X = w["X"]
    assert X.dtype == torch.bfloat16 and X.shape == (n, sp.d)
    assert abs(float(X.float().mean())) < 0.01 and abs(float(X.float().std()) - 1) < 0.01
    lab, y = _np(w["lab_idx"]), _np(w["lab_y"])
    assert np.all(lab < sp.n_user) and np.all(np.diff(lab) > 0)
    assert abs(len(lab) / sp.n_user - G.LABELLED_FRACTION) < 0.01 and 0.02 < y.mean() < 0.08


def test_ring_parts_share_ids_and_feature_rows():
    sp = hgsynth.spec("ring16-2m", n_user=9_000, n_risk=1_000, num_edges=50_000, n_overlap=2_000, num_subgraphs=3)
    table = D.ring_features(sp, device="cpu")
    parts = [D.make_ring_part(sp, k, table, device="cpu") for k in range(3)]
    a, b, c = (_np(p["gid"]) for p in parts)
    ab, ia, ib = np.intersect1d(a, b, return_indices=True)
    assert len(ab) == sp.n_overlap and len(np.intersect1d(a, c)) == 0
    assert torch.equal(parts[0]["X"][torch.from_numpy(ia)], parts[1]["X"][torch.from_numpy(ib)])
    assert not torch.equal(parts[0]["graph"]["src"], parts[1]["graph"]["src"])  # own edges per part
