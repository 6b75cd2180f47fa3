"""CSR / CSC construction on the GPU, bit-exact against the oracle (plus dropped-edge counts,
degenerate graphs and hub rows that span many chunks)."""
import numpy as np
import pytest
import torch

import hgsynth
import oracle
from tests.gpu_util import dev, lib, need_gpu
from tests.test_oracle_graph import random_coo

pytestmark = pytest.mark.gpu


def gpu_csr(hg, src, dst, rel, offs, rels):
    G = hg.hg_build_csr(dev(src, torch.int32), dev(dst, torch.int32), dev(rel, torch.int32), offs, rels)
    bad = hg.hg_graph_check(G)
    return G, bad


def compare_node_order(hg, G, ref, offs, rels):
    for t in range(len(offs) - 1):
        o = hg.hg_graph_node_order(G, t)
        perm, tmask = oracle.node_order(ref, offs, rels, t, tile_rows=o["tile_rows"])
        assert o["n"] == len(perm) and o["tiles"] == len(tmask)
        assert np.array_equal(o["perm"].cpu().numpy(), perm), f"perm t{t}"
        assert np.array_equal(o["tile_mask"].cpu().numpy(), tmask), f"tile_mask t{t}"


def compare_layout(hg, G, ref, rels):
    for r in range(len(rels)):
        v = hg.hg_graph_view(G, r)
        c = ref[r]
        rp = v["row_ptr"].cpu().numpy().astype(np.int64)
        a, b = rp[0], rp[-1]
        assert np.array_equal(rp - a, c["row_ptr"]), f"row_ptr r{r}"
        assert np.array_equal(v["col"][a:b].cpu().numpy(), c["col"]), f"col r{r}"
        assert np.array_equal(v["eid"][a:b].cpu().numpy(), c["eid"]), f"eid r{r}"
        cp = v["csc_ptr"].cpu().numpy().astype(np.int64)
        a, b = cp[0], cp[-1]
        assert np.array_equal(cp - a, c["csc_ptr"]), f"csc_ptr r{r}"
        assert np.array_equal(v["csc_col"][a:b].cpu().numpy(), c["csc_col"]), f"csc_col r{r}"
        assert np.array_equal(v["csc_eid"][a:b].cpu().numpy(), c["csc_eid"]), f"csc_eid r{r}"
        coef = v["csc_coef"][a:b].cpu().numpy()
        assert np.array_equal(coef.view(np.uint32), c["csc_coef"].view(np.uint32)), f"csc_coef r{r}"


@pytest.mark.parametrize("seed", [0, 1])
def test_random_coo_with_invalid_edges(seed):
    need_gpu()
    hg = lib()
    src, dst, rel, offs, rels = random_coo(seed, n_user=300, n_risk=70, num_edges=20_000, bad=300)
    G, bad = gpu_csr(hg, src, dst, rel, offs, rels)
    assert bad == int((~oracle.valid_edges(src, dst, rel, offs, rels)).sum()) == 300
    ref = oracle.build_csr(src, dst, rel, offs, rels)
    compare_layout(hg, G, ref, rels)
    compare_node_order(hg, G, ref, offs, rels)


def test_tiny_workload_graph():
    need_gpu()
    hg = lib()
    g = hgsynth.make_graph(hgsynth.spec("tiny-10k"))
    G, bad = gpu_csr(hg, g["src"], g["dst"], g["rel"], g["type_offsets"], g["rels"])
    assert bad == 0
    ref = oracle.build_csr(g["src"], g["dst"], g["rel"], g["type_offsets"], g["rels"])
    compare_layout(hg, G, ref, g["rels"])
    compare_node_order(hg, G, ref, g["type_offsets"], g["rels"])


def test_hub_rows_and_degenerate_graphs():
    need_gpu()
    hg = lib()
    rels = ((0, 0), (0, 1), (1, 0))
    offs = np.array([0, 3000, 3010], np.int64)
    rng = np.random.default_rng(5)
    # one destination with 5000 in-edges and one source with 7000 out-edges, plus noise
    src = np.concatenate([rng.integers(0, 3000, 5000), np.full(7000, 17), rng.integers(0, 3000, 2000)])
    dst = np.concatenate([np.full(5000, 42), 3000 + rng.integers(0, 10, 7000), rng.integers(0, 3000, 2000)])
    rel = np.concatenate([np.zeros(5000), np.ones(7000), np.zeros(2000)]).astype(np.int64)
    perm = rng.permutation(len(src))
    src, dst, rel = src[perm], dst[perm], rel[perm]
    G, bad = gpu_csr(hg, src, dst, rel, offs, rels)
    assert bad == 0
    ref = oracle.build_csr(src, dst, rel, offs, rels)
    compare_layout(hg, G, ref, rels)
    compare_node_order(hg, G, ref, offs, rels)
    # no edges at all
    e = np.zeros(0, np.int64)
    G, bad = gpu_csr(hg, e, e, e, offs, rels)
    assert bad == 0
    ref = oracle.build_csr(e, e, e, offs, rels)
    compare_layout(hg, G, ref, rels)
    compare_node_order(hg, G, ref, offs, rels)
    # every edge invalid
    G, bad = gpu_csr(hg, np.full(10, 5000), np.zeros(10, np.int64), np.zeros(10, np.int64), offs, rels)
    assert bad == 10
    # an empty node type
    offs2 = np.array([0, 50, 50], np.int64)
    s2 = rng.integers(0, 50, 400)
    d2 = rng.integers(0, 50, 400)
    r2 = np.zeros(400, np.int64)
    G, bad = gpu_csr(hg, s2, d2, r2, offs2, rels)
    assert bad == 0
    ref = oracle.build_csr(s2, d2, r2, offs2, rels)
    compare_layout(hg, G, ref, rels)
    compare_node_order(hg, G, ref, offs2, rels)


def test_build_is_repeatable():
    need_gpu()
    hg = lib()
    src, dst, rel, offs, rels = random_coo(3, n_user=2000, n_risk=300, num_edges=200_000, bad=10)
    ref = oracle.build_csr(src, dst, rel, offs, rels)
    for _ in range(2):
        G, bad = gpu_csr(hg, src, dst, rel, offs, rels)
        assert bad == 10
        compare_layout(hg, G, ref, rels)
        compare_node_order(hg, G, ref, offs, rels)


def test_node_order_with_eight_relations_into_one_type():
    # 2^8 relation masks over 50,000 destinations (25 blocks of the counting sort, a ragged last tile):
    # Zipf-like destinations per relation so that every mask value from sparse to dense occurs
    need_gpu()
    hg = lib()
    rels = tuple([(0, 0)] * 4 + [(1, 0)] * 4)
    offs = np.array([0, 50_001, 53_001], np.int64)
    rng = np.random.default_rng(11)
    src, dst, rel = [], [], []
    for r, (ts, _) in enumerate(rels):
        k = 20_000 + 6_000 * r
        d = np.minimum((rng.pareto(0.8 + 0.1 * r, k) * 50).astype(np.int64), 50_000)
        dst.append(d)
        src.append(offs[ts] + rng.integers(0, offs[ts + 1] - offs[ts], k))
        rel.append(np.full(k, r))
    src, dst, rel = np.concatenate(src), np.concatenate(dst), np.concatenate(rel)
    perm = rng.permutation(len(src))
    src, dst, rel = src[perm], dst[perm], rel[perm]
    G, bad = gpu_csr(hg, src, dst, rel, offs, rels)
    assert bad == 0
    ref = oracle.build_csr(src, dst, rel, offs, rels)
    compare_node_order(hg, G, ref, offs, rels)
    mask = sum((ref[r]["deg"] > 0).astype(np.int64) << r for r in range(8))
    assert len(np.unique(mask)) > 200  # nearly every mask value occurs


def test_25_bit_row_keys():
    # three relations into a 6M-node type: 18M CSR rows and 18M CSC rows (25-bit keys, four radix
    # passes each, the last on a 1-bit digit), 23-bit node ids; bit-exact against the oracle on 2M
    # random edges with parallel edges
    need_gpu()
    hg = lib()
    n0 = 6_000_000
    offs = np.array([0, n0, n0 + 100], np.int64)
    rels = ((0, 0), (0, 0), (0, 0))
    rng = np.random.default_rng(21)
    E = 2_000_000
    src = rng.integers(0, n0, E)
    dst = np.minimum((rng.pareto(1.2, E) * 1000).astype(np.int64), n0 - 1)
    rel = rng.integers(0, 3, E)
    src[:50_000] = src[50_000:100_000]
    dst[:50_000] = dst[50_000:100_000]
    rel[:50_000] = rel[50_000:100_000]
    G, bad = gpu_csr(hg, src, dst, rel, offs, rels)
    assert bad == 0
    ref = oracle.build_csr(src, dst, rel, offs, rels)
    compare_layout(hg, G, ref, rels)
    compare_node_order(hg, G, ref, offs, rels)
