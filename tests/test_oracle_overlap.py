"""Pins of the overlapping-subgraph construction oracle (Section 3.1, Eq. 4-5, Algorithm 1)."""
import numpy as np
import pytest

from oracle import overlap_build as ob


def test_splitmix64_published_check_values():
    # the first three outputs of the SplitMix64 generator started from state 0
    x = np.array([0, 0x9E3779B97F4A7C15, 2 * 0x9E3779B97F4A7C15 % 2**64], dtype=np.uint64)
    got = [int(v) for v in ob.splitmix64(x)]
    assert got == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def _random_graph(seed, n, e, self_loops=True):
    rng = np.random.default_rng(seed)
    src = rng.integers(0, n, e)
    dst = rng.integers(0, n, e)
    if not self_loops:
        dst = np.where(dst == src, (dst + 1) % n, dst)
    rel = rng.integers(0, 3, e)
    return src.astype(np.int64), dst.astype(np.int64), rel.astype(np.int64)


@pytest.mark.parametrize("seed", range(4))
def test_h_index_matches_definition_by_loops(seed):
    src, dst, _ = _random_graph(seed, 60, 300)
    np.testing.assert_array_equal(ob.h_index(src, dst, 60), ob.h_index_loops(src, dst, 60))


def test_h_index_closed_forms():
    # star: the centre and every leaf have h-index 1
    n = 9
    src = np.zeros(n, np.int64)
    dst = np.arange(1, n + 1, dtype=np.int64)
    h = ob.h_index(src, dst, n + 1)
    assert h[0] == 1 and np.all(h[1:] == 1)
    # clique K_5 (one edge per pair): degree 4 everywhere, h-index 4
    i, j = np.triu_indices(5, 1)
    assert np.all(ob.h_index(i.astype(np.int64), j.astype(np.int64), 5) == 4)
    # isolated node: 0; a self-loop alone: degree 2, two incident entries of degree 2 -> h = 2
    h = ob.h_index(np.array([1], np.int64), np.array([1], np.int64), 3)
    assert list(h) == [0, 2, 0]
    # path 0-1-2-3-4: only the middle node has two neighbours of degree >= 2
    assert list(ob.h_index(np.array([0, 1, 2, 3]), np.array([1, 2, 3, 4]), 5)) == [1, 1, 2, 1, 1]


def test_candidates_by_brute_force():
    src, dst, _ = _random_graph(7, 80, 400)
    part = ob.partition(80, 4, 11)
    for k in range(4):
        want = sorted({int(s) for s, t in zip(src, dst) if part[t] == k and part[s] != k})
        assert list(ob.candidates(src, dst, part, k)) == want


def test_partition_is_a_partition_and_balanced():
    p = ob.partition(100_000, 8, 3)
    assert p.min() == 0 and p.max() == 7
    counts = np.bincount(p, minlength=8)
    assert np.all(np.abs(counts - 12_500) < 5 * np.sqrt(12_500))
    assert not np.array_equal(p, ob.partition(100_000, 8, 4))  # the seed matters


@pytest.mark.parametrize("K,k,theta,M", [(4, 0, 2, 10), (4, 3, 1, 1000), (3, 1, 5, 0), (1, 0, 2, 50), (6, 2, 0, 7)])
def test_build_invariants_and_brute_force(K, k, theta, M):
    n_user, n_risk = 90, 30
    N = n_user + n_risk
    src, dst, rel = _random_graph(K * 10 + k, N, 500)
    offs = np.array([0, n_user, N], np.int64)
    out = ob.build(src, dst, rel, offs, K, k, theta, M, part_seed=5, sample_seed=9)
    part = ob.partition(N, K, 5)
    h = ob.h_index_loops(src, dst, N)
    base = {v for v in range(N) if part[v] == k}
    cand = {int(s) for s, t in zip(src, dst) if part[t] == k and part[s] != k}
    filt = sorted(v for v in cand if h[v] <= theta)
    keys = ob.sample_keys(np.array(filt, np.int64), k, 9)
    chosen = sorted(v for _, v in sorted(zip([int(x) for x in keys], filt))[:M])
    assert out["num_candidates"] == len(cand) and out["num_filtered"] == len(filt)
    assert list(out["expanded"]) == chosen
    assert len(chosen) == min(M, len(filt)) and not (set(chosen) & base)
    members = sorted(base | set(chosen))
    assert list(out["gid"]) == members and out["n_base"] == len(base)
    # local ids keep the global order, so the type ranges stay contiguous
    gid = out["gid"]
    assert list(out["type_offsets"]) == [0, sum(1 for v in members if v < n_user), len(members)]
    # induced edges, in input order
    ms = set(members)
    want = [(e, s, t, r) for e, (s, t, r) in enumerate(zip(src, dst, rel)) if s in ms and t in ms]
    assert list(out["eid"]) == [w[0] for w in want]
    assert list(gid[out["src"]]) == [w[1] for w in want]
    assert list(gid[out["dst"]]) == [w[2] for w in want]
    assert list(out["rel"]) == [w[3] for w in want]
    if K == 1:
        assert out["num_candidates"] == 0 and len(gid) == N


def test_overlap_between_subgraphs_exists():
    n = 2000
    src, dst, rel = _random_graph(3, n, 8000, self_loops=False)
    offs = np.array([0, 1500, n], np.int64)
    a = ob.build(src, dst, rel, offs, 4, 0, 50, 200, 1, 2)
    b = ob.build(src, dst, rel, offs, 4, 1, 50, 200, 1, 2)
    shared = np.intersect1d(a["gid"], b["gid"])
    assert len(shared) > 0  # Eq. 5: the expanded sets create overlaps between subgraphs


def test_out_of_range_edges_are_ignored():
    src, dst, rel = _random_graph(21, 50, 200)
    offs = np.array([0, 40, 50], np.int64)
    clean = ob.build(src, dst, rel, offs, 3, 1, 3, 20, 1, 2)
    bad_src = np.concatenate([src, [-1, 7, 60]])
    bad_dst = np.concatenate([dst, [3, 99, 2]])
    bad_rel = np.concatenate([rel, [0, 1, 2]])
    dirty = ob.build(bad_src, bad_dst, bad_rel, offs, 3, 1, 3, 20, 1, 2)
    for key in ("gid", "expanded", "src", "dst", "rel", "eid", "h"):
        np.testing.assert_array_equal(clean[key], dirty[key])
