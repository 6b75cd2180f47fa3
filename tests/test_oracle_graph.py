"""Pins of the oracle's graph layout and overlap intersection (CPU only).

CSR/CSC: brute force with Python sorted() on small random COO lists (multi-edges, self-loops,
invalid edges), plus the invariants that determine the layout uniquely.  Intersection: Python
set intersection.
"""
import numpy as np
import pytest

import oracle
from hgsynth import RELATIONS


def random_coo(seed, n_user=30, n_risk=12, num_rels=5, num_edges=400, bad=20):
    rng = np.random.default_rng(seed)
    rels = RELATIONS[:num_rels]
    offs = np.array([0, n_user, n_user + n_risk], np.int64)
    size = (n_user, n_risk)
    r = rng.integers(0, num_rels, num_edges)
    src = np.array([offs[rels[k][0]] + rng.integers(0, size[rels[k][0]]) for k in r])
    dst = np.array([offs[rels[k][1]] + rng.integers(0, size[rels[k][1]]) for k in r])
    # duplicate some edges (multi-edges) and plant invalid ones
    src[:10] = src[10:20]
    dst[:10] = dst[10:20]
    r[:10] = r[10:20]
    bad_pos = rng.choice(np.arange(20, num_edges), bad, replace=False)
    for k, p in enumerate(bad_pos):
        if k % 4 == 0:
            src[p] = offs[-1] + 3
        elif k % 4 == 1:
            r[p] = num_rels
        elif k % 4 == 2:
            dst[p] = -1
        else:  # wrong endpoint type for the relation
            src[p] = offs[1 - rels[r[p]][0]]
    return src.astype(np.int32), dst.astype(np.int32), r.astype(np.int32), offs, rels


def brute_force_rows(src, dst, rel, offs, rels, by_dst=True):
    n = int(offs[-1])
    out = {}
    for rr, (ts, tt) in enumerate(rels):
        key_t = tt if by_dst else ts
        n_rows = int(offs[key_t + 1] - offs[key_t])
        rows = [[] for _ in range(n_rows)]
        for e in range(len(src)):
            s, t, k = int(src[e]), int(dst[e]), int(rel[e])
            if k != rr or not (0 <= s < n and 0 <= t < n):
                continue
            if not (offs[ts] <= s < offs[ts + 1] and offs[tt] <= t < offs[tt + 1]):
                continue
            key = t if by_dst else s
            other = s if by_dst else t
            rows[key - offs[key_t]].append((e, other))
        out[rr] = [sorted(x, key=lambda eo: (eo[1], eo[0])) for x in rows]  # ascending (other end, edge id)
    return out


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_csr_matches_brute_force(seed):
    src, dst, rel, offs, rels = random_coo(seed)
    csr = oracle.build_csr(src, dst, rel, offs, rels)
    bf = brute_force_rows(src, dst, rel, offs, rels, by_dst=True)
    bc = brute_force_rows(src, dst, rel, offs, rels, by_dst=False)
    for r in range(len(rels)):
        c = csr[r]
        for j, row in enumerate(bf[r]):
            a, b = c["row_ptr"][j], c["row_ptr"][j + 1]
            assert list(c["eid"][a:b]) == [e for e, _ in row]
            assert list(c["col"][a:b]) == [s for _, s in row]
            assert c["deg"][j] == len(row)
        for i, row in enumerate(bc[r]):
            a, b = c["csc_ptr"][i], c["csc_ptr"][i + 1]
            assert list(c["csc_eid"][a:b]) == [e for e, _ in row]
            assert list(c["csc_col"][a:b]) == [t for _, t in row]
            tt = rels[r][1]
            for k, (_, t) in enumerate(row):
                assert c["csc_coef"][a + k] == np.float32(1.0) / np.float32(len(bf[r][t - offs[tt]]))


@pytest.mark.parametrize("seed", [0, 3])
def test_node_order_matches_brute_force(seed):
    # the forward projection's node order: a Python sorted() by (mask, id), the mask built edge by
    # edge from the valid COO entries; tile masks by OR loops over tiles of 8 rows (ragged last tile)
    src, dst, rel, offs, rels = random_coo(seed, n_user=61, n_risk=13, num_edges=300)
    csr = oracle.build_csr(src, dst, rel, offs, rels)
    ok = oracle.valid_edges(src, dst, rel, offs, rels)
    for t in range(len(offs) - 1):
        n = int(offs[t + 1] - offs[t])
        into = [r for r, (_, tt) in enumerate(rels) if tt == t]
        mask = [0] * n
        for e in range(len(src)):
            if ok[e] and rel[e] in into:
                mask[int(dst[e] - offs[t])] |= 1 << into.index(int(rel[e]))
        want = sorted(range(n), key=lambda j: (mask[j], j))
        perm, tmask = oracle.node_order(csr, offs, rels, t, tile_rows=8)
        assert list(perm) == want
        for q in range(len(tmask)):
            m = 0
            for j in want[8 * q:8 * q + 8]:
                m |= mask[j]
            assert tmask[q] == m
        assert len(tmask) == (n + 7) // 8
    # a type without incoming relations (type 1 when the only relation is user -> user) keeps its
    # local order, every mask 0
    perm, tmask = oracle.node_order(csr[:1], offs, [(0, 0)], 1)
    assert list(perm) == list(range(int(offs[2] - offs[1]))) and not tmask.any()


def test_csr_invariants():
    src, dst, rel, offs, rels = random_coo(7, num_edges=2000, bad=50)
    csr = oracle.build_csr(src, dst, rel, offs, rels)
    ok = oracle.valid_edges(src, dst, rel, offs, rels)
    assert ok.sum() == len(src) - 50
    seen = []
    for r, c in enumerate(csr):
        assert np.all(np.diff(c["row_ptr"]) >= 0) and c["row_ptr"][0] == 0
        assert c["row_ptr"][-1] == c["csc_ptr"][-1] == np.sum(ok & (rel == r))
        # every edge sits in the row of its destination, in ascending (source, edge id) order
        rows = np.repeat(np.arange(len(c["deg"])), c["deg"])
        assert np.all(dst[c["eid"]] - offs[rels[r][1]] == rows)
        assert np.all(src[c["eid"]] == c["col"])
        same_row = rows[1:] == rows[:-1]
        ds, de = np.diff(c["col"].astype(np.int64))[same_row], np.diff(c["eid"])[same_row]
        assert np.all((ds > 0) | ((ds == 0) & (de > 0)))
        seen.append(c["eid"])
    seen = np.sort(np.concatenate(seen))
    assert np.array_equal(seen, np.flatnonzero(ok))  # a permutation of the valid edges


def test_intersect_matches_python_sets():
    rng = np.random.default_rng(3)
    for _ in range(5):
        a = np.sort(rng.choice(10_000, 800, replace=False)).astype(np.int64)
        b = np.sort(rng.choice(10_000, 1200, replace=False)).astype(np.int64)
        ia, ib = oracle.overlap_intersect(a, b)
        common = sorted(set(a.tolist()) & set(b.tolist()))
        assert [int(a[i]) for i in ia] == common
        assert [int(b[i]) for i in ib] == common
    ia, ib = oracle.overlap_intersect(np.array([1, 2], np.int64), np.array([3, 4], np.int64))
    assert len(ia) == len(ib) == 0
