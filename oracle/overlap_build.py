"""CPU oracle of the overlapping-subgraph construction.  TEST INFRASTRUCTURE ONLY.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg import this module; the
product path never calls it and shares no code with it.  Plain numpy (integer work, no floating point).

What is computed (Section 3.1, Eq. 4-5 and the construction part of Algorithm 1):

* partition ...... random hash partitioning of the node set into K disjoint base partitions
                   (Section 3.1, "Graph Partition"): node v goes to part hash(seed, v) mod K.
* degrees ........ number of incident edges of every node over all relations, both directions.
* h_index ........ the h-index of a node (Section 3.1, Hirsch's index on a graph): the largest h
                   such that at least h of its incident edges lead to a node of degree >= h.
* candidates ..... the expansion candidate set C_k of Eq. 4: nodes outside V_k with an edge into
                   a node of V_k.
* build .......... C'_k = candidates with h-index <= theta; C_{k,M} = M of them (all when fewer);
                   V~_k = V_k united with C_{k,M} (Eq. 5); the induced subgraph G[V~_k] with local
                   ids (ascending global id, so the node types stay contiguous) and its edges in
                   input order.

Readings where the paper is silent or ambiguous (listed again in the design notes):
  hash = the SplitMix64 output function applied to (seed XOR value), as published by its authors
  (a counter-based generator, so both sides implement it from its definition);
  A_vu != 0 in Eq. 4 is an edge v -> u (messages from v reach the partition);
  a node's incident edges count both directions and every relation, multi-edges and self-loops
  included (a self-loop is incident twice); edges with an endpoint outside the node range are
  ignored;
  the paper writes "sample b nodes" and "TopM": the M candidates with the smallest sampling keys
  hash(sample_seed XOR (k << 40) XOR v) (high 32 bits), ties by global id -- a uniform sample
  without replacement in a reproducible order.
"""
from __future__ import annotations

import numpy as np

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)


def splitmix64(x) -> np.ndarray:
    """SplitMix64 output for generator state x (uint64, elementwise): z = x + golden gamma, then
    two xor-shift-multiply steps and a final xor-shift."""
    with np.errstate(over="ignore"):
        z = np.asarray(x, dtype=np.uint64) + _GOLDEN
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
        return z ^ (z >> np.uint64(31))


def partition(num_nodes: int, K: int, seed: int) -> np.ndarray:
    """Base partition of every global node id: splitmix64(seed ^ v) mod K (int32)."""
    v = np.arange(num_nodes, dtype=np.uint64)
    return (splitmix64(np.uint64(seed) ^ v) % np.uint64(K)).astype(np.int32)


def degrees(src, dst, num_nodes: int) -> np.ndarray:
    """Incident edges per node, both directions (a self-loop counts twice)."""
    return (np.bincount(src, minlength=num_nodes) + np.bincount(dst, minlength=num_nodes)).astype(np.int64)


def h_index(src, dst, num_nodes: int) -> np.ndarray:
    """h-index of every node: the largest h such that at least h of its incident edges lead to a
    node of degree >= h.  Written out per node: sort the degrees of the other endpoints in
    descending order and count the positions k (1-based) whose degree is >= k."""
    deg = degrees(src, dst, num_nodes)
    node = np.concatenate([src, dst]).astype(np.int64)
    other = np.concatenate([dst, src]).astype(np.int64)
    od = deg[other]
    order = np.lexsort((-od, node))  # by node, then neighbour degree descending
    node, od = node[order], od[order]
    start = np.searchsorted(node, np.arange(num_nodes))
    rank = np.arange(len(node)) - start[node] + 1  # 1-based position inside the node's list
    h = np.zeros(num_nodes, dtype=np.int64)
    np.add.at(h, node, (od >= rank).astype(np.int64))
    return h


def h_index_loops(src, dst, num_nodes: int) -> np.ndarray:
    """The same definition by plain loops (small inputs only): for each node, try every h."""
    deg = [0] * num_nodes
    nbr = [[] for _ in range(num_nodes)]
    for s, t in zip(src.tolist(), dst.tolist()):
        deg[s] += 1
        deg[t] += 1
        nbr[s].append(t)
        nbr[t].append(s)
    out = []
    for v in range(num_nodes):
        best = 0
        for h in range(1, len(nbr[v]) + 1):
            if sum(1 for w in nbr[v] if deg[w] >= h) >= h:
                best = h
        out.append(best)
    return np.array(out, dtype=np.int64)


def candidates(src, dst, part: np.ndarray, k: int) -> np.ndarray:
    """Eq. 4: ascending global ids of the nodes outside V_k with an edge v -> u, u in V_k."""
    src = np.asarray(src, np.int64)
    dst = np.asarray(dst, np.int64)
    m = (part[dst] == k) & (part[src] != k)
    return np.unique(src[m])


def sample_keys(ids: np.ndarray, k: int, seed: int) -> np.ndarray:
    """Sampling key of candidate v in subgraph k: the high 32 bits of
    splitmix64(seed ^ (k << 40) ^ v)."""
    x = np.uint64(seed) ^ (np.uint64(k) << np.uint64(40)) ^ np.asarray(ids, np.uint64)
    return (splitmix64(x) >> np.uint64(32)).astype(np.uint64)


def build(src, dst, rel, type_offsets, K: int, k: int, theta: int, M: int, part_seed: int,
          sample_seed: int) -> dict:
    """Overlapping subgraph k (Algorithm 1, construction loop body).  Returns the global ids of
    V~_k ascending (gid), the size of the base part (n_base), the selected expansion nodes
    (expanded, ascending), the local type offsets, the induced edges in input order with local
    endpoints (src, dst, rel) and their input edge ids (eid), and the sizes of C_k and C'_k."""
    src = np.asarray(src, np.int64)
    dst = np.asarray(dst, np.int64)
    rel = np.asarray(rel, np.int64)
    N = int(type_offsets[-1])
    ok = (src >= 0) & (src < N) & (dst >= 0) & (dst < N)  # other edges are ignored
    part = partition(N, K, part_seed)
    c_all = candidates(src[ok], dst[ok], part, k)
    h = h_index(src[ok], dst[ok], N)
    cand = c_all[h[c_all] <= theta]  # C'_k
    keys = sample_keys(cand, k, sample_seed)
    order = np.lexsort((cand, keys))  # key ascending, ties by global id
    chosen = np.sort(cand[order[:M]])  # C_{k,M}
    member = part == k
    member[chosen] = True
    gid = np.nonzero(member)[0].astype(np.int64)
    local = np.full(N, -1, dtype=np.int64)
    local[gid] = np.arange(len(gid))
    keep = ok.copy()
    keep[ok] = member[src[ok]] & member[dst[ok]]
    eid = np.nonzero(keep)[0].astype(np.int64)
    offs = np.searchsorted(gid, np.asarray(type_offsets, np.int64))
    return {"gid": gid, "n_base": int((part == k).sum()), "expanded": chosen, "h": h,
            "type_offsets": offs.astype(np.int64), "src": local[src[keep]], "dst": local[dst[keep]],
            "rel": rel[keep], "eid": eid, "num_candidates": int(len(c_all)), "num_filtered": int(len(cand))}
