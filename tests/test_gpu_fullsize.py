"""Full-size bf16 workloads (1M nodes / 20M edges, the benchmark's; 5M nodes / 100M edges at d=256
with a 2M out-degree cap; 10M nodes / 200M edges with 500k-edge hubs), in the launch configuration
the benchmark times: the CSR layout is checked by the invariants that determine it uniquely, the
layer on sampled rows the oracle computes one by one, and the weight gradients exactly by giving
the upstream gradient a sampled support (only those rows contribute)."""
import numpy as np
import pytest
import torch

import hgsynth
import oracle
from tests.gpu_util import BF16_RELU_MARGIN, TOL, dev, grad_bufs, host, layer_params, lib, need_gpu, relerr, tdtype

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", params=["sub-1m", "tail-5m", "big-10m"])
def full(request):
    need_gpu()
    hg = lib()
    sp = hgsynth.spec(request.param)
    # wide bias margins keep the ReLU decisions unambiguous (see test_gpu_layer); every value check
    # below is against the plain fp64 definition
    w = hgsynth.make_workload(sp, random_affine=True, with_ids=True, bias_margin=BF16_RELU_MARGIN)
    g = w.graph
    G = hg.hg_build_csr(dev(g["src"]), dev(g["dst"]), dev(g["rel"]), g["type_offsets"], g["rels"])
    assert hg.hg_graph_check(G) == 0
    return hg, sp, w, G


def test_full_csr_invariants(full):
    hg, sp, w, G = full
    g = w.graph
    src, dst, rel = g["src"].astype(np.int64), g["dst"].astype(np.int64), g["rel"]
    offs = g["type_offsets"]
    seen = np.zeros(len(src), bool)
    for r, (ts, tt) in enumerate(g["rels"]):
        v = hg.hg_graph_view(G, r)
        rp = v["row_ptr"].cpu().numpy().astype(np.int64)
        a, b = rp[0], rp[-1]
        eid = v["eid"][a:b].cpu().numpy().astype(np.int64)
        col = v["col"][a:b].cpu().numpy()
        deg = np.diff(rp)
        rows = np.repeat(np.arange(len(deg)), deg)
        assert np.all(deg >= 0) and b - a == int((rel == r).sum())
        assert np.all(rel[eid] == r) and np.all(dst[eid] - offs[tt] == rows) and np.array_equal(src[eid], col)
        same = rows[1:] == rows[:-1]
        ds, de = np.diff(col.astype(np.int64))[same], np.diff(eid)[same]
        assert np.all((ds > 0) | ((ds == 0) & (de > 0)))  # ascending (source, edge id) within a row
        assert not seen[eid].any()
        seen[eid] = True
        cp = v["csc_ptr"].cpu().numpy().astype(np.int64)
        ca, cb = cp[0], cp[-1]
        ceid = v["csc_eid"][ca:cb].cpu().numpy().astype(np.int64)
        crow = np.repeat(np.arange(len(cp) - 1), np.diff(cp))
        assert np.all(src[ceid] - offs[ts] == crow) and np.all(rel[ceid] == r)
        ccol = v["csc_col"][ca:cb].cpu().numpy().astype(np.int64)
        same = crow[1:] == crow[:-1]
        ds, de = np.diff(ccol)[same], np.diff(ceid)[same]
        assert np.all((ds > 0) | ((ds == 0) & (de > 0)))  # ascending (destination, edge id)
        coef = v["csc_coef"][ca:cb].cpu().numpy()
        want = np.float32(1) / deg[dst[ceid] - offs[tt]].astype(np.float32)
        assert np.array_equal(coef.view(np.uint32), want.view(np.uint32))
    assert seen.all()
    # the forward projection's node order, bit-exact against its definition on in-degrees counted
    # from the COO list
    degs = [dict(deg=np.bincount(dst[rel == r] - offs[tt], minlength=int(offs[tt + 1] - offs[tt])))
            for r, (_, tt) in enumerate(g["rels"])]
    for t in range(len(offs) - 1):
        o = hg.hg_graph_node_order(G, t)
        perm, tmask = oracle.node_order(degs, offs, g["rels"], t, tile_rows=o["tile_rows"])
        assert np.array_equal(o["perm"].cpu().numpy(), perm), f"perm t{t}"
        assert np.array_equal(o["tile_mask"].cpu().numpy(), tmask), f"tile_mask t{t}"


def sample_rows(w, k, seed):
    """Random rows of both types plus the largest in-degree hubs and some rows with no in-edges."""
    g = w.graph
    n = int(g["type_offsets"][-1])
    rng = np.random.default_rng(seed)
    indeg = np.bincount(g["dst"], minlength=n)
    hubs = np.argsort(-indeg, kind="stable")[:8]
    isolated = np.flatnonzero(indeg == 0)[:8]
    risk = int(g["type_offsets"][1]) + rng.choice(n - int(g["type_offsets"][1]), k // 4, replace=False)
    return np.unique(np.concatenate([rng.choice(n, k, replace=False), hubs, isolated, risk]))


def test_full_layer_sampled_rows(full):
    hg, sp, w, G = full
    g = w.graph
    td = tdtype(sp.dtype)
    p = w.params[0]
    P = layer_params(hg, p, sp.dtype)
    sb, kb = hg.hg_layer_workspace_size(G, P)
    saved = torch.empty(sb, dtype=torch.uint8, device="cuda")
    scratch = torch.empty(kb, dtype=torch.uint8, device="cuda")
    X = dev(w.X, td)
    out = torch.empty_like(X)
    hg.hg_layer_fwd(G, P, X, out, saved, scratch)
    rows = sample_rows(w, 3000, 1)
    ref, _ = oracle.layer_forward_rows(g["src"], g["dst"], g["rel"], g["type_offsets"], g["rels"], p, w.X, rows)
    assert relerr(host(out[torch.from_numpy(rows).cuda()]), ref) <= TOL[sp.dtype]
    # backward with an upstream gradient supported on a row sample S
    S = sample_rows(w, 2000, 2)
    dH_out = torch.zeros_like(X)
    dH_out[torch.from_numpy(S).cuda()] = dev(w.dH_top[S], td)
    dH_in = torch.empty_like(X)
    grads = grad_bufs(len(g["rels"]), 2, sp.d)
    hg.hg_layer_bwd(G, P, X, saved, dH_out, dH_in, grads, scratch)
    # query rows: S itself, sources of edges into S (they receive the transposed gather) and others
    into_S = np.unique(g["src"][np.isin(g["dst"], S)])
    rng = np.random.default_rng(3)
    q = np.unique(np.concatenate([S[:500], rng.choice(into_S, min(1500, len(into_S)), replace=False),
                                  rng.choice(int(g["type_offsets"][-1]), 500, replace=False)]))
    dq, gref = oracle.layer_backward_rows(g["src"], g["dst"], g["rel"], g["type_offsets"], g["rels"], p, w.X, S,
                                          w.dH_top[S], q)
    tol = TOL[sp.dtype]
    assert relerr(host(dH_in[torch.from_numpy(q).cuda()]), dq) <= tol
    for k, v in gref.items():
        assert relerr(host(grads[k]), v) <= tol, (k, relerr(host(grads[k]), v))


def test_full_fused_layer_equals_plain(full):
    """The fused mean layer (relation means never stored) against the plain layer at full size, bit
    for bit: outputs, input gradients and every weight gradient (the plain layer is checked against
    the definition above)."""
    hg, sp, w, G = full
    if not (sp.dtype == "bf16" and sp.d == 128):
        pytest.skip("the fused layer is built for bf16, d = 128")
    g = w.graph
    X = dev(w.X, torch.bfloat16)
    dH_out = dev(w.dH_top, torch.bfloat16)
    res = []
    for fused in (False, True):
        P = layer_params(hg, w.params[0], "bf16", fused=fused)
        sb, kb = hg.hg_layer_workspace_size(G, P)
        saved = torch.empty(sb, dtype=torch.uint8, device="cuda")
        scratch = torch.empty(kb, dtype=torch.uint8, device="cuda")
        out = torch.empty_like(X)
        hg.hg_layer_fwd(G, P, X, out, saved, scratch)
        dH_in = torch.empty_like(X)
        grads = grad_bufs(len(g["rels"]), 2, sp.d)
        hg.hg_layer_bwd(G, P, X, saved, dH_out, dH_in, grads, scratch)
        torch.cuda.synchronize()
        res.append((out, dH_in, grads, sb))
        del saved, scratch
    (o0, d0, g0, s0), (o1, d1, g1, s1) = res
    assert s1 < s0
    assert torch.equal(o0.view(torch.int16), o1.view(torch.int16)), "H_out"
    assert torch.equal(d0.view(torch.int16), d1.view(torch.int16)), "dH_in"
    for k in g0:
        assert torch.equal(g0[k], g1[k]), k
    assert hg.hg_device_status() == 0


def test_full_overlap_and_alignment(full):
    hg, sp, w, G = full
    td = tdtype(sp.dtype)
    n_a, n_b = len(w.gid_a), len(w.gid_b)
    cap = min(n_a, n_b)
    idx_a = torch.empty(cap, dtype=torch.int32, device="cuda")
    idx_b = torch.empty(cap, dtype=torch.int32, device="cuda")
    n_dev = torch.zeros(1, dtype=torch.int64, device="cuda")
    scr = torch.empty(hg.hg_overlap_intersect_workspace_size(n_a, n_b), dtype=torch.uint8, device="cuda")
    hg.hg_overlap_intersect(dev(w.gid_a), dev(w.gid_b), idx_a, idx_b, n_dev, scr)
    ia, ib = oracle.overlap_intersect(w.gid_a, w.gid_b)
    n = int(n_dev.item())
    assert n == len(ia) == sp.n_overlap
    assert np.array_equal(idx_a[:n].cpu().numpy(), ia) and np.array_equal(idx_b[:n].cpu().numpy(), ib)
    if sp.overlap == "longtail":
        # the overlap rows are long-tail nodes (total degree <= 2, hence h-index <= 2)
        deg = np.bincount(w.graph["src"], minlength=sp.num_nodes) + np.bincount(w.graph["dst"], minlength=sp.num_nodes)
        assert deg[ia].max() <= 2
    s, k = hg.hg_overlap_align_workspace_size(cap, sp.d)
    saved = torch.empty(s, dtype=torch.uint8, device="cuda")
    scratch = torch.empty(k, dtype=torch.uint8, device="cuda")
    loss = torch.empty(3, dtype=torch.float32, device="cuda")
    A, B = dev(w.X, td), dev(w.H_b, td)
    hg.hg_overlap_align_loss(A, idx_a, B, idx_b, cap, n_dev, 2e-4, 1e-8, loss, saved, scratch)
    dA = torch.zeros_like(A)
    hg.hg_overlap_align_bwd(A, idx_a, B, idx_b, cap, n_dev, 2e-4, 1e-8, 0.1, saved, dA, None, scratch)
    ref = oracle.align_forward(w.X, ia, w.H_b, ib, 2e-4, 1e-8)
    assert relerr(host(loss), np.array(ref)) <= 1e-4
    rA, _ = oracle.align_backward(w.X, ia, w.H_b, ib, 2e-4, 1e-8, 0.1)
    assert relerr(host(dA)[ia], rA[ia]) <= TOL[sp.dtype]


def test_full_size_overlap_construction():
    """The 1M-node / 20M-edge graph as the global graph of the subgraph construction, K = 8,
    theta = 2 and a 15 % budget (the paper's setting): every output bit-exact against the oracle."""
    need_gpu()
    from tests.test_gpu_overlap_build import compare, run
    g = hgsynth.make_graph(hgsynth.spec("sub-1m"))
    offs = [int(x) for x in g["type_offsets"]]
    M = int(0.15 * offs[-1] / 8)
    out, ref = run(lib(), g["src"], g["dst"], g["rel"], offs, 8, 3, 2, M, ps=21, ss=22)
    compare(out, ref)
    assert out["counts"]["expanded"] == min(M, out["counts"]["filtered"]) > 0


def test_full_size_head():
    """The head on the 1M-node bf16 d=128 workload: 11.7 % of the 900k users labelled, 130,435
    overlap rows averaged with a bank view; every output against the oracle."""
    need_gpu()
    from tests.test_gpu_head import check, head_gpu
    sp = hgsynth.spec("sub-1m")
    lab, y = hgsynth.make_labels(sp)
    p = hgsynth.make_head_params(sp, random_bias=True, bias_margin=BF16_RELU_MARGIN)  # see test_gpu_head
    rng = np.random.default_rng(5)
    N, d = sp.num_nodes, sp.d
    H = hgsynth.bf16_round(rng.standard_normal((N, d), dtype=np.float32))
    Hr = hgsynth.bf16_round(rng.standard_normal((N, d), dtype=np.float32))
    ia = np.sort(rng.choice(N, sp.n_overlap, replace=False)).astype(np.int32)
    ib = np.sort(rng.choice(N, sp.n_overlap, replace=False)).astype(np.int32)
    got = head_gpu(lib(), H, Hr, ia, ib, lab, y, p, "bf16", cca=3.0, lam=0.1)
    check(got, H, Hr, ia, ib, lab, y, p, "bf16", cca=3.0, lam=0.1)


def test_full_size_temporal():
    """The temporal module over the 1M nodes of the benchmark workload (w = 3, bf16 d = 128, the
    tensor-core path): every output row the oracle computes on 3,000 sampled nodes (the module is
    row by row), and the weight gradients exactly for an upstream gradient supported on those
    nodes (the other rows then contribute nothing)."""
    need_gpu()
    from oracle import temporal as OT
    hg = lib()
    sp = hgsynth.spec("sub-1m")
    n, d, w = sp.num_nodes, sp.d, hgsynth.TEMPORAL_WINDOW
    rng = np.random.default_rng(31)
    X = hgsynth.bf16_round(rng.standard_normal((n, d), dtype=np.float32))
    C = hgsynth.make_context(sp)
    p = hgsynth.make_temporal_params(sp)
    rows = np.unique(np.concatenate([rng.choice(n, 3000, replace=False), [0, n - 1]]))
    dOut = np.zeros((n, d), np.float32)
    dOut[rows] = hgsynth.bf16_round(rng.standard_normal((len(rows), d), dtype=np.float32))
    td = torch.bfloat16
    keys = ("Wa", "r", "W_i", "W_h", "b_i", "b_h")
    prm = hg.TemporalParams(*(dev(p[k], td) for k in keys), w=w)
    sb, kb = hg.hg_temporal_workspace_size(n, d, w, td)
    saved = torch.empty(sb, dtype=torch.uint8, device="cuda")
    scratch = torch.empty(kb, dtype=torch.uint8, device="cuda")
    Xd, Cd = dev(X, td), dev(C, td)
    out = torch.empty(n, d, dtype=td, device="cuda")
    hg.hg_temporal_fwd(prm, Xd, Cd, out, saved, scratch)
    f = dict(dtype=torch.float32, device="cuda")
    grads = {"Wa": torch.empty(d, d, **f), "r": torch.empty(d, **f), "W_i": torch.empty(d, 3 * d, **f),
             "W_h": torch.empty(d, 3 * d, **f), "b_i": torch.empty(3 * d, **f), "b_h": torch.empty(3 * d, **f)}
    dX = torch.empty_like(out)
    hg.hg_temporal_bwd(prm, Xd, Cd, saved, dev(dOut, td), dX, grads, scratch)
    torch.cuda.synchronize()
    ref = OT.temporal_backward(X[rows], C[:, rows], p, dOut[rows])
    tol = TOL["bf16"]
    assert relerr(host(out)[rows], ref["out"]) <= tol
    assert relerr(host(dX)[rows], ref["dX"]) <= tol
    for k in keys:
        assert relerr(host(grads[k]), ref["d" + k]) <= tol, k
    assert hg.hg_device_status() == 0


def test_full_size_attention_layer_sampled_targets():
    """The attention layer (4 heads) on the benchmark graph (1M nodes, 20M edges, hubs of ~1M
    in-edges): the output rows of sampled targets -- random rows, the largest in-degree hubs and
    rows without in-edges -- against the oracle run on the subgraph of their in-edges (a row's
    output depends only on its own features and those of its in-neighbours)."""
    need_gpu()
    from oracle import hgt as OH
    hg = lib()
    sp = hgsynth.spec("sub-1m")
    w = hgsynth.make_workload(sp, with_ids=False)
    g = w.graph
    p = hgsynth.make_hgt_params(sp, 4, bias_margin=BF16_RELU_MARGIN)
    td = torch.bfloat16
    G = hg.hg_build_csr(dev(g["src"]), dev(g["dst"]), dev(g["rel"]), g["type_offsets"], g["rels"])
    P = hg.HgtParams({k: dev(v, torch.float32 if k == "mu" else td) for k, v in p.items()}, 4)
    sb, kb = hg.hg_hgt_workspace_size(G, P)
    saved = torch.empty(sb, dtype=torch.uint8, device="cuda")
    scratch = torch.empty(kb, dtype=torch.uint8, device="cuda")
    X = dev(w.X, td)
    out = torch.empty_like(X)
    hg.hg_hgt_fwd(G, P, X, out, saved, scratch)
    torch.cuda.synchronize()
    rows = sample_rows(w, 400, 33)
    keep = np.isin(g["dst"], rows)
    nodes = np.unique(np.concatenate([rows, g["src"][keep]]))
    # the subgraph keeps global ids (rows outside it have no in-edges and are not compared)
    ref, _ = OH.hgt_forward(g["src"][keep], g["dst"][keep], g["rel"][keep], g["type_offsets"], g["rels"], p,
                            np.where(np.isin(np.arange(sp.num_nodes), nodes)[:, None], w.X, 0.0), 4)
    assert relerr(host(out)[rows], ref[rows]) <= TOL["bf16"]
    assert hg.hg_device_status() == 0
