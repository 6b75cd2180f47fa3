"""The bench's per-kernel work models and roofline arithmetic (CPU).

The aggregation models split every layer's edges between the row kernels and the hub-chunk
kernels exactly as the library does: forward rows are the CSR rows of each (relation, destination),
backward rows are node-major (a node's out-edges of every relation), and a row above 512 edges goes
through 512-edge chunks.  Here those rows are rebuilt from the oracle's CSR / CSC, and the roofline
figures are recomputed by hand from a fake timing report."""
import numpy as np

import bench
import hgsynth
import oracle


def rows_from_oracle(w):
    g = w.graph
    offs = g["type_offsets"]
    csr = oracle.build_csr(g["src"], g["dst"], g["rel"], offs, g["rels"])
    N = int(offs[-1])
    fwd = []  # (relation, source ids) per forward CSR row
    node_len = np.zeros(N, np.int64)
    node_reads = [[] for _ in range(N)]
    for r, ((ts, tt), c) in enumerate(zip(g["rels"], csr)):
        rp = c["row_ptr"]
        for j in range(len(rp) - 1):
            fwd.append((r, c["col"][rp[j]:rp[j + 1]]))
        cp = c["csc_ptr"]
        for i in range(len(cp) - 1):
            node = int(offs[ts]) + i
            node_len[node] += cp[i + 1] - cp[i]
            node_reads[node].extend((r, int(x)) for x in c["csc_col"][cp[i]:cp[i + 1]])
    return fwd, node_len, node_reads


def test_graph_stats_follow_the_kernels_rows():
    sp = hgsynth.spec("tiny-10k", n_user=3_000, n_risk=500, num_edges=60_000, n_overlap=300)
    w = hgsynth.make_workload(sp, with_ids=False)
    st = bench.graph_stats(w)
    fwd, node_len, node_reads = rows_from_oracle(w)
    H = bench.HUB
    f_hub = [(r, row) for r, row in fwd if len(row) > H]
    f_small = [(r, row) for r, row in fwd if len(row) <= H]
    assert f_hub, "the case needs hub rows on both sides"
    assert st["fwd"]["E_h"] == sum(len(row) for _, row in f_hub)
    assert st["fwd"]["E_nh"] == sum(len(row) for _, row in f_small)
    assert st["fwd"]["chunks"] == sum(-(-len(row) // bench.CHUNK) for _, row in f_hub)
    # distinct source rows read, counted once per relation (as each relation's pass reads them)
    assert st["fwd"]["U_h"] == len({(r, int(x)) for r, row in f_hub for x in row})
    assert st["fwd"]["U_nh"] == len({(r, int(x)) for r, row in f_small for x in row})
    hub_nodes = node_len > H
    assert hub_nodes.any()
    assert st["bwd"]["E_h"] == int(node_len[hub_nodes].sum())
    assert st["bwd"]["E_nh"] == int(node_len[~hub_nodes].sum())
    assert st["bwd"]["chunks"] == int(sum(-(-n // bench.CHUNK) for n in node_len[hub_nodes]))
    assert st["bwd"]["U_h"] == len({x for i in np.flatnonzero(hub_nodes) for x in node_reads[i]})
    assert st["bwd"]["U_nh"] == len({x for i in np.flatnonzero(~hub_nodes) for x in node_reads[i]})
    assert st["E"] == st["fwd"]["E_h"] + st["fwd"]["E_nh"] == st["bwd"]["E_h"] + st["bwd"]["E_nh"]


def test_aggregation_models_count_every_gathered_edge_once():
    sp = hgsynth.spec("sub-1m", n_user=9_000, n_risk=1_000, num_edges=150_000, n_overlap=800)
    w = hgsynth.make_workload(sp, with_ids=False)
    st = bench.graph_stats(w)
    m = bench.kernel_models(st, sp)
    per_edge = 4 + sp.d * 2  # the 4-byte index and one bf16 feature row
    assert m["agg_fwd_rows"][0] + m["agg_fwd_chunks"][0] == sp.layers * sp.num_edges * per_edge
    assert m["agg_bwd_nodes"][0] + m["agg_bwd_chunks"][0] == sp.layers * sp.num_edges * per_edge
    for k in ("agg_fwd_rows", "agg_bwd_nodes"):
        assert m["compulsory"][k] > 0
    # radix sort: 8-bit passes over row keys in [0, rows], 24 bytes moved per edge and pass
    p_csr = (len(bin(st["RR"])) - 2 + 7) // 8
    p_csc = (len(bin(st["CC"])) - 2 + 7) // 8
    assert m["radix_scatter"][0] == 24 * sp.num_edges * (p_csr + p_csc)
    # the benchmarked 1M-node graph: 2.9M rows in each layout, 22-bit keys, three passes each
    big = bench.kernel_models(dict(st, RR=2_900_000, CC=2_900_000, E=20_000_000), hgsynth.spec("sub-1m"))
    assert big["radix_scatter"][0] == 24 * 20_000_000 * 6
    # the 10M-node graph: 38M rows per layout, 26-bit keys, four passes each
    big = bench.kernel_models(dict(st, RR=38_000_000, CC=38_000_000, E=200_000_000), hgsynth.spec("big-10m"))
    assert big["radix_scatter"][0] == 24 * 200_000_000 * 8


def test_roofline_arithmetic():
    peaks = {"hbm_gbs": 6000.0, "sm_max_mhz": 2000.0}
    # kernel: 10 launches taking 2 ms in total over 5 steps, 1.2e9 model bytes per step
    report = {"k_hbm": (10, 2.0), "k_simt": (4, 1.0)}
    models = {"k_hbm": (1.2e9, 0), "k_simt": (1e6, 4e10), "compulsory": {"k_hbm": 0.6e9}}
    rf, shares = bench.roofline(report, models, 5, peaks, "test")
    assert rf["kernel"] == "k_hbm" and rf["bound"] == "hbm"
    achieved = 1.2e9 * 5 / 2e-3 / 1e9  # GB/s
    assert abs(rf["achieved"] - achieved) < 0.1
    assert abs(rf["frac"] - achieved / 6000.0) < 1e-4
    assert abs(rf["frac_of_nominal"] - achieved / bench.NOMINAL_HBM_GBS) < 1e-4
    assert rf["algorithmic_bytes_per_launch"] == int(1.2e9 * 5 / 10)
    assert abs(rf["compulsory_frac"] - 0.6e9 * 5 / 2e-3 / 1e9 / 6000.0) < 1e-4
    assert "no cache reuse" in rf["model"]
    assert abs(sum(shares.values()) - 1.0) < 1e-3 and shares["k_hbm"] > shares["k_simt"]
    rs, _ = bench.roofline(report, models, 5, peaks, "test", dom="k_simt")
    assert rs["bound"] == "alu" and rs["unit"] == "TFLOP/s"
    assert abs(rs["peak"] - 152 * 128 * 2 * 2000e6 / 1e12) < 0.1
    assert abs(rs["achieved"] - 4e10 * 5 / 1e-3 / 1e12) < 1e-3
