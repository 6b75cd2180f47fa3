"""The bench's per-kernel work models and roofline arithmetic (CPU).

The aggregation models split every layer's work between the row kernels and the hub-chunk kernels
exactly as the library does: forward rows are the CSR rows of each (relation, destination),
backward rows are node-major (a node's out-edges of every relation), parallel edges of a node pair
are one run with their multiplicity, and a row above 512 runs goes through 512-run chunks.  Here
those rows are rebuilt from the oracle's CSR / CSC, and the roofline figures are recomputed by hand
from a fake timing report."""
import numpy as np

import bench
import hgsynth
import oracle


def rows_from_oracle(w):
    g = w.graph
    offs = g["type_offsets"]
    csr = oracle.build_csr(g["src"], g["dst"], g["rel"], offs, g["rels"])
    N = int(offs[-1])
    fwd = []  # (relation, source ids) per forward CSR row, in the row's (source, edge id) order
    node_reads = [[] for _ in range(N)]
    for r, ((ts, tt), c) in enumerate(zip(g["rels"], csr)):
        rp = c["row_ptr"]
        for j in range(len(rp) - 1):
            fwd.append((r, c["col"][rp[j]:rp[j + 1]]))
        cp = c["csc_ptr"]
        for i in range(len(cp) - 1):
            node_reads[int(offs[ts]) + i].extend((r, int(x)) for x in c["csc_col"][cp[i]:cp[i + 1]])
    return fwd, node_reads


def runs(seq) -> list:
    """Distinct entries of a row whose equal entries are adjacent, in order."""
    out = []
    for x in seq:
        if not out or out[-1] != x:
            out.append(x)
    return out


def test_graph_stats_follow_the_kernels_rows():
    sp = hgsynth.spec("sub-1m", n_user=30_000, n_risk=3_000, num_edges=600_000, n_overlap=3_000)
    w = hgsynth.make_workload(sp, with_ids=False)
    st = bench.graph_stats(w)
    fwd, node_reads = rows_from_oracle(w)
    H = bench.HUB
    f_runs = [(r, runs([int(x) for x in row]), len(row)) for r, row in fwd]
    f_hub = [x for x in f_runs if len(x[1]) > H]
    f_small = [x for x in f_runs if len(x[1]) <= H]
    assert f_hub, "the case needs hub rows on both sides"
    assert st["fwd"]["R_h"] == sum(len(u) for _, u, _ in f_hub)
    assert st["fwd"]["R_nh"] == sum(len(u) for _, u, _ in f_small)
    assert st["fwd"]["E_h"] == sum(e for _, _, e in f_hub) and st["fwd"]["E_nh"] == sum(e for _, _, e in f_small)
    assert st["fwd"]["chunks"] == sum(-(-len(u) // bench.CHUNK) for _, u, _ in f_hub)
    # distinct source rows read, counted once per relation (as each relation's pass reads them)
    assert st["fwd"]["U_h"] == len({(r, x) for r, u, _ in f_hub for x in u})
    assert st["fwd"]["U_nh"] == len({(r, x) for r, u, _ in f_small for x in u})
    b_runs = [runs(sorted(reads)) for reads in node_reads]  # node rows: (relation, destination) order
    hub = np.array([len(u) > H for u in b_runs])
    assert hub.any()
    assert st["bwd"]["R_h"] == sum(len(u) for u, h in zip(b_runs, hub) if h)
    assert st["bwd"]["R_nh"] == sum(len(u) for u, h in zip(b_runs, hub) if not h)
    assert st["bwd"]["E_h"] == sum(len(x) for x, h in zip(node_reads, hub) if h)
    assert st["bwd"]["chunks"] == sum(-(-len(u) // bench.CHUNK) for u, h in zip(b_runs, hub) if h)
    assert st["bwd"]["U_h"] == len({x for u, h in zip(b_runs, hub) if h for x in u})
    assert st["bwd"]["U_nh"] == len({x for u, h in zip(b_runs, hub) if not h for x in u})
    assert st["E"] == st["fwd"]["E_h"] + st["fwd"]["E_nh"] == st["bwd"]["E_h"] + st["bwd"]["E_nh"]
    # the fused layer's split: rows of at most FUSE runs are streamed by its kernels, longer rows
    # are summed beforehand (their means stored)
    F = bench.FUSE
    assert any(len(u) > F for _, u, _ in f_small), "the case needs long rows below the hub size"
    assert st["fwd"]["R_short"] == sum(len(u) for _, u, _ in f_runs if len(u) <= F)
    assert st["fwd"]["U_short"] == len({(r, x) for r, u, _ in f_runs if len(u) <= F for x in u})
    assert st["fwd"]["rows_long"] == sum(1 for _, u, _ in f_runs if len(u) > F)
    # runs are far fewer than edges in this recipe (Zipf sources meet Zipf destinations)
    assert st["fwd"]["R_h"] + st["fwd"]["R_nh"] < 0.8 * st["E"]


def test_aggregation_models_are_compulsory_bytes():
    sp = hgsynth.spec("sub-1m", n_user=9_000, n_risk=1_000, num_edges=150_000, n_overlap=800)
    w = hgsynth.make_workload(sp, with_ids=False)
    st = bench.graph_stats(w)
    m = bench.kernel_models(st, sp)
    row, L, f = sp.d * 2, sp.layers, st["fwd"]
    assert m["agg_fwd_chunks"][0] == L * (8 * f["R_h"] + row * f["U_h"] + 4 * sp.d * f["chunks"])
    # the forward rows write only the stored (non-empty) relation rows
    assert 0 < st["NNZ"] < st["RR"]
    assert st["NNZ"] == sum(int(np.count_nonzero(np.bincount(w.graph["dst"][w.graph["rel"] == r], minlength=sp.num_nodes)))
                            for r in range(sp.num_rels))
    assert m["agg_fwd_rows"][0] == L * (12 * st["NNZ"] + 8 * f["R_nh"] + row * f["U_nh"] + row * st["NNZ"] +
                                        4 * sp.d * f["chunks"])
    # the fused layer reads no stored mean for the short rows: the projection's model is the plain
    # one without the stored rows' read, plus run lists, row metadata and source rows of the short
    # rows and the long rows' means; the weight gradient's reads dU and the same gather inputs
    fuse_in = 8 * f["R_short"] + 24 * st["NNZ"] + row * f["U_short"] + row * f["rows_long"]
    assert m["proj_fwd_gather_tc"][0] == m["proj_fwd_tc"][0] - L * row * st["NNZ"] + L * fuse_in
    assert m["proj_fwd_gather_tc"][1] == m["proj_fwd_tc"][1]
    assert m["wgrad_gather_tc"][0] == L * ((row + 4) * st["NNZ"] + fuse_in)
    assert m["gathered"]["proj_fwd_gather_tc"] == L * f["R_short"] * (8 + row)
    # one gathered row and run entry per run, over both kernels of a direction
    runs_f = st["fwd"]["R_h"] + st["fwd"]["R_nh"]
    assert m["gathered"]["agg_fwd_rows"] + m["gathered"]["agg_fwd_chunks"] == L * runs_f * (8 + row)
    # radix sort: 8-bit passes over the source keys (node ids), the CSR row keys and the CSC row
    # keys, 24 bytes moved per edge and pass
    p = lambda n: (len(bin(n)) - 2 + 7) // 8  # noqa: E731
    assert m["radix_scatter"][0] == 24 * sp.num_edges * (p(st["N"]) + p(st["RR"]) + p(st["CC"]))
    # the benchmarked 10M-node graph: 24-bit node ids, 38M rows per layout (26-bit keys): 3 + 4 + 4 passes
    big = bench.kernel_models(dict(st, N=10_000_000, RR=38_000_000, CC=38_000_000, E=200_000_000),
                              hgsynth.spec("big-10m"))
    assert big["radix_scatter"][0] == 24 * 200_000_000 * 11


def test_roofline_arithmetic():
    peaks = {"hbm_gbs": 6000.0, "sm_max_mhz": 2000.0}
    # kernel: 10 launches taking 2 ms in total over 5 steps, 1.2e9 model bytes per step
    report = {"k_hbm": (10, 2.0), "k_simt": (4, 1.0)}
    models = {"k_hbm": (1.2e9, 0), "k_simt": (1e6, 4e10), "gathered": {"k_hbm": 3.6e9}}
    rf, shares = bench.roofline(report, models, 5, peaks, "test")
    assert rf["kernel"] == "k_hbm" and rf["bound"] == "hbm"
    achieved = 1.2e9 * 5 / 2e-3 / 1e9  # GB/s
    assert abs(rf["achieved"] - achieved) < 0.1
    assert abs(rf["frac"] - achieved / 6000.0) < 1e-4
    assert abs(rf["frac_of_nominal"] - achieved / bench.NOMINAL_HBM_GBS) < 1e-4
    assert rf["algorithmic_bytes_per_launch"] == int(1.2e9 * 5 / 10)
    assert rf["gathered_bytes_per_launch"] == int(3.6e9 * 5 / 10)
    assert abs(rf["gathered_gbs"] - 3.6e9 * 5 / 2e-3 / 1e9) < 0.1
    assert "compulsory" in rf["model"]
    assert abs(sum(shares.values()) - 1.0) < 1e-3 and shares["k_hbm"] > shares["k_simt"]
    rs, _ = bench.roofline(report, models, 5, peaks, "test", dom="k_simt")
    assert rs["bound"] == "alu" and rs["unit"] == "TFLOP/s"
    assert abs(rs["peak"] - 152 * 128 * 2 * 2000e6 / 1e12) < 0.1
    assert abs(rs["achieved"] - 4e10 * 5 / 1e-3 / 1e12) < 1e-3


def test_ncu_traffic_folding(tmp_path):
    """ncu's per-launch CSV folds into bytes per launch per kernel function, stamped with the source
    hash that measured_traffic checks."""
    head = ('"ID","Process ID","Process Name","Host Name","Kernel Name","Context","Stream","Block Size","Grid Size",'
            '"Device","CC","Section Name","Metric Name","Metric Unit","Metric Value"\n')
    rows = []
    for i, (read, write) in enumerate([(100, 50), (300, 150)]):
        k = f'"{i}","1","py","h","void hg::agg_chunks<__nv_bfloat16, 128>(const int *, int *)","1","7","(256, 1, 1)","(1, 1, 1)","0","10.3","m"'
        rows += [k + f',"dram__bytes_read.sum","byte","{read}"\n', k + f',"dram__bytes_write.sum","Kbyte","{write / 1000}"\n',
                 k + ',"gpu__time_duration.sum","usecond","2.5"\n']
    k = '"2","1","py","h","edge_keys(const int *, const int *)","1","7","(256, 1, 1)","(1, 1, 1)","0","10.3","m"'
    rows += [k + ',"dram__bytes_read.sum","Mbyte","1.5"\n', k + ',"dram__bytes_write.sum","byte","500"\n']
    csv_path = tmp_path / "t.csv"
    csv_path.write_text("==PROF== noise\n" + head + "".join(rows))
    out = bench.fold_ncu_traffic(str(csv_path), str(tmp_path / "traffic.json"))
    assert out["agg_chunks"]["launches"] == 2 and out["agg_chunks"]["bytes_per_launch"] == 300
    assert out["agg_chunks"]["ns_per_launch"] == 2500 and out["agg_chunks"]["source"] == "agg.cu"
    assert out["edge_keys"]["bytes_per_launch"] == 1_500_500 and out["edge_keys"]["source"] == "graph.cu"
    assert out["agg_chunks"]["sha256"] == bench._source_hash("agg.cu")
