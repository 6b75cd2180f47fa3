#!/usr/bin/env python
"""Benchmark of the hot path: GNN layer forward+backward edges/s on one GB300.

One step = one pass of the whole hot path over one overlapping subgraph: the relation-typed CSR /
CSC build, L layers forward, the overlap intersection, the alignment loss, the head's loss and
gradient (joint objective of Eq. 20), the alignment gradient and L layers backward, dL/dX included.
value = L * E * steps * ranks / (max over ranks of the device time of the timed steps).  The
default workload is the largest single-GPU one: 10M nodes, 200M edges (Zipf s = 1.2, top-100 hubs
of >= 500k out-edges), bf16 d = 128, 3 layers.  Inputs are seeded synthetic instances of the
workload recipe drawn on the GPU (hgsynth.device), resident in HBM before timing and larger than
L2, which is not flushed.  Beside the headline the line reports the L-layer stack alone (forward +
backward, the metric's own definition), the CSR build, the other workloads (tiny-10k, sub-1m,
tail-5m) and one full pass over the sixteen-subgraph ring.  Multi-GPU (torchrun): every rank runs
its own subgraph (weak scaling), no collective on the data path.  `--impl reference` times the CPU
oracle on a bounded sample of the same workload.

Prints one JSON line (rank 0).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import hgsynth  # noqa: E402

METRIC = "GNN layer fwd+bwd edges/sec on 1 GB300; achieved HBM GB/s vs roofline"
UNIT = "edges/s"
SAMPLE_EDGES = 150_000   # the CPU oracle runs on instances of about this many edges (same recipe)
BUILD_K, BUILD_THETA, BUILD_BUDGET = 8, 2, 0.15  # overlapping-subgraph construction: parts, h-index bound, M / N
FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "sm_max_mhz": 2070.0}
NOMINAL_HBM_GBS = 7900.0  # GB300 HBM3e data-sheet bandwidth, reported beside the measured copy peak
EXTRA_WORKLOADS = ("tiny-10k", "sub-1m", "tail-5m")
SIDE_WORKLOAD = "sub-1m"  # the construction, temporal module and attention layer are measured here
HGT_HEADS = 4  # attention heads (Section 4.1)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="big-10m", choices=sorted(hgsynth.WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-extra", action="store_true", help="skip the other workloads and the ring pass")
    ap.add_argument("--no-build", action="store_true", help="skip the subgraph-construction measurement")
    ap.add_argument("--no-head", action="store_true",
                    help="drive the layers with a synthetic upstream gradient instead of the head and joint loss")
    ap.add_argument("--no-temporal", action="store_true", help="skip the temporal-module measurement")
    ap.add_argument("--no-hgt", action="store_true", help="skip the attention-layer measurement")
    ap.add_argument("--no-fused", action="store_true", help="skip the fused mean layer's measurement")
    ap.add_argument("--scale", type=int, default=1, help=argparse.SUPPRESS)  # profiling: a 1/k-size instance
    ap.add_argument("--ncu-traffic", default="",
                    help="fold an ncu CSV (--metrics dram__bytes_read.sum,dram__bytes_write.sum,gpu__time_duration.sum "
                         "--csv) into profiles/traffic.json, each kernel stamped with its source hash, and exit")
    ap.add_argument("--oracle-child", default="", help=argparse.SUPPRESS)  # internal: child process kind
    ap.add_argument("--oracle-k", type=int, default=1, help=argparse.SUPPRESS)
    ap.add_argument("--oracle-steps", type=int, default=1, help=argparse.SUPPRESS)
    ap.add_argument("--oracle-warmup", type=int, default=0, help=argparse.SUPPRESS)
    return ap.parse_args()


def scaled(spec, k: int):
    """A 1/k-size instance of the same recipe (nodes, edges, overlap set, hub floor and out-degree
    cap all divided by k)."""
    if k <= 1:
        return spec
    floor = None if spec.hub_floor is None else (spec.hub_floor[0], max(1, spec.hub_floor[1] // k))
    cap = None if spec.out_cap is None else max(1, spec.out_cap // k)
    return hgsynth.spec(spec.name, n_user=max(1, spec.n_user // k), n_risk=max(1, spec.n_risk // k),
                        num_edges=spec.num_edges // k, n_overlap=max(2, spec.n_overlap // k), hub_floor=floor,
                        out_cap=cap)


def sample_scale(sp) -> int:
    return max(1, sp.num_edges // SAMPLE_EDGES)


def workload_desc(sp) -> str:
    return (f"{sp.name}: {sp.num_nodes:,} nodes ({sp.n_user:,} user / {sp.n_risk:,} risk), {sp.num_rels} relations, "
            f"{sp.num_edges:,} edges, Zipf s={sp.zipf_s}, d={sp.d} {sp.dtype}, {sp.layers} layers, "
            f"{sp.n_overlap:,} overlap rows ({sp.overlap}), second view: {sp.view_b}")


# ------------------------------------------------------------------------------------------------
# oracle timing (CPU baseline / reference arm): a child process with the numpy oracle on a 1/k
# instance drawn by hgsynth.graphs, its BLAS allowed every host core
# ------------------------------------------------------------------------------------------------
def oracle_child_main(kind: str, name: str, k: int, steps: int, warmup: int, with_head: bool):
    import oracle
    sp = scaled(hgsynth.spec(name), k)
    times = []
    if kind == "step":
        w = hgsynth.make_workload(sp)
        vb = {"idx": w.overlap_local, "X_b": w.X_b} if sp.view_b == "perturbed" else \
            {"H_b": w.H_b, "gid_a": w.gid_a, "gid_b": w.gid_b}
        head = None
        if with_head:
            lab, y = hgsynth.make_labels(sp)
            head = {"params": hgsynth.make_head_params(sp), "lab_idx": lab, "lab_y": y}
        units = sp.layers * sp.num_edges
        for i in range(warmup + steps):
            t0 = time.perf_counter()
            oracle.step(w.graph, w.X, w.params, w.dH_top, vb, head=head)
            if i >= warmup:
                times.append(time.perf_counter() - t0)
    elif kind == "build":
        from oracle import overlap_build as ob
        g = hgsynth.make_graph(sp)
        offs = np.asarray(g["type_offsets"], np.int64)
        units = sp.num_edges
        for i in range(warmup + steps):
            t0 = time.perf_counter()
            ob.build(g["src"], g["dst"], g["rel"], offs, BUILD_K, 0, BUILD_THETA, int(BUILD_BUDGET * offs[-1] / BUILD_K),
                     21, 22)
            if i >= warmup:
                times.append(time.perf_counter() - t0)
    elif kind == "temporal":
        from oracle import temporal as OT
        sp = hgsynth.spec(name)
        n = max(1, sp.num_nodes // k)
        rng = np.random.default_rng(7)
        X = hgsynth.bf16_round(rng.standard_normal((n, sp.d), dtype=np.float32))
        C = hgsynth.make_context(sp, rows=n)
        p = hgsynth.make_temporal_params(sp)
        dOut = hgsynth.bf16_round(rng.standard_normal((n, sp.d), dtype=np.float32))
        units = n
        for i in range(warmup + steps):
            t0 = time.perf_counter()
            OT.temporal_backward(X, C, p, dOut)
            if i >= warmup:
                times.append(time.perf_counter() - t0)
    elif kind == "hgt":
        from oracle import hgt as OH
        w = hgsynth.make_workload(sp, with_ids=False)
        g = w.graph
        ps = [hgsynth.make_hgt_params(sp, HGT_HEADS, layer=l) for l in range(sp.layers)]
        args = (g["src"], g["dst"], g["rel"], g["type_offsets"], g["rels"])
        units = sp.layers * sp.num_edges
        for i in range(warmup + steps):
            t0 = time.perf_counter()
            hs = [np.asarray(w.X, np.float64)]
            for p in ps:
                hs.append(OH.hgt_forward(*args, p, hs[-1], HGT_HEADS)[0])
            dh = np.asarray(w.dH_top, np.float64)
            for l in range(sp.layers - 1, -1, -1):
                dh, _ = OH.hgt_backward(*args, ps[l], hs[l], dh, HGT_HEADS)
            if i >= warmup:
                times.append(time.perf_counter() - t0)
    else:
        raise ValueError(kind)
    print(json.dumps({"seconds": times, "units": units, "edges": sp.num_edges, "value": units * len(times) / sum(times)}))


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def time_oracle(name: str, k: int, kind: str = "step", with_head: bool = True, steps: int = 1, warmup: int = 0) -> dict:
    cores = host_cores()
    env = dict(os.environ, OMP_NUM_THREADS=str(cores), OPENBLAS_NUM_THREADS=str(cores), MKL_NUM_THREADS=str(cores),
               CUDA_VISIBLE_DEVICES="")
    cmd = [sys.executable, os.path.abspath(__file__), "--workload", name, "--oracle-child", kind, "--oracle-k", str(k),
           "--oracle-steps", str(steps), "--oracle-warmup", str(warmup)] + ([] if with_head else ["--no-head"])
    r = subprocess.run(cmd, capture_output=True, text=True, env=env)
    if r.returncode != 0:
        raise RuntimeError(f"oracle sample failed: {r.stderr[-2000:]}")
    out = json.loads(r.stdout.strip().splitlines()[-1])
    out["cores"] = cores
    return out


def oracle_sample_text(o: dict, what: str) -> str:
    return (f"{what}: {o['edges']:,}-edge instance of the same recipe, the fp64 numpy oracle as it stands, "
            f"{len(o['seconds'])} run(s) of {statistics.median(o['seconds']):.2f} s, BLAS allowed {o['cores']} "
            f"host threads (the segment sums run on one)")


# ------------------------------------------------------------------------------------------------
# clocks during the timed region
# ------------------------------------------------------------------------------------------------
class Clocks:
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.3)
        self.proc.terminate()
        out, _ = self.proc.communicate(timeout=10)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------------------------------------
# algorithmic bytes / flops per step for each kernel (from the graph's own statistics)
# ------------------------------------------------------------------------------------------------
HUB, CHUNK = 512, 512
FUSE = 32  # the fused mean layer streams rows of at most this many runs in its projection


def _graph_of(w):
    """(graph dict, overlap rows) of a hgsynth Workload (numpy) or a hgsynth.device workload (torch)."""
    if isinstance(w, dict):
        return w["graph"], int(len(w["overlap_local"]))
    return w.graph, int(len(w.overlap_local))


def graph_stats(w) -> dict:
    """Row, run and edge counts as the mean layer's aggregation kernels see them (torch, on the
    arrays' device).  A run is one entry of an aggregation list: the parallel edges of a node pair
    (same relation) with their multiplicity.  Forward rows are the CSR rows of each (relation,
    destination); backward rows are node-major (a node's out-edges of every relation); a row above
    HUB runs goes through chunks of CHUNK runs."""
    import torch
    g, n_ov = _graph_of(w)
    tt_ = lambda a: a if torch.is_tensor(a) else torch.from_numpy(np.ascontiguousarray(a))  # noqa: E731
    src, dst, rel = tt_(g["src"]).long(), tt_(g["dst"]).long(), tt_(g["rel"]).long()
    offs = [int(x) for x in g["type_offsets"]]
    N, R = offs[-1], len(g["rels"])
    nz = lambda x: int(torch.count_nonzero(x))  # noqa: E731
    blank = lambda: dict(E_nh=0, E_h=0, R_nh=0, R_h=0, U_nh=0, U_h=0, chunks=0, R_short=0, U_short=0,  # noqa: E731
                         rows_long=0)
    st = dict(N=N, E=int(src.shape[0]), RR=0, CC=0, n_ov=n_ov, fwd=blank(), bwd=blank(), types=[], rels=[])
    for t in range(len(offs) - 1):
        st["types"].append(dict(n=offs[t + 1] - offs[t], R=sum(1 for r in g["rels"] if r[1] == t), nnz=0))
    for r, (ts, tt) in enumerate(g["rels"]):
        m = rel == r
        s_r, d_r = src[m], dst[m]
        st["RR"] += offs[tt + 1] - offs[tt]
        st["CC"] += offs[ts + 1] - offs[ts]
        st["rels"].append(dict(n_t=offs[tt + 1] - offs[tt], n_s=offs[ts + 1] - offs[ts], E=int(s_r.shape[0]),
                               nnz=nz(torch.bincount(d_r - offs[tt], minlength=offs[tt + 1] - offs[tt]))))
        # forward: one CSR row per (relation, destination); its runs are the distinct sources
        u = torch.unique(d_r * N + s_r)
        u_dst, u_src = u // N, u % N
        runs = torch.bincount(u_dst, minlength=N)
        hub_run = runs[u_dst] > HUB
        edges = torch.bincount(d_r, minlength=N)
        a = st["fwd"]
        a["R_h"] += nz(hub_run)
        a["R_nh"] += int(u.shape[0]) - nz(hub_run)
        a["E_h"] += int(edges[runs > HUB].sum())
        a["E_nh"] += int(edges[runs <= HUB].sum())
        a["U_h"] += nz(torch.bincount(u_src[hub_run], minlength=N))
        a["U_nh"] += nz(torch.bincount(u_src[~hub_run], minlength=N))
        hr = runs[runs > HUB]
        a["chunks"] += int(((hr + CHUNK - 1) // CHUNK).sum())
        short = runs[u_dst] <= FUSE  # runs the fused projection streams itself
        a["R_short"] += nz(short)
        a["U_short"] += nz(torch.bincount(u_src[short], minlength=N))
        a["rows_long"] += nz(runs > FUSE)
        del u, u_dst, u_src, runs, hub_run, edges, short
    for r, (_, tt) in enumerate(g["rels"]):
        st["types"][tt]["nnz"] += st["rels"][r]["nnz"]  # stored relation rows (non-empty CSR rows)
    st["NNZ"] = sum(r["nnz"] for r in st["rels"])
    # backward: one node-major row per node; its runs are the distinct (relation, destination) dMs
    # rows it reads
    read = rel * N + dst
    u = torch.unique(src * (R * N) + read)
    u_src, u_read = u // (R * N), u % (R * N)
    runs = torch.bincount(u_src, minlength=N)
    hub_run = runs[u_src] > HUB
    edges = torch.bincount(src, minlength=N)
    a = st["bwd"]
    a["R_h"] = nz(hub_run)
    a["R_nh"] = int(u.shape[0]) - a["R_h"]
    a["E_h"] = int(edges[runs > HUB].sum())
    a["E_nh"] = int(edges[runs <= HUB].sum())
    a["U_h"] = nz(torch.bincount(u_read[hub_run], minlength=R * N))
    a["U_nh"] = nz(torch.bincount(u_read[~hub_run], minlength=R * N))
    hr = runs[runs > HUB]
    a["chunks"] = int(((hr + CHUNK - 1) // CHUNK).sum())
    return st


def kernel_models(st: dict, sp) -> dict:
    """{kernel: (bytes per step, flops per step)}: compulsory traffic (each distinct row read once,
    every output written once, index arrays read once) and the arithmetic of the definition."""
    b, d, L, N, RR, CC = (4 if sp.dtype == "f32" else 2), sp.d, sp.layers, st["N"], st["RR"], st["CC"]
    f, bw = st["fwd"], st["bwd"]
    row = d * b
    m = {}
    # aggregation (mean layer), compulsory bytes per step: each distinct row it reads once, the
    # run lists (column and count, 8 bytes per run) and row pointers once, every output row written
    # once, the fp32 chunk partials written and read.  The rows gathered per run (one per run, served
    # by L1 / L2 where a row recurs) are reported beside them as `gathered` (not HBM traffic).
    NNZ = st.get("NNZ", RR)  # stored (non-empty) relation rows
    m["agg_fwd_rows"] = (L * (12 * NNZ + 8 * f["R_nh"] + row * f["U_nh"] + row * NNZ + 4 * d * f["chunks"]), 0)
    m["agg_fwd_chunks"] = (L * (8 * f["R_h"] + row * f["U_h"] + 4 * d * f["chunks"]), 0)
    m["agg_bwd_nodes"] = (L * (4 * (N + 1) + 8 * bw["R_nh"] + row * bw["U_nh"] + 2 * row * N + 4 * d * bw["chunks"]), 0)
    m["agg_bwd_chunks"] = (L * (8 * bw["R_h"] + row * bw["U_h"] + 4 * d * bw["chunks"]), 0)
    m["gathered"] = {"agg_fwd_rows": L * f["R_nh"] * (8 + row), "agg_fwd_chunks": L * f["R_h"] * (8 + row),
                     "agg_bwd_nodes": L * bw["R_nh"] * (8 + row), "agg_bwd_chunks": L * bw["R_h"] * (8 + row)}
    fb = ff = bb = bf = 0
    for t in st["types"]:
        n, R = t["n"], t["R"]
        fb += n * row * (R + 4) + 8 * n
        ff += 2 * n * d * (R * d + d)
        bb += n * row * (6 + R) + 8 * n
        bf += 2 * n * d * (d + R * d)
    m["proj_fwd_simt"] = (L * fb, L * ff)
    m["proj_bwd_simt"] = (L * bb, L * bf)
    m["wgrad_partial"] = (L * 2 * row * (N + RR), L * 2 * d * d * (N + RR))
    # tensor-core path (fused weights V_r = W_r W_agg as hi / lo bf16 pairs), M_r and dM_r stored
    # for the non-empty relation rows only: per node of type t with R relations into t, nnz of them
    # stored
    tf = tfl = lb = pb = pfl = 0
    for t in st["types"]:
        n, R, nnz = t["n"], t["R"], t.get("nnz", t["n"] * t["R"])
        tf += n * (3 * row + 8) + row * nnz   # read H_in, the stored M_r rows; write U, H_out, statistics
        tfl += 2 * 2 * n * d * d * R         # two products per relation (hi, lo)
        lb += n * (5 * row + 8)              # read dH_out, U, H_in, statistics; write dY, dU
        pb += nnz * (2 * row + 12)           # gather dU, write dM_r, read the row list and degrees
        pfl += 2 * 2 * nnz * d * d
    m["proj_fwd_tc"] = (L * tf, L * tfl)
    m["ln_act_bwd"] = (L * lb, 0)
    m["proj_bwd_tc"] = (L * pb, L * pfl)
    m["wgrad_tc"] = (L * (2 * row + 4) * NNZ, L * 2 * d * d * NNZ)  # G_r = M_r^T dU over the stored rows
    # the fused mean layer: the projection and the weight gradient sum the rows of at most FUSE runs
    # themselves (run lists, 24 bytes of row metadata per stored row, each distinct source row once)
    # and read the longer rows' means; M_r is neither written nor read back
    fuse_in = 8 * f["R_short"] + 24 * NNZ + row * f["U_short"] + row * f["rows_long"]
    m["proj_fwd_gather_tc"] = (L * (tf - row * NNZ + fuse_in), L * tfl)
    m["wgrad_gather_tc"] = (L * ((row + 4) * NNZ + fuse_in), L * 2 * d * d * NNZ)
    m["gathered"].update({"proj_fwd_gather_tc": L * f["R_short"] * (8 + row), "wgrad_gather_tc": L * f["R_short"] * (8 + row)})
    # per 8-bit pass over the keys: read and write of key, edge id and endpoint; three stable sorts
    # (by source id, then CSR row: (row, source, edge id); that order by CSC row)
    passes = lambda rows: max(1, -(-int(rows).bit_length() // 8))  # noqa: E731
    m["radix_scatter"] = (2 * 12 * st["E"] * (passes(N) + passes(RR) + passes(CC)), 0)
    nl = st.get("n_lab", 0)
    if nl:
        # per labelled row: its H row (and a replica row for overlap rows, not counted), the saved Hm
        # and dA rows written, the label; backward: dA read, dH row read and written
        m["head_fwd_simt"] = (nl * (3 * row + 8), 2 * nl * d * d)
        m["head_bwd_dx_simt"] = (nl * (3 * row + 8), 2 * nl * d * d)
        wb, wf = m["wgrad_tc"]
        m["wgrad_tc"] = (wb + 2 * nl * row, wf + 2 * nl * d * d)  # dW1 = Hm^T dA shares the kernel
    no = st["n_ov"]
    m["align_colstats"] = (3 * 2 * no * (row + 4), 0)        # 3 passes over both gathered views
    m["align_gram_tc"] = (2 * no * (row + 4), 2 * 2 * no * d * d)
    m["align_bwd_tc"] = (2 * no * (4 * row + 8), 2 * 2 * no * d * d)  # per view: H_a, H_b, dH read, dH write
    return m


def load_peaks() -> tuple:
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as fh:
            return json.load(fh), "measured"
    return dict(FALLBACK), "fallback"


# kernels the library times under another name than their function's
KERNEL_ALIASES = {"agg_fwd_chunks": "agg_chunks", "agg_bwd_chunks": "agg_chunks"}


def _source_hash(source: str) -> str:
    import glob
    import hashlib
    csrc = os.path.join(ROOT, "paper_2608_02168_gb300", "csrc")
    h = hashlib.sha256()
    for f in [os.path.join(csrc, source)] + sorted(glob.glob(os.path.join(csrc, "*.cuh"))):
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def _kernel_source(fn: str) -> str | None:
    """The .cu file of paper_2608_02168_gb300/csrc that defines kernel `fn`."""
    import glob
    import re
    pat = re.compile(r"__global__[^;{]*?\b" + re.escape(fn) + r"\s*\(", re.S)
    for f in sorted(glob.glob(os.path.join(ROOT, "paper_2608_02168_gb300", "csrc", "*.cu"))):
        with open(f) as fh:
            if pat.search(fh.read()):
                return os.path.basename(f)
    return None


def fold_ncu_traffic(csv_path: str, out_path: str) -> dict:
    """DRAM bytes per launch of every kernel in an ncu metrics CSV (one row per launch and metric),
    keyed by kernel function name, with the launch count and the SHA-256 of the kernel's source file
    and the shared headers (measured_traffic uses an entry only while that hash still matches)."""
    import csv
    import re
    acc = {}
    with open(csv_path, newline="") as fh:
        lines = [ln for ln in fh if ln.startswith('"')]
    for row in csv.DictReader(lines):
        name = row.get("Kernel Name", "")
        m = re.match(r"(?:void\s+)?(?:[\w:]*::)?(\w+)", name.replace("hg::", ""))
        if not m:
            continue
        fn = m.group(1)
        e = acc.setdefault(fn, {"ids": set(), "read": 0.0, "write": 0.0, "ns": 0.0})
        e["ids"].add(row["ID"])
        v = float(row["Metric Value"].replace(",", ""))
        unit = row.get("Metric Unit", "")
        scale = {"byte": 1, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9, "nsecond": 1, "usecond": 1e3, "msecond": 1e6}
        v *= scale.get(unit, 1)
        metric = row["Metric Name"]
        if metric == "dram__bytes_read.sum":
            e["read"] += v
        elif metric == "dram__bytes_write.sum":
            e["write"] += v
        elif metric == "gpu__time_duration.sum":
            e["ns"] += v
    out = {}
    for fn, e in sorted(acc.items()):
        src = _kernel_source(fn)
        if src is None or not (e["read"] or e["write"]):
            continue
        n = len(e["ids"])
        out[fn] = {"launches": n, "bytes_per_launch": int(round((e["read"] + e["write"]) / n)),
                   "ns_per_launch": int(round(e["ns"] / n)), "source": src, "sha256": _source_hash(src)}
    with open(out_path, "w") as fh:
        json.dump(out, fh, indent=1, sort_keys=True)
    return out


def measured_traffic(kernel: str):
    """DRAM bytes per launch of `kernel` from the committed ncu capture (profiles/traffic.json), or
    None when there is none or the kernel's sources changed since it was taken."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as fh:
        entry = json.load(fh).get(KERNEL_ALIASES.get(kernel, kernel))
    if not entry:
        return None
    return int(entry["bytes_per_launch"]) if _source_hash(entry["source"]) == entry["sha256"] else None


def roofline(report: dict, models: dict, steps: int, peaks: dict, src: str, dom=None) -> tuple:
    total = sum(ms for _, ms in report.values()) or 1.0
    shares = {k: round(ms / total, 4) for k, (_, ms) in sorted(report.items(), key=lambda kv: -kv[1][1])}
    dom = dom or max(report, key=lambda k: report[k][1])
    n, ms = report[dom]
    by, fl = models.get(dom, (0, 0))
    secs = ms / 1e3
    alu_peak = 152 * 128 * 2 * peaks.get("sm_max_mhz", 2070.0) * 1e6 / 1e12  # fp32 FMA, TFLOP/s
    if dom.endswith("_simt") or dom == "wgrad_partial":  # CUDA-core kernels: fp32 FMA bound
        ach = fl * steps / secs / 1e12 if secs > 0 else 0.0
        rf = dict(bound="alu", achieved=round(ach, 3), peak=round(alu_peak, 1), unit="TFLOP/s",
                  peak_source="derived: 152 SMs x 128 fp32 lanes x 2 flop x max SM clock")
    else:
        ach = by * steps / secs / 1e9 if secs > 0 else 0.0
        rf = dict(bound="hbm", achieved=round(ach, 1), peak=peaks["hbm_gbs"], unit="GB/s",
                  peak_source=f"{src} hbm_gbs")
    rf["frac"] = round(rf["achieved"] / rf["peak"], 4) if rf["peak"] else None
    if rf["bound"] == "hbm":
        rf["frac_of_nominal"] = round(rf["achieved"] / NOMINAL_HBM_GBS, 4)
    rf["traffic"] = measured_traffic(dom)
    rf.update(kernel=dom, launches=n, avg_launch_ms=round(ms / max(n, 1), 4),
              algorithmic_bytes_per_launch=int(by * steps / max(n, 1)), flops_per_launch=int(fl * steps / max(n, 1)))
    gat = models.get("gathered", {}).get(dom)
    if gat is not None:
        rf["model"] = ("compulsory: each distinct row read once, run lists and pointers once, outputs written once; "
                       "gathered_*: one feature row and its 8-byte run entry per run, repeated rows served by L1/L2")
        rf["gathered_bytes_per_launch"] = int(gat * steps / max(n, 1))
        rf["gathered_gbs"] = round(gat * steps / secs / 1e9, 1) if secs > 0 else None
    return rf, shares


def measure_overlap_build(w: dict, steps: int, warmup: int, dev, with_cpu: bool) -> dict:
    """The overlapping-subgraph construction (Section 3.1; done once before training, so it is not
    part of the step) on the workload's graph taken as the global graph: subgraph 0 of BUILD_K,
    h-index bound BUILD_THETA, budget BUILD_BUDGET * N / BUILD_K.  Device time per call."""
    import torch
    from paper_2608_02168_gb300 import hg
    g = w["graph"]
    offs = [int(x) for x in g["type_offsets"]]
    src, dst, rel = g["src"], g["dst"], g["rel"]
    E = int(src.shape[0])
    ws = torch.empty(hg.hg_overlap_build_workspace_size(offs[-1], E), dtype=torch.uint8, device=dev)
    M = int(BUILD_BUDGET * offs[-1] / BUILD_K)

    def call():
        return hg.hg_overlap_build(src, dst, rel, offs, BUILD_K, 0, BUILD_THETA, M, 21, 22, workspace=ws)

    for _ in range(max(warmup, 1)):
        out = call()
    torch.cuda.synchronize()
    # the binding reads the counts back (one synchronisation per call): time with events per call
    times = []
    for _ in range(steps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        out = call()
        e1.record()
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
    hg.hg_timing_enable(True)
    hg.hg_timing_report()
    call()
    torch.cuda.synchronize()
    hg.hg_timing_enable(False)
    rep = hg.hg_timing_report()
    tot = sum(ms for _, ms in rep.values()) or 1.0
    ms = statistics.median(times)
    # algorithmic bytes of one call: per edge, the endpoint reads of the degree, list-fill, candidate
    # and keep passes (4 x 8 B), the neighbour degrees and list slots written by the fill (2 x 8 B),
    # one read of both incidence entries by the h-index (8 B) and the keep flag (4 B); per node, the
    # ten 4-byte node arrays written and read once (40 B)
    peaks, psrc = load_peaks()
    byt = 60 * E + 40 * offs[-1]
    ach = byt / (ms / 1e3) / 1e9
    res = {"workload": workload_desc(w["spec"]), "ms": round(ms, 4), "edges_per_s": E / (ms / 1e3),
           "counts": out["counts"],
           "roofline": {"bound": "hbm", "achieved": round(ach, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
                        "peak_source": f"{psrc} hbm_gbs", "frac": round(ach / peaks["hbm_gbs"], 4),
                        "frac_of_nominal": round(ach / NOMINAL_HBM_GBS, 4),
                        "algorithmic_bytes_per_call": int(byt), "scope": "whole call"},
           "config": {"K": BUILD_K, "k": 0, "theta": BUILD_THETA, "M": M},
           "kernel_time_share": {k: round(v / tot, 4) for k, (_, v) in sorted(rep.items(), key=lambda kv: -kv[1][1])},
           "cpu_baseline": None}
    if with_cpu:
        o = time_oracle(w["spec"].name, sample_scale(w["spec"]), "build")
        res["cpu_baseline"] = {"value": o["value"], "unit": "edges/s", "cores": o["cores"], "kind": "oracle",
                               "sample": oracle_sample_text(o, "the construction")}
    return res


def measure_temporal(sp, steps: int, warmup: int, dev, with_cpu: bool) -> dict:
    """The temporal module (Section 3.2, Eq. 12-13: attention over each node's last w = 3 states and
    the GRU cell), forward and backward over every node of the workload, with synthetic spatial
    embeddings, context states and upstream gradient.  Device time per forward + backward."""
    import torch
    from paper_2608_02168_gb300 import hg
    n, d, w = sp.num_nodes, sp.d, hgsynth.TEMPORAL_WINDOW
    td = torch.float32 if sp.dtype == "f32" else torch.bfloat16
    rng = np.random.default_rng(7)
    X = torch.from_numpy(hgsynth.bf16_round(rng.standard_normal((n, d), dtype=np.float32))).to(dev, td)
    C = torch.from_numpy(hgsynth.make_context(sp)).to(dev, td)
    dOut = torch.from_numpy(hgsynth.bf16_round(rng.standard_normal((n, d), dtype=np.float32))).to(dev, td)
    p = hgsynth.make_temporal_params(sp)
    prm = hg.TemporalParams(*(torch.from_numpy(p[k]).to(dev, td) for k in ("Wa", "r", "W_i", "W_h", "b_i", "b_h")),
                            w=w)
    s_b, k_b = hg.hg_temporal_workspace_size(n, d, w, td)
    saved = torch.empty(s_b, dtype=torch.uint8, device=dev)
    scratch = torch.empty(k_b, dtype=torch.uint8, device=dev)
    out = torch.empty(n, d, dtype=td, device=dev)
    dX = torch.empty_like(out)
    f = dict(dtype=torch.float32, device=dev)
    grads = {"Wa": torch.empty(d, d, **f), "r": torch.empty(d, **f), "W_i": torch.empty(d, 3 * d, **f),
             "W_h": torch.empty(d, 3 * d, **f), "b_i": torch.empty(3 * d, **f), "b_h": torch.empty(3 * d, **f)}

    def call():
        hg.hg_temporal_fwd(prm, X, C, out, saved, scratch)
        hg.hg_temporal_bwd(prm, X, C, saved, dOut, dX, grads, scratch)

    for _ in range(max(warmup, 1)):
        call()
    torch.cuda.synchronize()
    times = []
    for _ in range(steps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        call()
        e1.record()
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
    hg.hg_timing_enable(True)
    hg.hg_timing_report()
    call()
    torch.cuda.synchronize()
    hg.hg_timing_enable(False)
    rep = hg.hg_timing_report()
    tot = sum(ms for _, ms in rep.values()) or 1.0
    ms = statistics.median(times)
    # algorithmic bytes per node: forward reads x and the w context rows and writes H^t, H~ and a;
    # backward reads x, the context, dH^t, H~ and a and writes dX
    b = 4 if sp.dtype == "f32" else 2
    per_node = (2 * (1 + w) + 2 + 1 + 1 + 1) * d * b + 2 * 4 * w
    flops = (2 * w + 12 + 36 + 4 * w) * d * d * n  # forward products, backward recomputation and gradients
    peaks, psrc = load_peaks()
    ach = per_node * n / (ms / 1e3) / 1e9
    res = {"ms": round(ms, 4), "nodes_per_s": n / (ms / 1e3), "nodes": n, "w": w, "d": d, "dtype": sp.dtype,
           "roofline": {"bound": "hbm", "achieved": round(ach, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
                        "peak_source": f"{psrc} hbm_gbs", "frac": round(ach / peaks["hbm_gbs"], 4),
                        "frac_of_nominal": round(ach / NOMINAL_HBM_GBS, 4),
                        "algorithmic_bytes_per_call": int(per_node * n), "scope": "forward + backward"},
           "tensor": {"achieved_tflops": round(flops / (ms / 1e3) / 1e12, 1), "peak": peaks.get("bf16_tflops"),
                      "flops_per_call": int(flops)},
           "kernel_time_share": {k: round(v / tot, 4) for k, (_, v) in sorted(rep.items(), key=lambda kv: -kv[1][1])},
           "cpu_baseline": None}
    if with_cpu:
        o = time_oracle(sp.name, max(1, n // 25_000), "temporal")
        res["cpu_baseline"] = {"value": o["value"], "unit": "nodes/s", "cores": o["cores"], "kind": "oracle",
                               "sample": oracle_sample_text(o, f"forward and backward over {o['units']:,} nodes")}
    return res


def measure_hgt(w: dict, steps: int, warmup: int, dev, with_cpu: bool) -> dict:
    """The attention variant of the layer (Eq. 6-11, HGT_HEADS heads): the workload's L layers
    forward and backward on its graph (CSR built once), synthetic upstream gradient.  Device time
    per forward + backward of the stack."""
    import torch
    from paper_2608_02168_gb300 import hg
    sp, g = w["spec"], w["graph"]
    td = torch.float32 if sp.dtype == "f32" else torch.bfloat16
    G = hg.hg_build_csr(g["src"], g["dst"], g["rel"], g["type_offsets"], g["rels"])
    params = []
    for l in range(sp.layers):
        p = hgsynth.make_hgt_params(sp, HGT_HEADS, layer=l)
        params.append(hg.HgtParams({k: torch.from_numpy(v).to(dev, torch.float32 if k == "mu" else td)
                                    for k, v in p.items()}, HGT_HEADS))
    sb, kb = hg.hg_hgt_workspace_size(G, params[0])
    saved = [torch.empty(sb, dtype=torch.uint8, device=dev) for _ in params]
    scratch = torch.empty(kb, dtype=torch.uint8, device=dev)
    N, d = sp.num_nodes, sp.d
    Hs = [w["X"]] + [torch.empty(N, d, dtype=td, device=dev) for _ in params]
    dHs = [torch.empty(N, d, dtype=td, device=dev) for _ in range(len(params))] + [w["dH_top"]]
    f = dict(dtype=torch.float32, device=dev)
    grads = [{k: torch.empty(np.shape(v), **f) for k, v in hgsynth.make_hgt_params(sp, HGT_HEADS).items()}
             for _ in params]

    def call():
        for l, P in enumerate(params):
            hg.hg_hgt_fwd(G, P, Hs[l], Hs[l + 1], saved[l], scratch)
        for l in range(len(params) - 1, -1, -1):
            hg.hg_hgt_bwd(G, params[l], Hs[l], saved[l], dHs[l + 1], dHs[l], grads[l], scratch)

    for _ in range(max(warmup, 1)):
        call()
    torch.cuda.synchronize()
    times = []
    for _ in range(steps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        call()
        e1.record()
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
    hg.hg_timing_enable(True)
    hg.hg_timing_report()
    call()
    torch.cuda.synchronize()
    hg.hg_timing_enable(False)
    rep = hg.hg_timing_report()
    tot = sum(ms for _, ms in rep.values()) or 1.0
    ms = statistics.median(times)
    # no-reuse model per layer: the forward and the two backward edge passes each read a run entry
    # (8 bytes: column and multiplicity) and gather two rows per run of parallel edges (K and V; K
    # and V; Q' and dS), plus the dense rows (K, V, Q', S written and read, the projection's and
    # the backward products' rows)
    b = 4 if sp.dtype == "f32" else 2
    offs = [int(x) for x in g["type_offsets"]]
    RR = sum(offs[t + 1] - offs[t] for _, t in g["rels"])
    runs = int(torch.unique((g["rel"].long() * N + g["dst"].long()) * N + g["src"].long()).numel())
    per_layer = 3 * runs * (8 + 2 * sp.d * b) + (2 * RR + 10 * sp.num_nodes) * sp.d * b
    peaks, psrc = load_peaks()
    ach = sp.layers * per_layer / (ms / 1e3) / 1e9
    res = {"workload": workload_desc(sp), "ms": round(ms, 4), "layers": sp.layers, "heads": HGT_HEADS,
           "layers_fwd_bwd_edges_per_s": sp.layers * sp.num_edges / (ms / 1e3),
           "roofline": {"bound": "hbm", "achieved": round(ach, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
                        "peak_source": f"{psrc} hbm_gbs", "frac": round(ach / peaks["hbm_gbs"], 4),
                        "frac_of_nominal": round(ach / NOMINAL_HBM_GBS, 4),
                        "model": "no-reuse: 3 edge passes x (8 + 2 d b) per run of parallel edges + (2 csr_rows + 10 N) d b per layer",
                        "runs": runs,
                        "algorithmic_bytes_per_call": int(sp.layers * per_layer)},
           "kernel_time_share": {k: round(v / tot, 4) for k, (_, v) in sorted(rep.items(), key=lambda kv: -kv[1][1])},
           "cpu_baseline": None}
    if with_cpu:
        o = time_oracle(sp.name, 4 * sample_scale(sp), "hgt")
        res["cpu_baseline"] = {"value": o["value"], "unit": UNIT, "cores": o["cores"], "kind": "oracle",
                               "sample": oracle_sample_text(o, f"{sp.layers} attention layers forward and backward")}
    return res


LAYER_KERNELS = ("agg_fwd_rows", "agg_fwd_chunks", "agg_bwd_nodes", "agg_bwd_chunks", "combine_chunk_partials",
                 "fuse_weights", "proj_fwd_tc", "ln_act_bwd", "proj_bwd_tc", "wgrad_tc", "wgrad_finish", "reduce_lanes",
                 "proj_fwd_simt", "proj_bwd_simt", "wgrad_partial")


def layer_stack_bytes(models: dict) -> int:
    """Algorithmic bytes of the L-layer forward + backward in one step: the aggregations' compulsory
    bytes (each distinct row once) and the projections' streamed bytes."""
    total = 0
    for k in ("agg_fwd_rows", "agg_fwd_chunks", "agg_bwd_nodes", "agg_bwd_chunks", "proj_fwd_tc", "ln_act_bwd",
              "proj_bwd_tc", "wgrad_tc"):
        total += models.get(k, (0, 0))[0]
    return int(total)


# ------------------------------------------------------------------------------------------------
# the hot-path step on one workload
# ------------------------------------------------------------------------------------------------
def step_inputs(w: dict, use_head: bool) -> dict:
    g = w["graph"]
    inp = {"src": g["src"], "dst": g["dst"], "rel": g["rel"], "X": w["X"]}
    if use_head:
        inp.update(lab_idx=w["lab_idx"], lab_y=w["lab_y"])
    else:
        inp["dH_top"] = w["dH_top"]
    if w["spec"].view_b == "perturbed":
        inp.update(X_b=w["X_b"], overlap_idx=w["overlap_local"])
    else:
        inp.update(gid_a=w["gid_a"], gid_b=w["gid_b"], H_bank=w["H_b"])
    return inp


def make_path(w: dict, dev, use_head: bool, fused: bool = False):
    from paper_2608_02168_gb300.step import HotPath
    sp, g = w["spec"], w["graph"]
    return HotPath(g["type_offsets"], g["rels"], int(g["src"].shape[0]), sp.d, sp.dtype, w["params"], view=sp.view_b,
                   n_overlap_max=int(len(w["overlap_local"])),
                   n_gid_a=0 if "gid_a" not in w else int(len(w["gid_a"])),
                   n_gid_b=0 if "gid_b" not in w else int(len(w["gid_b"])), device=dev,
                   head_params=hgsynth.make_head_params(sp) if use_head else None,
                   n_lab_max=int(len(w["lab_idx"])) if use_head else 0, fused=fused)


def path_digest(path) -> dict:
    """Integer sums of the bit patterns of the path's last step: every layer output, every input
    gradient and every weight gradient.  Equal digests of two runs mean equal results, bit for bit,
    in practice."""
    import torch

    def bits(t):
        return int(t.view(torch.int16 if t.element_size() == 2 else torch.int32).sum(dtype=torch.int64))
    return {"H": [bits(t) for stack in path.H for t in stack], "dH": [bits(t) for stack in path.dH for t in stack],
            "grads": [bits(gd[k]) for stack in path.grads for gd in stack for k in sorted(gd)]}


def run_hot_path(w: dict, dev, steps: int, warmup: int, world: int, use_head: bool, clocks=None, e2e: bool = False,
                 fused: bool = False) -> dict:
    """Times `steps` steps (after `warmup`), then the phases of the step and the per-kernel report;
    optionally the same steps end to end from pinned host inputs.  fused: the fused mean layer."""
    import torch
    from paper_2608_02168_gb300 import hg
    sp = w["spec"]
    path = make_path(w, dev, use_head, fused)
    devin = step_inputs(w, use_head)
    stream = torch.cuda.current_stream()

    def step(inp, marks=None):
        kw = {k: inp[k] for k in ("X_b", "overlap_idx", "gid_a", "gid_b", "H_bank", "lab_idx", "lab_y") if k in inp}
        path.step(inp["src"], inp["dst"], inp["rel"], inp["X"], inp.get("dH_top"), marks=marks, **kw)

    for _ in range(max(warmup, 0)):
        step(devin)
    torch.cuda.synchronize()
    if clocks is not None:
        clocks.start()
    rank_barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        torch.cuda.nvtx.range_push("step")  # profilers select the timed steps by this range
        step(devin)
        torch.cuda.nvtx.range_pop()
    e1.record(stream)
    torch.cuda.synchronize()
    rank_barrier(world)
    clk = clocks.stop() if clocks is not None else None
    t = max_time_over_ranks(e0.elapsed_time(e1) / 1e3, world, dev)
    # phases of the step (uninstrumented)
    phase_ms = {}
    for _ in range(steps):
        marks = []
        m0 = torch.cuda.Event(enable_timing=True)
        m0.record(stream)
        step(devin, marks)
        torch.cuda.synchronize()
        prev = m0
        for name, ev in marks:
            phase_ms[name] = phase_ms.get(name, 0.0) + prev.elapsed_time(ev) / steps
            prev = ev
    # per-kernel durations from a second, instrumented run of the same steps (the library records
    # CUDA events around each of its launches, which the headline timing leaves out)
    hg.hg_timing_enable(True)
    hg.hg_timing_report()
    for _ in range(steps):
        step(devin)
    torch.cuda.synchronize()
    hg.hg_timing_enable(False)
    report = hg.hg_timing_report()
    units = sp.layers * int(w["graph"]["src"].shape[0])
    res = {"t": t, "value": weak_scaling_value(world, units, steps, t), "ms_per_step": 1e3 * t / steps,
           "phases_ms": {k: round(v, 4) for k, v in phase_ms.items()}, "report": report, "clocks": clk,
           "launches_per_step": sum(n for n, _ in report.values()) / max(steps, 1)}
    lay = phase_ms.get("forward", 0) + phase_ms.get("backward", 0)
    res["layers_fwd_bwd_edges_per_s"] = units / (lay / 1e3) if lay else None
    res["csr_build_edges_per_s"] = units / sp.layers / (phase_ms["graph"] / 1e3) if phase_ms.get("graph") else None
    if e2e:
        res["e2e"] = run_e2e(path, step, devin, dev, steps, world, units, use_head)
    res["loss"] = [float(x) for x in path.loss.cpu()]
    res["head_loss"] = [float(x) for x in path.head_loss.cpu()] if use_head else None
    res["digest"] = path_digest(path)
    res["saved_bytes_per_layer"] = int(path.saved[0][0].numel())
    del path
    return res


def fused_summary(res: dict, rf: dict) -> dict:
    """The fused mean layer (M_r never stored) against the plain layer on the same workload."""
    lay = res["phases_ms"].get("forward", 0) + res["phases_ms"].get("backward", 0)
    lay_f = rf["phases_ms"].get("forward", 0) + rf["phases_ms"].get("backward", 0)
    per = lambda rep, k: round(rep[k][1] / rep[k][0], 4) if k in rep and rep[k][0] else None  # noqa: E731
    kern = {k: {"ms_per_launch": per(rf["report"], k), "launches_per_step": rf["report"][k][0] / max(rf["steps"], 1)}
            for k in ("proj_fwd_gather_tc", "wgrad_gather_tc", "agg_fwd_long_rows", "agg_fwd_chunks") if k in rf["report"]}
    return {"ms_per_step": round(rf["ms_per_step"], 4), "phases_ms": rf["phases_ms"],
            "layers_fwd_bwd_edges_per_s": rf["layers_fwd_bwd_edges_per_s"],
            "layer_stack_ms": round(lay_f, 4), "plain_layer_stack_ms": round(lay, 4),
            "bitwise_equal_to_plain": {k: rf["digest"][k] == res["digest"][k] for k in res["digest"]},
            "saved_bytes_per_layer": rf["saved_bytes_per_layer"],
            "plain_saved_bytes_per_layer": res["saved_bytes_per_layer"], "kernels": kern,
            "plain_kernels": {k: per(res["report"], k) for k in ("proj_fwd_tc", "agg_fwd_rows", "wgrad_tc")}}


def run_e2e(path, step, devin, dev, steps, world, units, use_head) -> dict:
    """Same steps through the public API with every step's inputs copied in from pinned host memory
    (the copy of step i+1's inputs overlaps step i) and its loss read back."""
    import torch
    stream = torch.cuda.current_stream()
    pinned = {k: v.cpu().pin_memory() for k, v in devin.items()}
    h2d = sum(v.numel() * v.element_size() for v in pinned.values())
    result = path.head_loss if use_head else path.loss  # L_total (Eq. 20), or the alignment loss
    loss_host = torch.empty(result.numel(), dtype=torch.float32).pin_memory()
    bufs = [devin, {k: torch.empty_like(v) for k, v in devin.items()}]
    copy_stream = torch.cuda.Stream(device=dev)
    copied = [torch.cuda.Event(), torch.cuda.Event()]
    consumed = [torch.cuda.Event(), torch.cuda.Event()]

    def copy_in(i):
        b = i % 2
        with torch.cuda.stream(copy_stream):
            copy_stream.wait_event(consumed[b])  # the step that last read this buffer set is done
            for k, v in pinned.items():
                bufs[b][k].copy_(v, non_blocking=True)
            copied[b].record(copy_stream)

    rank_barrier(world)
    torch.cuda.synchronize()
    for ev in consumed:
        ev.record(stream)
    t0 = time.perf_counter()
    copy_in(0)
    for i in range(steps):
        if i + 1 < steps:
            copy_in(i + 1)
        stream.wait_event(copied[i % 2])
        step(bufs[i % 2])
        consumed[i % 2].record(stream)
        loss_host.copy_(result, non_blocking=True)
        stream.synchronize()  # the loss of step i is on the host
    torch.cuda.synchronize()
    te = max_time_over_ranks(time.perf_counter() - t0, world, dev)
    out = {"value": weak_scaling_value(world, units, steps, te), "unit": UNIT, "h2d_bytes_per_step": int(h2d),
           "d2h_bytes_per_step": int(loss_host.numel() * 4)}
    del bufs, pinned
    return out


def workload_summary(w: dict, res: dict, models: dict, steps: int, peaks: dict, psrc: str) -> dict:
    """The per-workload figures: whole step, layer stack (with its roofline over the summed
    algorithmic bytes of the layer kernels), CSR build, phases, dominant kernel."""
    sp = w["spec"]
    lay_ms = res["phases_ms"].get("forward", 0) + res["phases_ms"].get("backward", 0)
    lb = layer_stack_bytes(models)
    ach = lb / (lay_ms / 1e3) / 1e9 if lay_ms else 0.0
    rf, shares = roofline(res["report"], models, steps, peaks, psrc)
    return {"workload": workload_desc(sp), "value": res["value"], "unit": UNIT, "ms_per_step": round(res["ms_per_step"], 4),
            "layers_fwd_bwd_edges_per_s": res["layers_fwd_bwd_edges_per_s"],
            "csr_build_edges_per_s": res["csr_build_edges_per_s"], "phases_ms": res["phases_ms"],
            "layer_stack_roofline": {"bound": "hbm", "achieved": round(ach, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
                                     "frac": round(ach / peaks["hbm_gbs"], 4), "algorithmic_bytes_per_step": lb,
                                     "model": "aggregations: each distinct row once; projections: rows streamed"},
            "roofline": rf, "kernel_time_share": dict(list(shares.items())[:12]),
            "gpu_launches_per_step": res["launches_per_step"]}


def measure_ring(sp, dev, warmup: int) -> dict:
    """One full pass over the ring of sparse overlapping subgraphs (Algorithm 1 run in sequence on one
    GPU): subgraph k aligns with the detached final embeddings of subgraph k-1 (the first has no
    alignment term), synthetic upstream gradient.  Device time of the 16 steps after `warmup`
    steps on the first subgraphs."""
    import torch
    from hgsynth import device as hd
    from paper_2608_02168_gb300.step import Ring
    table = hd.ring_features(sp, dev)
    parts = [hd.make_ring_part(sp, k, table, dev) for k in range(sp.num_subgraphs)]
    del table
    dH = hd.make_features(sp, 0, dev, 4)
    params = [hgsynth.make_layer_params(sp, l) for l in range(sp.layers)]
    g0 = parts[0]["graph"]
    E = int(g0["src"].shape[0])
    ring = Ring(g0["type_offsets"], g0["rels"], E, sp.d, sp.dtype, params, device=dev)

    def run(p):
        g = p["graph"]
        ring.step(g["src"], g["dst"], g["rel"], p["X"], dH, p["gid"])

    for k in range(max(warmup, 1)):
        run(parts[k % len(parts)])
    ring.have_bank = False  # the timed pass starts a fresh sequence
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for p in parts:
        run(p)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    units = sp.num_subgraphs * sp.layers * E
    n_ov = int(ring.path.n_dev.item())
    del ring, parts
    return {"workload": workload_desc(sp), "subgraphs": sp.num_subgraphs, "ms_per_pass": round(ms, 3),
            "edges_per_s": units / (ms / 1e3), "overlap_rows_last_step": n_ov,
            "objective": "synthetic upstream gradient + 0.1 L_CCA against the previous subgraph"}


# ------------------------------------------------------------------------------------------------
def main():
    args = parse()
    if args.ncu_traffic:
        out = fold_ncu_traffic(args.ncu_traffic, os.path.join(ROOT, "profiles", "traffic.json"))
        print(json.dumps({k: v["bytes_per_launch"] for k, v in out.items()}))
        return
    if args.oracle_child:
        oracle_child_main(args.oracle_child, args.workload, args.oracle_k, args.oracle_steps, args.oracle_warmup,
                          not args.no_head)
        return
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    sp = hgsynth.spec(args.workload)
    if args.scale > 1:  # a smaller instance of the same recipe, for profiler captures only
        sp = scaled(sp, args.scale)
    if args.impl == "reference":
        if rank != 0:
            return
        run_reference(args, sp)
        return
    run_ours(args, sp, rank, world)


# ------------------------------------------------------------------------------------------------
# multi-GPU harness: one independent subgraph per rank (no collective on the data path); the
# timed region is bracketed by barriers and its duration is the maximum over the ranks
# ------------------------------------------------------------------------------------------------
def rank_barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_time_over_ranks(x: float, world: int, device) -> float:
    """The largest of the ranks' durations (every rank gets it)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def weak_scaling_value(world: int, edges_per_step: int, steps: int, seconds: float) -> float:
    """Whole-job throughput: every rank processes its own subgraph of the same size, so the units
    of all ranks over the slowest rank's time."""
    return world * edges_per_step * steps / seconds


def run_reference(args, sp):
    """The oracle, as it stands, on a bounded sample of the workload (one child process, its BLAS on
    every host core): warm-up and timed steps each one full step of the oracle."""
    k = sample_scale(sp)
    o = time_oracle(sp.name, k, "step", with_head=not args.no_head, steps=args.steps, warmup=args.warmup)
    secs = sum(o["seconds"])
    value = o["units"] * len(o["seconds"]) / secs
    sample = oracle_sample_text(o, "one step per timed step" + ("" if args.no_head else ", with the head and joint loss"))
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * secs / max(len(o["seconds"]), 1),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": workload_desc(sp), "sample": f"1/{k}-size instance of the same recipe"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": o["cores"], "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


def free_device_memory():
    import gc
    import torch
    gc.collect()
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def run_ours(args, sp, rank, world):
    import torch
    if world > 1:
        import torch.distributed as dist
        local = int(os.environ.get("LOCAL_RANK", "0"))
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    from paper_2608_02168_gb300 import build as hbuild
    hbuild.build()
    from hgsynth import device as hd

    dev = torch.device("cuda", torch.cuda.current_device())
    use_head = not args.no_head
    peaks, psrc = load_peaks()
    # the headline workload: this rank's subgraph, drawn on the device
    w = hd.make_workload(sp, sub=rank, device=dev, with_dH_top=not use_head)
    torch.cuda.synchronize()
    clocks = Clocks(dev.index if dev.index is not None else 0)
    res = run_hot_path(w, dev, args.steps, args.warmup, world, use_head, clocks=clocks, e2e=not args.no_e2e)
    stats = graph_stats(w)
    stats["n_lab"] = int(len(w["lab_idx"])) if use_head else 0
    models = kernel_models(stats, sp)
    fused = None
    if sp.dtype == "bf16" and sp.d == 128 and not args.no_fused:
        fs = min(args.steps, 5)
        rfu = run_hot_path(w, dev, fs, min(max(args.warmup, 1), 3), world, use_head, fused=True)
        rfu["steps"] = fs
        fused = fused_summary(res, rfu)
        fused["kernel_rooflines"] = [roofline(rfu["report"], models, fs, peaks, psrc, dom=k)[0]
                                     for k in ("proj_fwd_gather_tc", "wgrad_gather_tc") if k in rfu["report"]]
        free_device_memory()
    head = workload_summary(w, res, models, args.steps, peaks, psrc)
    rf, shares = roofline(res["report"], models, args.steps, peaks, psrc)
    top = [k for k in shares if k in models and k != "gathered"][:8]
    kernel_rooflines = [roofline(res["report"], models, args.steps, peaks, psrc, dom=k)[0] for k in top]
    del w
    free_device_memory()
    if rank != 0:
        if world > 1:
            torch.distributed.destroy_process_group()
        return
    # the other workloads (fewer steps) and one pass over the ring
    extra = {}
    if not args.no_extra and args.scale == 1:
        for name in EXTRA_WORKLOADS:
            if name == sp.name:
                continue
            spx = hgsynth.spec(name)
            wx = hd.make_workload(spx, device=dev, with_dH_top=not use_head)
            rx = run_hot_path(wx, dev, min(args.steps, 5), min(max(args.warmup, 1), 2), 1, use_head)
            stx = graph_stats(wx)
            stx["n_lab"] = int(len(wx["lab_idx"])) if use_head else 0
            extra[name] = workload_summary(wx, rx, kernel_models(stx, spx), min(args.steps, 5), peaks, psrc)
            del wx
            free_device_memory()
        extra["ring16-2m"] = measure_ring(hgsynth.spec("ring16-2m"), dev, warmup=2)
        free_device_memory()
    side_needed = not (args.no_build and args.no_temporal and args.no_hgt)
    ws = hd.make_workload(hgsynth.spec(SIDE_WORKLOAD), device=dev, with_dH_top=True) if side_needed else None
    with_cpu = not args.no_cpu_baseline
    build = None if args.no_build else measure_overlap_build(ws, args.steps, args.warmup, dev, with_cpu)
    temporal = None if args.no_temporal else measure_temporal(hgsynth.spec(SIDE_WORKLOAD), args.steps, args.warmup,
                                                                dev, with_cpu)
    hgt = None if args.no_hgt else measure_hgt(ws, args.steps, args.warmup, dev, with_cpu)
    del ws
    cpu = None
    if with_cpu:
        o = time_oracle(sp.name, sample_scale(sp), "step", with_head=use_head)
        cpu = {"value": o["value"], "unit": UNIT, "cores": o["cores"], "kind": "oracle",
               "sample": oracle_sample_text(o, "one full step" + (" with the head and joint loss" if use_head else ""))}
    out = {
        "metric": METRIC, "value": res["value"], "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": res["ms_per_step"], "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": sp.dtype, "data": "synthetic",
        "config": {"workload": workload_desc(sp), "l2": "inputs larger than L2 (not flushed)",
                   "parallelism": f"{world} independent subgraph(s), one per GPU",
                   "generator": "hgsynth.device: the workload recipe drawn on the GPU (seeded)",
                   "objective": ("L_BCE over the labelled users + 0.1 L_CCA (head: MeanAgg, 2-layer MLP)"
                                 if use_head else "synthetic upstream gradient + 0.1 L_CCA")},
        "roofline": rf, "kernel_rooflines": kernel_rooflines, "kernel_time_share": shares,
        "phases_ms": res["phases_ms"],
        "layers_fwd_bwd_edges_per_s": res["layers_fwd_bwd_edges_per_s"],
        "layer_stack_roofline": head["layer_stack_roofline"],
        "csr_build_edges_per_s": res["csr_build_edges_per_s"],
        "cpu_baseline": cpu, "e2e": res.get("e2e"), "clocks": res["clocks"], "workloads": extra,
        "overlap_build": build, "temporal": temporal, "hgt": hgt, "fused_layer": fused,
        "gpu_launches": int(sum(n for n, _ in res["report"].values())),
        "loss": res["loss"], "head_loss": res["head_loss"],
    }
    print(json.dumps(out))
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
