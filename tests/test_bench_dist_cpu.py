"""The multi-GPU harness of bench.py on CPU: two gloo ranks on 127.0.0.1 (world size 2).

Each rank works on its own subgraph (weak scaling, no collective on the data path); the timed
region is bracketed by barriers, its duration is the maximum over the ranks, and the reported value
counts every rank's units over that duration.  The reference arm runs on rank 0 only."""
import json
import os
import socket
import subprocess
import sys

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def rank_main(rank: int, world: int, port: int, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import bench
    import hgsynth
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench.rank_barrier(world)
        # a slower second rank: both ranks must report the slower one's time
        t = bench.max_time_over_ranks(0.25 * (rank + 1), world, "cpu")
        sp = hgsynth.spec("tiny-10k", n_user=800, n_risk=200, num_edges=5_000, n_overlap=50)
        w = hgsynth.make_workload(sp, sub=rank)
        sig = (int(w.graph["src"].astype(np.int64).sum()), int(w.graph["dst"].astype(np.int64).sum()),
               float(w.X.sum()))
        sigs = [None] * world
        dist.all_gather_object(sigs, sig)
        value = bench.weak_scaling_value(world, sp.layers * sp.num_edges, 3, t)
        bench.rank_barrier(world)
        out.put((rank, t, sigs, value, sp.layers * sp.num_edges))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_harness():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = free_port()
    procs = [ctx.Process(target=rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = [q.get(timeout=240) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    res.sort()
    for rank, t, sigs, value, units in res:
        assert t == 0.5  # the maximum over the ranks, seen by every rank
        assert sigs[0] != sigs[1]  # each rank has its own subgraph (sub = rank)
        assert value == 2 * units * 3 / 0.5  # all ranks' units over the slowest rank's time


def test_reference_arm_only_on_rank_zero():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1", CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny-10k",
                        "--steps", "1", "--warmup", "0"], capture_output=True, text=True, env=env, timeout=300)
    assert r.returncode == 0 and r.stdout.strip() == ""
    env.update(RANK="0", LOCAL_RANK="0")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny-10k",
                        "--steps", "1", "--warmup", "0"], capture_output=True, text=True, env=env, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    line = json.loads(r.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["value"] > 0 and line["e2e"]["h2d_bytes_per_step"] == 0
    assert line["cpu_baseline"]["kind"] == "oracle"


def test_bench_generator_references_exist():
    """Every hgsynth name bench.py uses exists (the bench runs only on a GPU machine)."""
    import ast
    import hgsynth
    src = open(os.path.join(ROOT, "bench.py")).read()
    names = {n.attr for n in ast.walk(ast.parse(src))
             if isinstance(n, ast.Attribute) and isinstance(n.value, ast.Name) and n.value.id == "hgsynth"}
    assert names and all(hasattr(hgsynth, n) for n in names), sorted(n for n in names if not hasattr(hgsynth, n))
