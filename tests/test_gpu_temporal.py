"""Temporal module (context attention, Eq. 12; GRU cell, Eq. 13) through the C ABI against the oracle.

bf16 with d <= 128 and (w + 1) d <= 512 runs the tensor-core kernels (ragged last tiles, w from 1 to
the largest the tensor memory holds); fp32, d = 256 and larger windows run the CUDA-core path."""
import math

import numpy as np
import pytest
import torch

from oracle import temporal as OT
from tests.gpu_util import TOL, dev, host, lib, need_gpu, relerr, tdtype
from hgsynth import bf16_round

pytestmark = pytest.mark.gpu

KEYS = ("Wa", "r", "W_i", "W_h", "b_i", "b_h")


def problem(seed, n, d, w, dt):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((n, d)).astype(np.float32)
    C = rng.standard_normal((w, n, d)).astype(np.float32)
    a = math.sqrt(6 / (2 * d))
    k = 1 / math.sqrt(d)
    p = {"Wa": rng.uniform(-a, a, (d, d)), "r": rng.standard_normal(d) / math.sqrt(d) * 2,
         "W_i": rng.uniform(-k, k, (d, 3 * d)), "W_h": rng.uniform(-k, k, (d, 3 * d)),
         "b_i": rng.uniform(-k, k, 3 * d), "b_h": rng.uniform(-k, k, 3 * d)}
    p = {key: v.astype(np.float32) for key, v in p.items()}
    if dt == "bf16":
        X, C = bf16_round(X), bf16_round(C)
        p = {key: bf16_round(v) for key, v in p.items()}
    return X, C, p


def temporal_gpu(hg, X, C, p, dOut, dt, w):
    td = tdtype(dt)
    n, d = X.shape
    prm = hg.TemporalParams(*(dev(p[k], td) for k in KEYS), w=w)
    s, k = hg.hg_temporal_workspace_size(n, d, w, td)
    saved = torch.empty(s, dtype=torch.uint8, device="cuda")
    scratch = torch.empty(k, dtype=torch.uint8, device="cuda")
    Xd, Cd = dev(X, td), dev(C, td)
    out = torch.full((n, d), float("nan"), dtype=td, device="cuda")
    hg.hg_temporal_fwd(prm, Xd, Cd, out, saved, scratch)
    f = dict(dtype=torch.float32, device="cuda")
    grads = {"Wa": torch.full((d, d), np.nan, **f), "r": torch.full((d,), np.nan, **f),
             "W_i": torch.full((d, 3 * d), np.nan, **f), "W_h": torch.full((d, 3 * d), np.nan, **f),
             "b_i": torch.full((3 * d,), np.nan, **f), "b_h": torch.full((3 * d,), np.nan, **f)}
    dX = torch.full((n, d), float("nan"), dtype=td, device="cuda")
    hg.hg_temporal_bwd(prm, Xd, Cd, saved, dev(dOut, td), dX, grads, scratch)
    torch.cuda.synchronize()
    return host(out), host(dX), {k: host(v) for k, v in grads.items()}


def check(X, C, p, dOut, dt, got_out, got_dX, got_g):
    ref = OT.temporal_backward(X, C, p, dOut)  # the plain fp64 definition (Eq. 12-13)
    tol = TOL[dt]
    assert relerr(got_out, ref["out"]) <= tol, ("out", relerr(got_out, ref["out"]))
    assert relerr(got_dX, ref["dX"]) <= tol, ("dX", relerr(got_dX, ref["dX"]))
    for k in KEYS:
        assert relerr(got_g[k], ref["d" + k]) <= tol, (k, relerr(got_g[k], ref["d" + k]))


@pytest.mark.parametrize("dt,d,n,w", [("f32", 64, 1000, 3), ("f32", 128, 777, 2), ("bf16", 128, 5000, 3),
                                      ("bf16", 64, 3001, 4), ("bf16", 256, 1500, 3), ("f32", 256, 300, 1),
                                      ("bf16", 128, 129, 1), ("bf16", 64, 200, 7), ("bf16", 128, 700, 4)])
def test_temporal_matches_oracle(dt, d, n, w):
    need_gpu()
    hg = lib()
    X, C, p = problem(d + n + w, n, d, w, dt)
    dOut = np.random.default_rng(n).standard_normal((n, d)).astype(np.float32)
    if dt == "bf16":
        dOut = bf16_round(dOut)
    out, dX, g = temporal_gpu(hg, X, C, p, dOut, dt, w)
    check(X, C, p, dOut, dt, out, dX, g)


def test_temporal_empty_and_deterministic():
    need_gpu()
    hg = lib()
    X, C, p = problem(3, 0, 64, 3, "f32")
    out, dX, g = temporal_gpu(hg, X, C, p, np.zeros((0, 64), np.float32), "f32", 3)
    for k in KEYS:
        assert np.all(g[k] == 0), k
    X, C, p = problem(4, 4000, 128, 3, "bf16")
    dOut = bf16_round(np.random.default_rng(5).standard_normal((4000, 128)).astype(np.float32))
    a = temporal_gpu(hg, X, C, p, dOut, "bf16", 3)
    b = temporal_gpu(hg, X, C, p, dOut, "bf16", 3)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
    for k in KEYS:
        assert np.array_equal(a[2][k], b[2][k]), k
