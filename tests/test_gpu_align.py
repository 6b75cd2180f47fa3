"""Overlap intersection (bit-exact) and the alignment loss / gradient against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from tests.gpu_util import TOL, dev, host, lib, need_gpu, relerr, tdtype
from hgsynth import bf16_round

pytestmark = pytest.mark.gpu


def intersect_gpu(hg, a, b):
    idx_a = torch.empty(max(1, min(len(a), len(b))), dtype=torch.int32, device="cuda")
    idx_b = torch.empty_like(idx_a)
    n = torch.zeros(1, dtype=torch.int64, device="cuda")
    scratch = torch.empty(hg.hg_overlap_intersect_workspace_size(len(a), len(b)), dtype=torch.uint8, device="cuda")
    hg.hg_overlap_intersect(dev(a, torch.int64), dev(b, torch.int64), idx_a, idx_b, n, scratch)
    k = int(n.item())
    return k, idx_a[:max(k, 0)].cpu().numpy(), idx_b[:max(k, 0)].cpu().numpy()


@pytest.mark.parametrize("na,nb", [(1000, 3000), (200_000, 150_000), (5, 0), (1, 1)])
def test_intersect_bit_exact(na, nb):
    need_gpu()
    hg = lib()
    rng = np.random.default_rng(na + nb)
    space = 4 * max(na, nb, 1)
    a = np.sort(rng.choice(space, na, replace=False)).astype(np.int64)
    b = np.sort(rng.choice(space, nb, replace=False)).astype(np.int64)
    k, ia, ib = intersect_gpu(hg, a, b)
    ra, rb = oracle.overlap_intersect(a, b)
    assert k == len(ra)
    assert np.array_equal(ia, ra) and np.array_equal(ib, rb)


def test_intersect_flags_unsorted_input():
    need_gpu()
    hg = lib()
    k, _, _ = intersect_gpu(hg, np.array([1, 5, 3, 9], np.int64), np.array([3, 5], np.int64))
    assert k == -1
    k, _, _ = intersect_gpu(hg, np.array([1, 5, 9], np.int64), np.array([5, 5, 9], np.int64))
    assert k == -1


def views(seed, N, n, d, dt):
    rng = np.random.default_rng(seed)
    Ha = (rng.standard_normal((N, d)) * rng.uniform(0.5, 2, d) + rng.uniform(-1, 1, d)).astype(np.float32)
    Hb = (0.7 * Ha + 0.5 * rng.standard_normal((N, d))).astype(np.float32)[rng.permutation(N)]
    if dt == "bf16":
        Ha, Hb = bf16_round(Ha), bf16_round(Hb)
    ia = np.sort(rng.choice(N, n, replace=False)).astype(np.int32)
    ib = rng.permutation(rng.choice(N, n, replace=False)).astype(np.int32)
    return Ha, ia, Hb, ib


def align_gpu(hg, Ha, ia, Hb, ib, dt, lam, eps, dloss, n_dev_val=None, both=True, n_max=None, base=0.0):
    td = tdtype(dt)
    d = Ha.shape[1]
    n_max = len(ia) if n_max is None else n_max
    s, k = hg.hg_overlap_align_workspace_size(n_max, d)
    saved = torch.empty(s, dtype=torch.uint8, device="cuda")
    scratch = torch.empty(k, dtype=torch.uint8, device="cuda")
    loss = torch.empty(3, dtype=torch.float32, device="cuda")
    A, B = dev(Ha, td), dev(Hb, td)
    IA = torch.zeros(n_max, dtype=torch.int32, device="cuda")
    IB = torch.zeros(n_max, dtype=torch.int32, device="cuda")
    IA[:len(ia)] = dev(ia)
    IB[:len(ib)] = dev(ib)
    n_dev = None if n_dev_val is None else torch.tensor([n_dev_val], dtype=torch.int64, device="cuda")
    hg.hg_overlap_align_loss(A, IA, B, IB, n_max, n_dev, lam, eps, loss, saved, scratch)
    base_a = base * torch.randn_like(A)
    base_b = base * torch.randn_like(B)
    dA, dB = base_a.clone(), base_b.clone()
    hg.hg_overlap_align_bwd(A, IA, B, IB, n_max, n_dev, lam, eps, dloss, saved, dA, dB if both else None, scratch)
    torch.cuda.synchronize()
    return host(loss), host(dA) - host(base_a), host(dB) - host(base_b), dB, base_b


@pytest.mark.parametrize("dt,d,n,N", [("f32", 64, 1000, 1300), ("bf16", 128, 5000, 7000), ("bf16", 256, 3000, 3100),
                                      ("bf16", 64, 2001, 2600), ("f32", 128, 70_001, 80_000)])
def test_align_matches_oracle(dt, d, n, N):
    need_gpu()
    hg = lib()
    Ha, ia, Hb, ib = views(d + n, N, n, d, dt)
    lam, eps, dloss = 2e-4, 1e-8, 0.1
    loss, gA, gB, _, _ = align_gpu(hg, Ha, ia, Hb, ib, dt, lam, eps, dloss)
    ref = oracle.align_forward(Ha, ia, Hb, ib, lam, eps)
    assert relerr(loss, ref) <= 1e-4, (loss, ref)
    rA, rB = oracle.align_backward(Ha, ia, Hb, ib, lam, eps, dloss)
    tol = TOL[dt]
    assert relerr(gA[ia], rA[ia]) <= tol, relerr(gA[ia], rA[ia])
    assert relerr(gB[ib], rB[ib]) <= tol, relerr(gB[ib], rB[ib])
    others = np.setdiff1d(np.arange(N), ia)
    assert np.abs(gA[others]).max() == 0


def test_align_fp32_tight_gradient():
    """fp32 storage: the gradient itself within 1e-5 (no bf16 accumulation)."""
    need_gpu()
    hg = lib()
    Ha, ia, Hb, ib = views(7, 4000, 3500, 64, "f32")
    td = torch.float32
    s, k = hg.hg_overlap_align_workspace_size(len(ia), 64)
    saved = torch.empty(s, dtype=torch.uint8, device="cuda")
    scratch = torch.empty(k, dtype=torch.uint8, device="cuda")
    loss = torch.empty(3, dtype=torch.float32, device="cuda")
    A, B = dev(Ha, td), dev(Hb, td)
    hg.hg_overlap_align_loss(A, dev(ia), B, dev(ib), len(ia), None, 0.05, 1e-6, loss, saved, scratch)
    dA = torch.zeros_like(A)
    dB = torch.zeros_like(B)
    hg.hg_overlap_align_bwd(A, dev(ia), B, dev(ib), len(ia), None, 0.05, 1e-6, 1.0, saved, dA, dB, scratch)
    rA, rB = oracle.align_backward(Ha, ia, Hb, ib, 0.05, 1e-6, 1.0)
    assert relerr(host(dA), rA) <= 1e-5 and relerr(host(dB), rB) <= 1e-5


def test_align_device_count_detached_view_and_degenerate_sizes():
    need_gpu()
    hg = lib()
    Ha, ia, Hb, ib = views(11, 900, 600, 64, "f32")
    # capacity 600, actual count 450 read from the device
    loss, gA, gB, dB, base_b = align_gpu(hg, Ha, ia, Hb, ib, "f32", 2e-4, 1e-8, 1.0, n_dev_val=450, both=False,
                                         base=1.0)
    ref = oracle.align_forward(Ha, ia[:450], Hb, ib[:450], 2e-4, 1e-8)
    assert relerr(loss, ref) <= 1e-4
    rA, _ = oracle.align_backward(Ha, ia[:450], Hb, ib[:450], 2e-4, 1e-8, 1.0)
    # accumulated onto N(0,1) values: the increment is exact up to fp32 rounding of the sum
    assert np.abs(gA - rA).max() <= 1e-6 * 8 + 1e-5 * np.abs(rA).max()
    assert np.abs(gA[np.setdiff1d(np.arange(900), ia[:450])]).max() == 0
    assert torch.equal(dB, base_b)  # detached view untouched
    # n = 1 and n = 0: zero loss, zero gradient
    for n_val in (1, 0):
        loss, gA, gB, _, _ = align_gpu(hg, Ha, ia, Hb, ib, "f32", 2e-4, 1e-8, 1.0, n_dev_val=n_val)
        assert np.all(loss == 0) and np.abs(gA).max() == 0 and np.abs(gB).max() == 0
    # identical views: L_inv = 0
    loss, _, _, _, _ = align_gpu(hg, Ha, ia, Ha, ia, "f32", 2e-4, 1e-8, 1.0)
    assert abs(loss[1]) <= 1e-5 * 64


@pytest.mark.parametrize("d", [64, 128, 256])
def test_align_bf16_device_count_far_below_capacity(d):
    """bf16 path with the live row count read from the device and far below the capacity (the
    step passes one capacity for every subgraph): the row splits of the Gram products and the
    persistent gradient CTAs follow the device count; strong decorrelation (lambda = 0.05) makes
    the Z (C - I) term of the gradient visible."""
    need_gpu()
    hg = lib()
    n_live = 13_001 if d < 256 else 4_001
    Ha, ia, Hb, ib = views(300 + d, 3 * n_live, n_live, d, "bf16")
    lam, eps, dloss = 0.05, 1e-8, 0.5
    loss, gA, gB, _, _ = align_gpu(hg, Ha, ia, Hb, ib, "bf16", lam, eps, dloss, n_dev_val=n_live,
                                   n_max=5 * n_live, base=0.0)
    ref = oracle.align_forward(Ha, ia, Hb, ib, lam, eps)
    assert relerr(loss, ref) <= 1e-3, (loss, ref)
    rA, rB = oracle.align_backward(Ha, ia, Hb, ib, lam, eps, dloss)
    assert relerr(gA[ia], rA[ia]) <= TOL["bf16"], relerr(gA[ia], rA[ia])
    assert relerr(gB[ib], rB[ib]) <= TOL["bf16"], relerr(gB[ib], rB[ib])
    assert np.abs(gA[np.setdiff1d(np.arange(len(Ha)), ia)]).max() == 0
    assert hg.hg_device_status() == 0
