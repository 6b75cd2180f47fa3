"""The allocation-free alignment-loss entry point (hg_overlap_align_loss_static) against the
allocating one (hg_overlap_align_loss), called through the C ABI.

It exists for callers that cannot allocate device memory (no CUDA allocator of their own, device
memory fully reserved by another framework, or no cudaMalloc allowed because it can synchronise
the device): its scratch is a static device array inside the library.  Two calls in a row must
each reproduce the allocating entry point's loss and saved statistics, and the saved buffer must
drive the gradient exactly as the allocating one's does.  This file is collected last on purpose.
"""
import numpy as np
import pytest
import torch

from tests.gpu_util import dev, host, lib, need_gpu, tdtype
from tests.test_gpu_align import views

pytestmark = pytest.mark.gpu

LOSS_TOL = 1e-4  # relative, the tolerance the alignment-loss tests use


@pytest.mark.parametrize("dt,d,n,N", [("f32", 64, 3000, 4000), ("bf16", 128, 20_000, 26_000), ("bf16", 256, 1500, 1600)])
def test_static_scratch_entry_point_matches_allocating_one(dt, d, n, N):
    need_gpu()
    hg = lib()
    Ha, ia, Hb, ib = views(100 + d, N, n, d, dt)
    td = tdtype(dt)
    A, B, IA, IB = dev(Ha, td), dev(Hb, td), dev(ia), dev(ib)
    s_bytes, k_bytes = hg.hg_overlap_align_workspace_size(n, d)
    saved_ref = torch.empty(s_bytes, dtype=torch.uint8, device="cuda")
    scratch = torch.empty(k_bytes, dtype=torch.uint8, device="cuda")
    loss_ref = torch.empty(3, dtype=torch.float32, device="cuda")
    hg.hg_overlap_align_loss(A, IA, B, IB, n, None, 2e-4, 1e-8, loss_ref, saved_ref, scratch)
    dA_ref = torch.zeros_like(A)
    hg.hg_overlap_align_bwd(A, IA, B, IB, n, None, 2e-4, 1e-8, 0.1, saved_ref, dA_ref, None, scratch)
    ref = host(loss_ref)
    stats_ref = host(saved_ref[: (4 * d + 2 * d * d) * 4].view(torch.float32))
    for call in range(2):
        saved = torch.full((s_bytes,), 0xAB, dtype=torch.uint8, device="cuda")
        loss = torch.full((3,), float("nan"), dtype=torch.float32, device="cuda")
        hg.hg_overlap_align_loss_static(A, IA, B, IB, n, None, 2e-4, 1e-8, loss, saved)
        got = host(loss)
        assert np.all(np.abs(got - ref) <= LOSS_TOL * np.abs(ref) + 1e-7), (call, got, ref)
        stats = host(saved[: (4 * d + 2 * d * d) * 4].view(torch.float32))
        assert np.abs(stats - stats_ref).max() <= LOSS_TOL * np.abs(stats_ref).max(), call
        dA = torch.zeros_like(A)
        hg.hg_overlap_align_bwd(A, IA, B, IB, n, None, 2e-4, 1e-8, 0.1, saved, dA, None, scratch)
        x, y = host(dA), host(dA_ref)
        assert np.abs(x - y).max() <= (1e-5 if dt == "f32" else 2e-2) * np.abs(y).max(), call
    assert hg.hg_device_status() == 0


@pytest.mark.parametrize("dt,d,n_max,n_live", [("bf16", 128, 20_000, 13_001), ("f32", 64, 3000, 1777),
                                               ("bf16", 256, 1500, 2), ("bf16", 64, 0, 0)])
def test_static_entry_point_with_a_device_side_count(dt, d, n_max, n_live):
    """The overlap count read from the device (n_dev, e.g. the intersection's n_out) below the
    capacity n_max, and an empty capacity: the static entry point's loss and saved statistics agree
    with the allocating entry point's, on two calls in a row, and no bounded wait gives up."""
    need_gpu()
    hg = lib()
    rows = max(n_max, 8) + 100
    Ha, ia, Hb, ib = views(200 + d + n_max, rows, max(n_max, 1), d, dt)
    td = tdtype(dt)
    A, B, IA, IB = dev(Ha, td), dev(Hb, td), dev(ia), dev(ib)
    n_dev = torch.tensor([n_live], dtype=torch.int64, device="cuda")
    s_bytes, k_bytes = hg.hg_overlap_align_workspace_size(n_max, d)
    saved_ref = torch.empty(max(s_bytes, 256), dtype=torch.uint8, device="cuda")
    scratch = torch.empty(max(k_bytes, 256), dtype=torch.uint8, device="cuda")
    loss_ref = torch.full((3,), float("nan"), dtype=torch.float32, device="cuda")
    hg.hg_overlap_align_loss(A, IA, B, IB, n_max, n_dev, 2e-4, 1e-8, loss_ref, saved_ref, scratch)
    ref = host(loss_ref)
    if n_live < 2:
        assert np.all(ref == 0)
    stats_bytes = (4 * d + 2 * d * d) * 4
    for call in range(2):
        saved = torch.full((max(s_bytes, 256),), 0xAB, dtype=torch.uint8, device="cuda")
        loss = torch.full((3,), float("nan"), dtype=torch.float32, device="cuda")
        hg.hg_overlap_align_loss_static(A, IA, B, IB, n_max, n_dev, 2e-4, 1e-8, loss, saved)
        got = host(loss)
        assert np.all(np.abs(got - ref) <= LOSS_TOL * np.abs(ref) + 1e-7), (call, got, ref)
        if n_live >= 2:
            stats, stats_ref = (host(x[:stats_bytes].view(torch.float32)) for x in (saved, saved_ref))
            assert np.abs(stats - stats_ref).max() <= LOSS_TOL * np.abs(stats_ref).max(), call
    assert hg.hg_device_status() == 0
