"""The bounded-wait path of the tensor-core kernels: a wait that runs out is recorded in the
library's device status word, reported once by hg_device_status (HG_ERR_TIMEOUT) and cleared, and
the context stays usable.  The wait is made to run out in the library's self-test kernel (an
mbarrier that nothing arrives at, with no copy, store or MMA in flight), never in a real kernel."""
import ctypes

import pytest
import torch

import hgsynth
import oracle
from tests.gpu_util import dev, grad_bufs, host, layer_params, lib, need_gpu, relerr

pytestmark = pytest.mark.gpu


def test_a_wait_that_runs_out_is_reported_once_and_the_context_stays_usable():
    need_gpu()
    hg = lib()
    so = hg.lib()
    assert hg.hg_device_status() == 0
    hg.hg_selftest_bounded_wait(1000)
    flags = ctypes.c_int32(0)
    assert so.hg_device_status(ctypes.byref(flags)) == 6  # HG_ERR_TIMEOUT
    assert flags.value == 1
    assert b"gave up" in so.hg_last_error()
    assert hg.hg_device_status() == 0  # reported once, then cleared
    # the same context runs a layer that still matches the oracle
    sp = hgsynth.spec("tiny-10k", n_user=2_000, n_risk=300, num_edges=20_000, n_overlap=100)
    w = hgsynth.make_workload(sp, random_affine=True, with_ids=False)
    g, p = w.graph, w.params[0]
    G = hg.hg_build_csr(dev(g["src"]), dev(g["dst"]), dev(g["rel"]), g["type_offsets"], g["rels"])
    P = layer_params(hg, p, sp.dtype)
    sb, kb = hg.hg_layer_workspace_size(G, P)
    saved = torch.empty(sb, dtype=torch.uint8, device="cuda")
    scratch = torch.empty(kb, dtype=torch.uint8, device="cuda")
    X = dev(w.X, torch.float32)
    out = torch.empty_like(X)
    hg.hg_layer_fwd(G, P, X, out, saved, scratch)
    dX = torch.empty_like(X)
    grads = grad_bufs(len(g["rels"]), 2, sp.d)
    hg.hg_layer_bwd(G, P, X, saved, dev(w.dH_top, torch.float32), dX, grads, scratch)
    torch.cuda.synchronize()
    csr = oracle.build_csr(g["src"], g["dst"], g["rel"], g["type_offsets"], g["rels"])
    ref, _ = oracle.layer_forward(csr, g["type_offsets"], g["rels"], p, w.X)
    dref, _ = oracle.layer_backward(csr, g["type_offsets"], g["rels"], p, w.X, w.dH_top)
    assert relerr(host(out), ref) <= 1e-5 and relerr(host(dX), dref) <= 1e-5
    assert hg.hg_device_status() == 0
