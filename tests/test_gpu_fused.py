"""The fused mean layer (hg_layer_params.fused): the relation means of rows with at most 32 runs are
summed inside the projection and never stored, and summed again for the weight gradient.  Its
results must equal the unfused layer's bit for bit (the same sums in the same order) and the plain
definition (Eq. 7, 10, 11 in fp64) within the bf16 tolerance, on graphs whose rows span every path:
no in-edges, short rows, rows above 32 runs and hub rows above 512 runs."""
import numpy as np
import pytest
import torch

import hgsynth
import oracle
from tests.gpu_util import BF16_RELU_MARGIN, TOL, dev, grad_bufs, host, layer_params, lib, need_gpu, relerr, tdtype

pytestmark = pytest.mark.gpu

CASES = {
    # power-law in-degrees with hub rows; a second shape with a ragged last tile of each type
    "sub-d128": ("sub-1m", dict(n_user=27_001, n_risk=3_003, num_edges=600_000, n_overlap=4_000)),
    "tail-d128": ("tail-5m", dict(n_user=9_007, n_risk=1_001, num_edges=200_000, n_overlap=1_000, out_cap=4_000,
                                 d=128, dtype="bf16")),
    # enough stored rows per relation that the weight gradient's split-K partition has several
    # 64-row chunks per split
    "mid-d128": ("sub-1m", dict(n_user=200_003, n_risk=20_011, num_edges=2_000_000, n_overlap=4_000)),
}


def run(hg, w, p, act, ln, fused):
    g = w.graph
    G = hg.hg_build_csr(dev(g["src"]), dev(g["dst"]), dev(g["rel"]), g["type_offsets"], g["rels"])
    P = layer_params(hg, p, "bf16", act, ln, fused=fused)
    sb, kb = hg.hg_layer_workspace_size(G, P)
    saved = torch.empty(sb, dtype=torch.uint8, device="cuda")
    scratch = torch.empty(kb, dtype=torch.uint8, device="cuda")
    X = dev(w.X, torch.bfloat16)
    out = torch.empty_like(X)
    hg.hg_layer_fwd(G, P, X, out, saved, scratch)
    dH_in = torch.empty_like(X)
    grads = grad_bufs(len(g["rels"]), len(g["type_offsets"]) - 1, 128)
    hg.hg_layer_bwd(G, P, X, saved, dev(w.dH_top, torch.bfloat16), dH_in, grads, scratch)
    torch.cuda.synchronize()
    return out, dH_in, grads, sb


def run_lengths(csr, rels):
    """Runs of equal source ids per CSR row, over all relations (the aggregation lists)."""
    out = []
    for r in range(len(rels)):
        ptr, col = csr[r]["row_ptr"], csr[r]["col"]
        for j in range(len(ptr) - 1):
            c = col[ptr[j]:ptr[j + 1]]
            out.append(int(np.count_nonzero(np.diff(c)) + 1) if len(c) else 0)
    return np.asarray(out)


@pytest.mark.parametrize("case", list(CASES))
@pytest.mark.parametrize("act,ln", [("relu", True), ("gelu_tanh", True), ("relu", False)])
def test_fused_layer_equals_unfused_and_definition(case, act, ln):
    need_gpu()
    if case != "sub-d128" and (act, ln) != ("relu", True):
        pytest.skip("activation variants covered on one shape")
    hg = lib()
    name, ov = CASES[case]
    sp = hgsynth.spec(name, **{**ov, "dtype": "bf16", "d": 128})
    margin = BF16_RELU_MARGIN if act == "relu" else None
    w = hgsynth.make_workload(sp, random_affine=True, with_ids=False, bias_margin=margin)
    g, p = w.graph, w.params[0]
    csr = oracle.build_csr(g["src"], g["dst"], g["rel"], g["type_offsets"], g["rels"])
    runs = run_lengths(csr, g["rels"])
    # every producer path is taken: empty rows, streamed rows, long rows, hub rows
    assert (runs == 0).any() and ((runs > 0) & (runs <= 32)).any() and (runs > 32).any()
    if case != "tail-d128":
        assert (runs > 512).any()
    if case == "mid-d128":
        nnz = [int(np.count_nonzero(np.diff(csr[r]["row_ptr"]))) for r in range(len(g["rels"]))]
        assert max(nnz) > 152 * 64 * 2, nnz
    o0, d0, g0, s0 = run(hg, w, p, act, ln, False)
    o1, d1, g1, s1 = run(hg, w, p, act, ln, True)
    assert s1 < s0  # no stored means for the short rows
    bad = (o0.view(torch.int16) != o1.view(torch.int16)).any(dim=1)
    assert not bad.any(), ("H_out differs from the unfused layer", int(bad.sum()), bad.nonzero()[:8].flatten().tolist())
    assert torch.equal(d0.view(torch.int16), d1.view(torch.int16)), "dH_in differs from the unfused layer"
    keys = ("W_rel", "W_agg", "b_agg") + (("ln_gamma", "ln_beta") if ln else ())
    for k in keys:
        assert torch.equal(g0[k], g1[k]), f"d{k} differs from the unfused layer"
    ref, _ = oracle.layer_forward(csr, g["type_offsets"], g["rels"], p, w.X, act, ln)
    tol = TOL["bf16"]
    assert relerr(host(o1), ref) <= tol, ("H_out", relerr(host(o1), ref))
    dref, gref = oracle.layer_backward(csr, g["type_offsets"], g["rels"], p, w.X, w.dH_top, act, ln)
    assert relerr(host(d1), dref) <= tol, ("dH_in", relerr(host(d1), dref))
    for k in keys:
        e = relerr(host(g1[k]), gref[k])
        assert e <= tol, (k, e)
    assert hg.hg_device_status() == 0


def test_fused_layer_without_edges():
    need_gpu()
    hg = lib()
    sp = hgsynth.spec("tiny-10k", n_user=700, n_risk=90, num_edges=0, n_overlap=50, dtype="bf16", d=128)
    w = hgsynth.make_workload(sp, random_affine=True, with_ids=False, bias_margin=BF16_RELU_MARGIN)
    o0, d0, g0, _ = run(hg, w, w.params[0], "relu", True, False)
    o1, d1, g1, _ = run(hg, w, w.params[0], "relu", True, True)
    assert torch.equal(o0.view(torch.int16), o1.view(torch.int16))
    assert torch.equal(d0.view(torch.int16), d1.view(torch.int16))
    for k in ("W_rel", "W_agg", "b_agg", "ln_gamma", "ln_beta"):
        assert torch.equal(g0[k], g1[k]), k


@pytest.mark.parametrize("dt,d", [("f32", 128), ("bf16", 64), ("bf16", 256)])
def test_fused_layer_rejects_other_shapes(dt, d):
    need_gpu()
    hg = lib()
    sp = hgsynth.spec("tiny-10k", dtype=dt, d=d)
    w = hgsynth.make_workload(sp, random_affine=True, with_ids=False)
    g = w.graph
    G = hg.hg_build_csr(dev(g["src"]), dev(g["dst"]), dev(g["rel"]), g["type_offsets"], g["rels"])
    P = layer_params(hg, w.params[0], dt, fused=True)
    with pytest.raises(Exception, match="unsupported"):
        hg.hg_layer_workspace_size(G, P)
