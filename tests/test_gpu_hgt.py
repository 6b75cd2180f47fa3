"""Attention layer (Heterogeneous Graph Transformer, Eq. 6-11) forward and backward through the C
ABI against the oracle, on seeded power-law graphs whose in- and out-degree hubs exceed the hub
degree (so the chunked paths of all three edge passes run), ragged type sizes and isolated nodes."""
import numpy as np
import pytest
import torch

import hgsynth
from oracle import hgt as OH
from tests.gpu_util import BF16_RELU_MARGIN, TOL, dev, host, lib, need_gpu, relerr, tdtype

pytestmark = pytest.mark.gpu

KEYS = ("W_K", "W_Q", "W_V", "b_K", "b_Q", "b_V", "W_att", "W_msg", "mu", "W_agg", "b_agg", "ln_gamma", "ln_beta")

CASES = {
    "tiny-f32-d64-h4": ("tiny-10k", {}, 4),
    "sub-bf16-d128-h4": ("sub-1m", dict(n_user=27_001, n_risk=3_003, num_edges=600_000, n_overlap=4_000), 4),
    "tiny-bf16-d64-h8": ("tiny-10k", dict(dtype="bf16"), 8),
    "sub-f32-d128-h1": ("sub-1m", dict(n_user=9_001, n_risk=1_003, num_edges=150_000, n_overlap=1_000, dtype="f32"), 1),
    "tail-bf16-d256-h4": ("tail-5m", dict(n_user=9_007, n_risk=1_001, num_edges=200_000, n_overlap=1_000,
                                          out_cap=4_000), 4),
}


def run_gpu(hg, w, p, heads, ln, dOut):
    sp, g = w.spec, w.graph
    td = tdtype(sp.dtype)
    G = hg.hg_build_csr(dev(g["src"]), dev(g["dst"]), dev(g["rel"]), g["type_offsets"], g["rels"])
    tens = {k: dev(p[k], torch.float32 if k == "mu" else td) for k in KEYS}
    P = hg.HgtParams(tens, heads, layernorm=ln)
    sb, kb = hg.hg_hgt_workspace_size(G, P)
    saved = torch.empty(sb, dtype=torch.uint8, device="cuda")
    scratch = torch.empty(kb, dtype=torch.uint8, device="cuda")
    X = dev(w.X, td)
    out = torch.empty_like(X)
    hg.hg_hgt_fwd(G, P, X, out, saved, scratch)
    dH = torch.empty_like(X)
    grads = {k: torch.full(np.shape(p[k]), np.nan, dtype=torch.float32, device="cuda") for k in KEYS}
    hg.hg_hgt_bwd(G, P, X, saved, dev(dOut, td), dH, grads, scratch)
    torch.cuda.synchronize()
    return host(out), host(dH), {k: host(v) for k, v in grads.items()}


@pytest.mark.parametrize("case", list(CASES))
@pytest.mark.parametrize("ln", [True, False])
def test_hgt_matches_oracle(case, ln):
    need_gpu()
    hg = lib()
    name, ov, heads = CASES[case]
    sp = hgsynth.spec(name, **ov)
    # bf16 ReLU: biases of +-8 keep the pre-activations clear of the kink (as for the mean layer)
    w = hgsynth.make_workload(sp, random_affine=True, with_ids=False)
    p = hgsynth.make_hgt_params(sp, heads, bias_margin=BF16_RELU_MARGIN if sp.dtype == "bf16" else None)
    g = w.graph
    out, dH, gr = run_gpu(hg, w, p, heads, ln, w.dH_top)
    args = (g["src"], g["dst"], g["rel"], g["type_offsets"], g["rels"], p, w.X)
    ref, _ = OH.hgt_forward(*args, heads, layernorm=ln)  # the plain fp64 definition (Eq. 6-11)
    tol = TOL[sp.dtype]
    assert relerr(out, ref) <= tol, ("H_out", relerr(out, ref))
    dref, gref = OH.hgt_backward(*args, w.dH_top, heads, layernorm=ln)
    assert relerr(dH, dref) <= tol, ("dH_in", relerr(dH, dref))
    for k in KEYS:
        if not ln and k in ("ln_gamma", "ln_beta"):
            continue
        e = relerr(gr[k], gref[k])
        assert e <= tol, (k, e)
    assert hg.hg_device_status() == 0


def test_hgt_is_bitwise_repeatable():
    need_gpu()
    hg = lib()
    name, ov, heads = CASES["sub-bf16-d128-h4"]
    sp = hgsynth.spec(name, **ov)
    w = hgsynth.make_workload(sp, random_affine=True, with_ids=False)
    p = hgsynth.make_hgt_params(sp, heads)
    a = run_gpu(hg, w, p, heads, True, w.dH_top)
    b = run_gpu(hg, w, p, heads, True, w.dH_top)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
    for k in KEYS:
        assert np.array_equal(a[2][k], b[2][k]), k
