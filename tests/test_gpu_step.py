"""A whole step (CSR build, 2 layers forward for two live views, alignment loss and gradient,
2 layers backward for both views) on the 10k-node fp32 workload against the oracle's step."""
import numpy as np
import pytest
import torch

import hgsynth
import oracle
from tests.gpu_util import BF16_RELU_MARGIN, TOL, dev, host, lib, need_gpu, relerr, tdtype

pytestmark = pytest.mark.gpu


def make_path(w, head=None):
    from paper_2608_02168_gb300.step import HotPath
    sp, g = w.spec, w.graph
    return HotPath(g["type_offsets"], g["rels"], len(g["src"]), sp.d, sp.dtype, w.params, view=sp.view_b,
                   n_overlap_max=len(w.overlap_local),
                   n_gid_a=0 if w.gid_a is None else len(w.gid_a), n_gid_b=0 if w.gid_b is None else len(w.gid_b),
                   head_params=None if head is None else head["params"],
                   n_lab_max=0 if head is None else len(head["lab_idx"]))


def run(path, w, head=None):
    g, td = w.graph, tdtype(w.spec.dtype)
    kw = {}
    if w.spec.view_b == "perturbed":
        kw = dict(X_b=dev(w.X_b, td), overlap_idx=dev(w.overlap_local))
    else:
        kw = dict(gid_a=dev(w.gid_a), gid_b=dev(w.gid_b), H_bank=dev(w.H_b, td))
    if head is not None:
        kw.update(lab_idx=dev(head["lab_idx"]), lab_y=dev(head["lab_y"]))
    path.step(dev(g["src"]), dev(g["dst"]), dev(g["rel"]), dev(w.X, td), dev(w.dH_top, td), **kw)
    torch.cuda.synchronize()


@pytest.mark.parametrize("variant,with_head", [("tiny-10k", False), ("sub-small-bank", False), ("tiny-10k", True),
                                               ("sub-small-bank", True)])
def test_step_matches_oracle(variant, with_head):
    need_gpu()
    lib()
    if variant == "tiny-10k":
        sp = hgsynth.spec("tiny-10k")
    else:
        sp = hgsynth.spec("sub-1m", n_user=18_000, n_risk=2_000, num_edges=300_000, n_overlap=2_609)
    # bf16: wide bias margins keep the ReLU decisions of the layers and the head unambiguous (see
    # test_gpu_layer); the comparison is with the plain fp64 definition
    bf = sp.dtype == "bf16"
    w = hgsynth.make_workload(sp, random_affine=True, bias_margin=BF16_RELU_MARGIN if bf else None)
    head = None
    if with_head:
        lab, y = hgsynth.make_labels(sp, positive_rate=0.3)
        head = {"params": hgsynth.make_head_params(sp, random_bias=True, bias_margin=BF16_RELU_MARGIN if bf else None),
                "lab_idx": lab, "lab_y": y}
    path = make_path(w, head)
    run(path, w, head)
    vb = {"idx": w.overlap_local, "X_b": w.X_b} if sp.view_b == "perturbed" else \
        {"H_b": w.H_b, "gid_a": w.gid_a, "gid_b": w.gid_b}
    # the plain fp64 definition; the layer outputs and their gradients are bf16 tensors of the
    # interface for a bf16 workload, so the oracle rounds them there (and nowhere else)
    ref = oracle.step(w.graph, w.X, w.params, w.dH_top, vb, head=head, interface=sp.dtype)
    tol = TOL[sp.dtype]
    assert relerr(host(path.loss), np.array(ref["loss"])) <= (1e-4 if sp.dtype == "f32" else 2e-2)
    if with_head:
        assert relerr(host(path.head_loss), np.array(ref["head_loss"])) <= (1e-5 if sp.dtype == "f32" else 1e-3)
        for k in ("W1", "b1", "w2", "b2"):
            got, want = host(path.head_grads[k]), ref["head_grads"]["d" + k]
            assert relerr(got.reshape(want.shape), want) <= tol, (k, relerr(got.reshape(want.shape), want))
    for l in range(1, sp.layers + 1):
        assert relerr(host(path.H[0][l]), ref["H"][l]) <= tol, ("H", l)
    assert relerr(host(path.dH[0][0]), ref["dX"]) <= tol, relerr(host(path.dH[0][0]), ref["dX"])
    for l in range(sp.layers):
        for k, v in ref["grads"][l].items():
            assert relerr(host(path.grads[0][l][k]), v) <= tol, (l, k, relerr(host(path.grads[0][l][k]), v))
    if sp.view_b == "perturbed":
        assert relerr(host(path.dH[1][0]), ref["dX_b"]) <= tol
        for l in range(sp.layers):
            for k, v in ref["grads_b"][l].items():
                assert relerr(host(path.grads[1][l][k]), v) <= tol, ("b", l, k)
    else:
        n = int(path.n_dev.item())
        assert n == len(ref["idx_a"]) == sp.n_overlap
        assert np.array_equal(path.idx_a[:n].cpu().numpy(), ref["idx_a"])
        assert np.array_equal(path.idx_b[:n].cpu().numpy(), ref["idx_b"])


def test_step_is_bitwise_repeatable():
    need_gpu()
    lib()
    w = hgsynth.make_workload(hgsynth.spec("tiny-10k"), random_affine=True)
    path = make_path(w)
    run(path, w)
    first = [t.clone() for t in (path.loss, path.H[0][2], path.dH[0][0], path.dH[1][0])] + \
        [v.clone() for v in path.grads[0][0].values()]
    run(path, w)
    again = [path.loss, path.H[0][2], path.dH[0][0], path.dH[1][0]] + list(path.grads[0][0].values())
    for a, b in zip(first, again):
        assert torch.equal(a, b)
