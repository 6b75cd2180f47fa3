"""Prediction head and joint objective (MeanAgg, Eq. 18-20) through the C ABI against the oracle."""
import math

import numpy as np
import pytest
import torch

from oracle import head as OH
from tests.gpu_util import BF16_RELU_MARGIN, TOL, dev, host, lib, need_gpu, relerr, tdtype
from hgsynth import bf16_round

pytestmark = pytest.mark.gpu


def problem(seed, N, d, n_lab, n_rep, dt, rows_rep=None, frac_y=False):
    rng = np.random.default_rng(seed)
    rows_rep = rows_rep or N
    H = rng.standard_normal((N, d)).astype(np.float32)
    Hr = (0.6 * rng.standard_normal((rows_rep, d))).astype(np.float32)
    ia = np.sort(rng.choice(N, n_rep, replace=False)).astype(np.int32)
    ib = rng.choice(rows_rep, n_rep, replace=False).astype(np.int32)
    # labelled rows: half of them drawn among the overlap rows, so MeanAgg is exercised
    k = min(n_lab // 2, n_rep)
    lab = np.concatenate([rng.choice(ia, k, replace=False),
                          rng.choice(np.setdiff1d(np.arange(N), ia), n_lab - k, replace=False)])
    lab = rng.permutation(lab).astype(np.int32)
    y = rng.random(n_lab).astype(np.float32) if frac_y else (rng.random(n_lab) < 0.3).astype(np.float32)
    a1, a2 = math.sqrt(6 / (2 * d)), math.sqrt(6 / (d + 1))
    p = {"W1": rng.uniform(-a1, a1, (d, d)).astype(np.float32), "b1": (0.1 * rng.standard_normal(d)).astype(np.float32),
         "w2": rng.uniform(-a2, a2, d).astype(np.float32), "b2": np.array([0.3], np.float32)}
    if dt == "bf16":
        # hidden biases of +-8 keep every pre-activation clear of the ReLU's kink: the tensor cores'
        # fp32 accumulation may put a pre-activation within 1e-5 of zero on the other side, and each
        # such decision moves its row's input gradient by percents (rows are not sums over rows)
        p["b1"] = (BF16_RELU_MARGIN * rng.choice([-1.0, 1.0], d)).astype(np.float32)
        H, Hr = bf16_round(H), bf16_round(Hr)
        p = {key: bf16_round(v) for key, v in p.items()}
    return H, Hr, ia, ib, lab, y, p


def head_gpu(hg, H, Hr, ia, ib, lab, y, p, dt, dloss=1.0, cca=None, lam=0.1, n_rep_dev=None, both=True, base=0.0,
             with_dH=True, rep_cap=None):
    td = tdtype(dt)
    N, d = H.shape
    prm = hg.HeadParams(dev(p["W1"], td), dev(p["b1"], td), dev(p["w2"], td), dev(p["b2"], td))
    s, k = hg.hg_head_workspace_size(N, len(lab), d, td)
    saved = torch.empty(max(s, 1), dtype=torch.uint8, device="cuda")
    scratch = torch.empty(max(k, 1), dtype=torch.uint8, device="cuda")
    A, B = dev(H, td), dev(Hr, td)
    cap = rep_cap or max(len(ia), 1)
    IA = torch.zeros(cap, dtype=torch.int32, device="cuda")
    IB = torch.zeros(cap, dtype=torch.int32, device="cuda")
    IA[:len(ia)] = dev(ia)
    IB[:len(ib)] = dev(ib)
    nd = None if n_rep_dev is None else torch.tensor([n_rep_dev], dtype=torch.int64, device="cuda")
    L = dev(lab if len(lab) else np.zeros(0, np.int32))
    Y = dev(y if len(y) else np.zeros(0, np.float32))
    loss = torch.full((2,), np.nan, dtype=torch.float32, device="cuda")
    logits = torch.full((max(len(lab), 1),), np.nan, dtype=torch.float32, device="cuda")
    cca_t = None if cca is None else torch.tensor([cca], dtype=torch.float32, device="cuda")
    hg.hg_head_loss(prm, A, B, IA, IB, len(ia) if rep_cap is None else cap, nd, L, Y, cca_t, lam, loss, logits, saved,
                    scratch)
    f = dict(dtype=torch.float32, device="cuda")
    grads = {"W1": torch.full((d, d), np.nan, **f), "b1": torch.full((d,), np.nan, **f),
             "w2": torch.full((d,), np.nan, **f), "b2": torch.full((1,), np.nan, **f)}
    base_a = base * torch.randn_like(A)
    base_b = base * torch.randn_like(B)
    dH, dR = base_a.clone(), base_b.clone()
    hg.hg_head_bwd(prm, L, dloss, saved, dH if with_dH else None, dR if both else None, grads, scratch)
    torch.cuda.synchronize()
    return dict(loss=host(loss), logits=host(logits)[:len(lab)], dW1=host(grads["W1"]), db1=host(grads["b1"]),
                dw2=host(grads["w2"]), db2=host(grads["b2"]), dH=host(dH) - host(base_a), dH_rep=host(dR) - host(base_b),
                dR_t=dR, base_b=base_b)


def check(got, H, Hr, ia, ib, lab, y, p, dt, dloss=1.0, cca=None, lam=0.1, ltol=None):
    # the plain fp64 definition of Eq. 18-20 for both storage types
    ref = OH.head_loss(H, ia, Hr, ib, lab, y, p, cca_loss=cca, lambda_cca=lam)
    g = OH.head_backward(H, ia, Hr, ib, lab, y, p, dloss=dloss)
    ltol = ltol or (1e-5 if dt == "f32" else 1e-4)
    assert abs(got["loss"][1] - ref["bce"]) <= ltol * max(abs(ref["bce"]), 1e-6), (got["loss"], ref["bce"])
    assert abs(got["loss"][0] - ref["total"]) <= ltol * max(abs(ref["total"]), 1e-6), (got["loss"], ref["total"])
    assert relerr(got["logits"], ref["logits"]) <= TOL[dt], relerr(got["logits"], ref["logits"])
    tol = TOL[dt]
    for k in ("dW1", "db1", "dw2", "db2"):
        assert relerr(got[k].reshape(g[k].shape), g[k]) <= tol, (k, relerr(got[k].reshape(g[k].shape), g[k]))
    assert relerr(got["dH"], g["dH"]) <= tol, relerr(got["dH"], g["dH"])
    assert relerr(got["dH_rep"], g["dH_rep"]) <= tol, relerr(got["dH_rep"], g["dH_rep"])
    # rows that are neither labelled nor a labelled row's replica get nothing
    assert np.abs(got["dH"][g["dH"] == 0]).max(initial=0) == 0
    return ref, g


@pytest.mark.parametrize("dt,d,N,n_lab,n_rep", [("f32", 64, 2000, 700, 300), ("bf16", 128, 9000, 3001, 1500),
                                                ("bf16", 256, 3000, 1000, 400), ("bf16", 64, 2600, 999, 500),
                                                ("f32", 128, 5000, 1777, 800), ("f32", 256, 1500, 130, 100)])
def test_head_matches_oracle(dt, d, N, n_lab, n_rep):
    need_gpu()
    hg = lib()
    H, Hr, ia, ib, lab, y, p = problem(d + n_lab, N, d, n_lab, n_rep, dt, rows_rep=N + 37)
    got = head_gpu(hg, H, Hr, ia, ib, lab, y, p, dt, cca=1.7, lam=0.1)
    check(got, H, Hr, ia, ib, lab, y, p, dt, cca=1.7, lam=0.1)


def test_head_fractional_labels_dloss_and_accumulation():
    need_gpu()
    hg = lib()
    H, Hr, ia, ib, lab, y, p = problem(5, 4000, 128, 1500, 900, "bf16", frac_y=True)
    got = head_gpu(hg, H, Hr, ia, ib, lab, y, p, "bf16", dloss=0.37, base=1.0)
    # accumulated onto N(0,1) bf16 values: the increment carries the rounding of the sum
    g = OH.head_backward(H, ia, Hr, ib, lab, y, p, dloss=0.37)
    for k in ("dW1", "db1", "dw2", "db2"):
        assert relerr(got[k].reshape(g[k].shape), g[k]) <= TOL["bf16"], k
    rows = np.unique(np.concatenate([lab]))
    assert np.abs(got["dH"][rows] - g["dH"][rows]).max() <= 2.0 ** -8 * 4 + TOL["bf16"] * np.abs(g["dH"]).max()


def test_head_fp32_tight():
    """fp32 storage: every output within 1e-5 normwise."""
    need_gpu()
    hg = lib()
    H, Hr, ia, ib, lab, y, p = problem(9, 3000, 64, 2500, 1200, "f32")
    got = head_gpu(hg, H, Hr, ia, ib, lab, y, p, "f32")
    ref, g = check(got, H, Hr, ia, ib, lab, y, p, "f32")
    assert relerr(got["dH"], g["dH"]) <= 1e-5 and relerr(got["dW1"], g["dW1"]) <= 1e-5


def test_head_device_count_detached_and_degenerate():
    need_gpu()
    hg = lib()
    H, Hr, ia, ib, lab, y, p = problem(13, 1800, 64, 600, 500, "f32")
    # capacity 500, 350 pairs counted on the device; the second view detached
    got = head_gpu(hg, H, Hr, ia, ib, lab, y, p, "f32", n_rep_dev=350, both=False, base=1.0, rep_cap=500)
    g = OH.head_backward(H, ia[:350], Hr, ib[:350], lab, y, p)
    ref = OH.head_loss(H, ia[:350], Hr, ib[:350], lab, y, p)
    assert abs(got["loss"][1] - ref["bce"]) <= 1e-5 * ref["bce"]
    assert np.abs(got["dH"] - g["dH"]).max() <= 1e-6 * 8 + 1e-5 * np.abs(g["dH"]).max()
    assert torch.equal(got["dR_t"], got["base_b"])  # detached view untouched
    # a negative device count means no replicas
    got = head_gpu(hg, H, Hr, ia, ib, lab, y, p, "f32", n_rep_dev=-1, rep_cap=500)
    check(got, H, Hr, ia[:0], ib[:0], lab, y, p, "f32")
    # no labelled rows: L_BCE = 0, L_total = lambda * L_CCA, zero gradients
    got = head_gpu(hg, H, Hr, ia, ib, lab[:0], y[:0], p, "f32", cca=2.0, lam=0.1)
    assert got["loss"][1] == 0 and abs(got["loss"][0] - 0.2) < 1e-7
    for k in ("dW1", "db1", "dw2", "db2", "dH", "dH_rep"):
        assert np.abs(got[k]).max() == 0, k
    # one labelled row
    got = head_gpu(hg, H, Hr, ia, ib, lab[:1], y[:1], p, "f32")
    check(got, H, Hr, ia, ib, lab[:1], y[:1], p, "f32")


def test_head_out_of_range_label_row():
    need_gpu()
    hg = lib()
    H, Hr, ia, ib, lab, y, p = problem(17, 1000, 64, 300, 200, "f32")
    bad = lab.copy()
    bad[7] = 1000  # == rows: out of range
    got = head_gpu(hg, H, Hr, ia, ib, bad, y, p, "f32")
    assert np.isnan(got["loss"][0]) and np.isnan(got["loss"][1])
    keep = np.delete(np.arange(len(lab)), 7)
    # the mean still divides by all 300 rows: the other rows' gradients are the oracle's on 299 rows
    # scaled by 299 / 300
    g = OH.head_backward(H, ia, Hr, ib, lab[keep], y[keep], p, dloss=299 / 300)
    for k in ("dW1", "db1", "dw2", "db2", "dH", "dH_rep"):
        assert relerr(got[k].reshape(g[k].shape), g[k]) <= 1e-5, k


def test_head_deterministic():
    need_gpu()
    hg = lib()
    H, Hr, ia, ib, lab, y, p = problem(21, 20000, 128, 9000, 4000, "bf16")
    a = head_gpu(hg, H, Hr, ia, ib, lab, y, p, "bf16")
    b = head_gpu(hg, H, Hr, ia, ib, lab, y, p, "bf16")
    for k in ("loss", "logits", "dW1", "db1", "dw2", "db2", "dH", "dH_rep"):
        assert np.array_equal(a[k], b[k]), k


def test_head_overwrite_mode():
    """overwrite=True: dH and dH_rep are cleared first, so they hold the head's gradient alone."""
    need_gpu()
    hg = lib()
    H, Hr, ia, ib, lab, y, p = problem(23, 2000, 64, 600, 300, "f32")
    td = torch.float32
    prm = hg.HeadParams(dev(p["W1"], td), dev(p["b1"], td), dev(p["w2"], td), dev(p["b2"], td))
    s, k = hg.hg_head_workspace_size(H.shape[0], len(lab), 64, td)
    saved = torch.empty(s, dtype=torch.uint8, device="cuda")
    scratch = torch.empty(k, dtype=torch.uint8, device="cuda")
    A, B = dev(H, td), dev(Hr, td)
    loss = torch.empty(2, dtype=torch.float32, device="cuda")
    hg.hg_head_loss(prm, A, B, dev(ia), dev(ib), len(ia), None, dev(lab), dev(y), None, 0.1, loss, None, saved, scratch)
    f = dict(dtype=torch.float32, device="cuda")
    grads = {"W1": torch.empty(64, 64, **f), "b1": torch.empty(64, **f), "w2": torch.empty(64, **f),
             "b2": torch.empty(1, **f)}
    dH = torch.randn_like(A)  # stale contents that must not survive
    dR = torch.randn_like(B)
    hg.hg_head_bwd(prm, dev(lab), 1.0, saved, dH, dR, grads, scratch, overwrite=True)
    torch.cuda.synchronize()
    g = OH.head_backward(H, ia, Hr, ib, lab, y, p)
    assert relerr(host(dH), g["dH"]) <= 1e-5 and relerr(host(dR), g["dH_rep"]) <= 1e-5
    assert np.all(host(dH)[g["dH"] == 0] == 0)
