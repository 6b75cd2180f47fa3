"""The full-size ring: sixteen overlapping subgraphs of 2M nodes / 40M edges (bf16, d = 128, two
layers) processed in sequence on one GPU, each aligned with the detached final embeddings of the one
before (Algorithm 1 run worker by worker).  Inputs come from the device-side generator (the same
recipe as the numpy one, drawn on the GPU), so sixteen instances take seconds.

For every subgraph: the overlap rows bit for bit, the alignment loss in full and the last layer's
upstream gradient (synthetic gradient plus lambda_CCA times the alignment gradient) in full, against
the oracle evaluated on the GPU's own final embeddings and bank (teacher forcing).  On four of the
subgraphs, each layer forward and backward on sampled rows against the oracle's sampled-row forms,
given the GPU's input of that layer (its output rows depend only on their in-neighbours; its input
gradient rows only on their own and their out-neighbours' upstream gradient)."""
import numpy as np
import pytest
import torch

import hgsynth
import oracle
from tests.gpu_util import BF16_RELU_MARGIN, TOL, host, lib, need_gpu, relerr

pytestmark = pytest.mark.gpu

LAYER_CHECKS = (0, 1, 8, 15)


def query_rows(src_np, n, k, seed):
    """k random rows of small out-degree (their out-neighbourhoods stay small) and their
    out-neighbours (the upstream support their input gradient depends on)."""
    rng = np.random.default_rng(seed)
    outdeg = np.bincount(src_np, minlength=n)
    pool = np.flatnonzero(outdeg <= 64)
    q = np.sort(rng.choice(pool, k, replace=False))
    return q


def test_full_ring_sequence():
    need_gpu()
    lib()
    from hgsynth import device as hd
    from paper_2608_02168_gb300.step import LAMBDA_CCA, LAMBDA_N, VAR_EPS, Ring
    sp = hgsynth.spec("ring16-2m")
    dev = torch.device("cuda")
    params = [hgsynth.make_layer_params(sp, l, random_affine=True, bias_margin=BF16_RELU_MARGIN)
              for l in range(sp.layers)]
    table = hd.ring_features(sp, dev)
    ring = None
    prev_final, prev_gid = None, None
    tol = TOL["bf16"]
    for k in range(sp.num_subgraphs):
        part = hd.make_ring_part(sp, k, table, dev)
        g = part["graph"]
        dH_top = hd.make_features(sp, k, dev, 4)
        if ring is None:
            ring = Ring(g["type_offsets"], g["rels"], int(g["src"].shape[0]), sp.d, sp.dtype, params, device=dev)
        p = ring.path
        final = ring.step(g["src"], g["dst"], g["rel"], part["X"], dH_top, part["gid"])
        torch.cuda.synchronize()
        gid = part["gid"].cpu().numpy()
        H_fin = host(final)
        if k > 0:
            ia, ib = oracle.overlap_intersect(gid, prev_gid)
            n = int(p.n_dev.item())
            assert n == len(ia) == sp.n_overlap, (k, n)
            assert np.array_equal(p.idx_a[:n].cpu().numpy(), ia) and np.array_equal(p.idx_b[:n].cpu().numpy(), ib)
            ref_loss = oracle.align_forward(H_fin, ia, prev_final, ib, LAMBDA_N, VAR_EPS)
            assert relerr(host(p.loss), np.array(ref_loss)) <= tol, (k, host(p.loss), ref_loss)
            dA, _ = oracle.align_backward(H_fin, ia, prev_final, ib, LAMBDA_N, VAR_EPS, LAMBDA_CCA)
        else:
            dA = 0.0
        # the last layer's upstream gradient: synthetic gradient plus the alignment term
        want_top = host(dH_top) + dA
        assert relerr(host(p.dH[0][sp.layers]), want_top) <= tol, k
        if k in LAYER_CHECKS:
            src, dst, rel = (g[x].cpu().numpy() for x in ("src", "dst", "rel"))
            offs, rels = g["type_offsets"], g["rels"]
            outs = [host(p.H[0][l]) for l in range(sp.layers)] + [H_fin]
            rng = np.random.default_rng(100 + k)
            rows = np.unique(np.concatenate([rng.choice(sp.num_nodes, 1500, replace=False),
                                             np.argsort(-np.bincount(dst, minlength=sp.num_nodes))[:4]]))
            q = query_rows(src, sp.num_nodes, 300, 200 + k)
            supp = np.unique(np.concatenate([q, dst[np.isin(src, q)]]))
            for l in range(sp.layers):
                ref, _ = oracle.layer_forward_rows(src, dst, rel, offs, rels, params[l], outs[l], rows)
                assert relerr(outs[l + 1][rows], ref) <= tol, ("forward", k, l)
                dup = host(p.dH[0][l + 1])
                dq, _ = oracle.layer_backward_rows(src, dst, rel, offs, rels, params[l], outs[l], supp, dup[supp], q)
                assert relerr(host(p.dH[0][l])[q], dq) <= tol, ("backward", k, l)
        prev_final, prev_gid = H_fin, gid
        del part, g, dH_top
    from paper_2608_02168_gb300 import hg
    assert hg.hg_device_status() == 0
