"""Several overlapping subgraphs processed in sequence on one GPU (the ring workload at reduced
size): each subgraph aligns with the detached final embeddings of the previous one; compared
step by step with the oracle running the same sequence on its own outputs."""
import numpy as np
import pytest
import torch

import hgsynth
import oracle
from tests.gpu_util import BF16_RELU_MARGIN, TOL, dev, host, lib, need_gpu, relerr, tdtype

pytestmark = pytest.mark.gpu


def test_ring_sequence_matches_oracle():
    need_gpu()
    lib()
    from paper_2608_02168_gb300.step import Ring
    sp = hgsynth.spec("ring16-2m", n_user=9_000, n_risk=1_000, num_edges=150_000, n_overlap=2_000, num_subgraphs=4)
    params = [hgsynth.make_layer_params(sp, l, random_affine=True, bias_margin=BF16_RELU_MARGIN)
              for l in range(sp.layers)]
    td = tdtype(sp.dtype)
    ring = None
    prev_H, prev_gid = None, None
    for k in range(sp.num_subgraphs):
        part = hgsynth.make_ring_part(sp, k)
        g = part.graph
        if ring is None:
            ring = Ring(g["type_offsets"], g["rels"], len(g["src"]), sp.d, sp.dtype, params)
        bank = ring.step(dev(g["src"]), dev(g["dst"]), dev(g["rel"]), dev(part.X, td), dev(part.dH_top, td),
                         dev(part.gid))
        torch.cuda.synchronize()
        vb = None if prev_H is None else {"H_b": prev_H, "gid_a": part.gid, "gid_b": prev_gid}
        # the plain fp64 definition, with the interface's bf16 layer outputs and gradients
        ref = oracle.step(g, part.X, params, part.dH_top, vb, interface="bf16")
        p = ring.path
        assert relerr(host(bank), ref["H"][-1]) <= TOL[sp.dtype], k
        if k > 0:
            assert int(p.n_dev.item()) == sp.n_overlap == len(ref["idx_a"])
            assert relerr(host(p.loss), np.array(ref["loss"])) <= 2e-2, k
        assert relerr(host(p.dH[0][0]), ref["dX"]) <= TOL[sp.dtype], k
        for l in range(sp.layers):
            for key, v in ref["grads"][l].items():
                assert relerr(host(p.grads[0][l][key]), v) <= TOL[sp.dtype], (k, l, key)
        prev_H, prev_gid = ref["H"][-1], part.gid
