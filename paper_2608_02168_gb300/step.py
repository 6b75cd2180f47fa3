"""One step of the hot path on one overlapping subgraph, driven through the C ABI.

A step (Algorithm 1, the per-worker part of one iteration, on one GPU):
  hg_build_csr           relation-typed CSR / CSC of the subgraph
  hg_layer_fwd x L       heterogeneous mean-aggregation layers (Eq. 7, 10, 11)
  hg_overlap_intersect   overlap rows with the neighbouring subgraph (Section 3.3)
  hg_overlap_align_loss  CCA alignment loss (Eq. 14-17)
  hg_head_loss           (with a head and labels) MeanAgg of the replicas, the two-layer MLP and
                         the masked BCE over the labelled rows, and L_total = L_BCE + lambda_CCA
                         L_CCA (Eq. 18-20)
  hg_head_bwd            its gradient, written as the last layer's upstream gradient (without a
                         head the caller supplies that gradient, dH_top)
  hg_overlap_align_bwd   the alignment gradient, scaled by lambda_CCA (Eq. 20), added to it
  hg_layer_bwd x L       gradients of every layer, including dL/dX of the first.
This module only allocates buffers (torch) and marshals arguments; every computation runs in
libhg's kernels.
"""
from __future__ import annotations

import torch

from . import hg

LAMBDA_N = 2e-4     # weight of the decorrelation term (Section 4.1, implementation details)
LAMBDA_CCA = 0.1    # weight of the alignment loss in the joint objective (Section 4.1)
VAR_EPS = 1e-8
LN_EPS = 1e-5


def _torch_dtype(dtype: str):
    return torch.float32 if dtype == "f32" else torch.bfloat16


class HotPath:
    """Buffers for one subgraph shape, reused across steps.

    view: "bank"      -> the second view is a detached embedding table of a neighbouring subgraph
                         (rows found by intersecting the two global-id lists);
          "perturbed" -> the second view is a second live stack run on other input features over the
                         same graph, aligned on the given overlap rows, with gradients into both.
    fused: run every layer as the fused mean layer (bf16, d = 128; the relation means are not kept
           between the forward and the backward pass, results unchanged bit for bit).
    """

    def __init__(self, type_offsets, rels, num_edges: int, d: int, dtype: str, layer_params: list,
                 view: str, n_overlap_max: int, n_gid_a: int = 0, n_gid_b: int = 0, act: str = "relu",
                 layernorm: bool = True, device="cuda", head_params: dict | None = None, n_lab_max: int = 0,
                 fused: bool = False):
        self.type_offsets = [int(x) for x in type_offsets]
        self.rels = [tuple(r) for r in rels]
        self.N = self.type_offsets[-1]
        self.d, self.dtype, self.view = d, dtype, view
        self.L = len(layer_params)
        self.device = torch.device(device)
        td = _torch_dtype(dtype)
        self.td = td
        dev = self.device
        self.params = []
        for p in layer_params:
            self.params.append(hg.LayerParams(
                torch.as_tensor(p["W_rel"], device=dev).to(td), torch.as_tensor(p["W_agg"], device=dev).to(td),
                torch.as_tensor(p["b_agg"], device=dev).to(td), torch.as_tensor(p["ln_gamma"], device=dev).to(td),
                torch.as_tensor(p["ln_beta"], device=dev).to(td), act=act, layernorm=layernorm, ln_eps=LN_EPS,
                fused=fused))
        self.graph_ws = torch.empty(hg.hg_graph_workspace_size(num_edges, self.type_offsets, self.rels),
                                    dtype=torch.uint8, device=dev)
        saved_b, scratch_b = self._layer_sizes(num_edges)
        stacks = 2 if view == "perturbed" else 1
        self.H = [[torch.empty(self.N, d, dtype=td, device=dev) for _ in range(self.L + 1)] for _ in range(stacks)]
        self.dH = [[torch.empty(self.N, d, dtype=td, device=dev) for _ in range(self.L + 1)] for _ in range(stacks)]
        self.saved = [[torch.empty(saved_b, dtype=torch.uint8, device=dev) for _ in range(self.L)] for _ in range(stacks)]
        self.scratch = torch.empty(scratch_b, dtype=torch.uint8, device=dev)
        self.grads = [[self._grad_bufs() for _ in range(self.L)] for _ in range(stacks)]
        # the alignment kernels read the actual overlap size from the device; n_overlap_max only bounds
        # buffers: the given size for fixed overlap rows, the smaller id list for an intersection
        self.n_overlap_max = int(n_overlap_max) if view == "perturbed" else max(1, min(n_gid_a, n_gid_b))
        a_s, a_k = hg.hg_overlap_align_workspace_size(self.n_overlap_max, d)
        self.align_saved = torch.empty(max(a_s, 256), dtype=torch.uint8, device=dev)
        self.align_scratch = torch.empty(max(a_k, 256), dtype=torch.uint8, device=dev)
        self.loss = torch.zeros(3, dtype=torch.float32, device=dev)
        self.n_dev = torch.zeros(1, dtype=torch.int64, device=dev)
        if view == "bank":
            cap = max(1, min(n_gid_a, n_gid_b))
            self.idx_a = torch.empty(cap, dtype=torch.int32, device=dev)
            self.idx_b = torch.empty(cap, dtype=torch.int32, device=dev)
            self.isect_scratch = torch.empty(hg.hg_overlap_intersect_workspace_size(n_gid_a, n_gid_b),
                                             dtype=torch.uint8, device=dev)
        self.head = None
        if head_params is not None:
            self.head = hg.HeadParams(*(torch.as_tensor(head_params[k], device=dev).to(td) for k in ("W1", "b1", "w2", "b2")))
            h_s, h_k = hg.hg_head_workspace_size(self.N, max(1, int(n_lab_max)), d, td)
            self.head_saved = torch.empty(h_s, dtype=torch.uint8, device=dev)
            self.head_scratch = torch.empty(h_k, dtype=torch.uint8, device=dev)
            self.head_loss = torch.zeros(2, dtype=torch.float32, device=dev)
            f = torch.float32
            self.head_grads = {"W1": torch.empty(d, d, dtype=f, device=dev), "b1": torch.empty(d, dtype=f, device=dev),
                               "w2": torch.empty(d, dtype=f, device=dev), "b2": torch.empty(1, dtype=f, device=dev)}
        self.graph = None

    def _layer_sizes(self, num_edges: int):
        """Layer buffer sizes depend on the node types, relations and edge count only; ask the
        library with a placeholder graph of that shape (edges of relation 0 spread over its rows)."""
        dev = self.device
        s_t, d_t = self.rels[0]
        n_s = max(1, self.type_offsets[s_t + 1] - self.type_offsets[s_t])
        n_d = max(1, self.type_offsets[d_t + 1] - self.type_offsets[d_t])
        k = torch.arange(num_edges, dtype=torch.int64, device=dev)
        src = (self.type_offsets[s_t] + k % n_s).to(torch.int32)
        dst = (self.type_offsets[d_t] + k % n_d).to(torch.int32)
        rel = torch.zeros(num_edges, dtype=torch.int32, device=dev)
        g = hg.hg_build_csr(src, dst, rel, self.type_offsets, self.rels, workspace=self.graph_ws)
        s, k2 = hg.hg_layer_workspace_size(g, self.params[0])
        del g
        return s, k2

    def _grad_bufs(self):
        d, dev = self.d, self.device
        R, T = len(self.rels), len(self.type_offsets) - 1
        f = torch.float32
        return {"W_rel": torch.empty(R, d, d, dtype=f, device=dev), "W_agg": torch.empty(T, d, d, dtype=f, device=dev),
                "b_agg": torch.empty(T, d, dtype=f, device=dev), "ln_gamma": torch.empty(T, d, dtype=f, device=dev),
                "ln_beta": torch.empty(T, d, dtype=f, device=dev)}

    # --------------------------------------------------------------------------------------------
    def step(self, src, dst, rel, X, dH_top, X_b=None, overlap_idx=None, gid_a=None, gid_b=None, H_bank=None,
             stream=None, marks=None, lab_idx=None, lab_y=None):
        """Run one step; all inputs are device tensors.  Returns nothing (results stay in the buffers:
        self.H, self.loss, self.grads, self.dH[s][0] = dL/dX; with a head, self.head_loss =
        [L_total, L_BCE] and self.head_grads).  With a head and labels (lab_idx, lab_y) the last
        layer's upstream gradient is the head's and dH_top is ignored.  `marks`, if a list, receives
        (phase, CUDA event) pairs recorded on the stream after the graph build, the forward layers,
        the alignment loss, the head (when it runs), the alignment gradient and the backward layers."""
        def mark(name):
            if marks is not None:
                ev = torch.cuda.Event(enable_timing=True)
                ev.record(stream if stream is not None else torch.cuda.current_stream())
                marks.append((name, ev))

        self.graph = hg.hg_build_csr(src, dst, rel, self.type_offsets, self.rels, workspace=self.graph_ws,
                                     stream=stream)
        mark("graph")
        g = self.graph
        stacks = [X] if self.view == "bank" else [X, X_b]
        for s, x in enumerate(stacks):
            self.H[s][0] = x
            for l in range(self.L):
                hg.hg_layer_fwd(g, self.params[l], self.H[s][l], self.H[s][l + 1], self.saved[s][l], self.scratch, stream)
        mark("forward")
        top = self.H[0][self.L]
        use_head = self.head is not None and lab_idx is not None
        if not use_head:  # with a head, hg_head_bwd writes the whole upstream gradient
            self.dH[0][self.L].copy_(dH_top)
        if self.view == "bank" and H_bank is None:
            # first subgraph of a sequence: no neighbour view yet, no alignment term
            self.loss.zero_()
            mark("alignment")
            if use_head:
                self._head(top, None, None, None, 0, None, None, lab_idx, lab_y, stream)
                mark("head")
            for l in range(self.L - 1, -1, -1):
                hg.hg_layer_bwd(g, self.params[l], self.H[0][l], self.saved[0][l], self.dH[0][l + 1], self.dH[0][l],
                                self.grads[0][l], self.scratch, stream)
            mark("backward")
            return
        if self.view == "bank":
            hg.hg_overlap_intersect(gid_a, gid_b, self.idx_a, self.idx_b, self.n_dev, self.isect_scratch, stream)
            n_max = self.n_overlap_max
            ia, ib, Hb, dHb, n_dev = self.idx_a, self.idx_b, H_bank, None, self.n_dev
        else:
            n_max = int(overlap_idx.numel())
            ia = ib = overlap_idx
            Hb = self.H[1][self.L]
            dHb, n_dev = self.dH[1][self.L], None
            if not use_head:
                dHb.zero_()
        hg.hg_overlap_align_loss(top, ia, Hb, ib, n_max, n_dev, LAMBDA_N, VAR_EPS, self.loss, self.align_saved,
                                 self.align_scratch, stream)
        mark("alignment")
        if use_head:  # L_total needs L_CCA; the head's gradient overwrites the upstream gradient buffers
            self._head(top, Hb, ia, ib, n_max, n_dev, dHb, lab_idx, lab_y, stream)
            mark("head")
        hg.hg_overlap_align_bwd(top, ia, Hb, ib, n_max, n_dev, LAMBDA_N, VAR_EPS, LAMBDA_CCA, self.align_saved,
                                self.dH[0][self.L], dHb, self.align_scratch, stream)
        mark("alignment_bwd")
        for s in range(len(stacks)):
            for l in range(self.L - 1, -1, -1):
                hg.hg_layer_bwd(g, self.params[l], self.H[s][l], self.saved[s][l], self.dH[s][l + 1], self.dH[s][l],
                                self.grads[s][l], self.scratch, stream)
        mark("backward")

    def _head(self, top, H_rep, ia, ib, n_max, n_dev, dH_rep, lab_idx, lab_y, stream):
        """Head loss (L_total with the alignment loss just computed) and its gradient into the last
        layer's upstream gradient (and the second view's, when that view is live)."""
        hg.hg_head_loss(self.head, top, H_rep, ia, ib, n_max, n_dev, lab_idx, lab_y, self.loss, LAMBDA_CCA,
                        self.head_loss, None, self.head_saved, self.head_scratch, stream)
        hg.hg_head_bwd(self.head, lab_idx, 1.0, self.head_saved, self.dH[0][self.L], dH_rep, self.head_grads,
                       self.head_scratch, stream, overwrite=True)


class Ring:
    """Overlapping subgraphs processed one after another on one GPU (the per-worker step of
    Algorithm 1 for each subgraph in turn).  Subgraph k aligns its overlap rows with the final
    embeddings of subgraph k-1, held as a detached view (no gradient flows into them); the first
    subgraph has no alignment term.  All subgraphs share the layer weights and sizes."""

    def __init__(self, type_offsets, rels, num_edges: int, d: int, dtype: str, layer_params: list, device="cuda"):
        n = int(type_offsets[-1])
        self.path = HotPath(type_offsets, rels, num_edges, d, dtype, layer_params, view="bank", n_overlap_max=n,
                            n_gid_a=n, n_gid_b=n, device=device)
        self.bank = torch.empty(n, d, dtype=self.path.td, device=self.path.device)
        self.bank_gid = torch.empty(n, dtype=torch.int64, device=self.path.device)
        self.have_bank = False

    def step(self, src, dst, rel, X, dH_top, gid, stream=None):
        p = self.path
        if self.have_bank:
            p.step(src, dst, rel, X, dH_top, gid_a=gid, gid_b=self.bank_gid, H_bank=self.bank, stream=stream)
        else:
            p.step(src, dst, rel, X, dH_top, stream=stream)
        # keep this subgraph's embeddings as the next one's view: swap buffers instead of copying
        p.H[0][p.L], self.bank = self.bank, p.H[0][p.L]
        self.bank_gid.copy_(gid)
        self.have_bank = True
        return self.bank
