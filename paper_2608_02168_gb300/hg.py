"""Python binding of libhg (include/hg.h): same entry-point names, argument marshalling only.

Device buffers are torch CUDA tensors (their data pointers are passed through); streams are torch
streams.  Every computation happens inside libhg's CUDA kernels.  A missing library raises
ImportError: there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, Structure, byref, c_char_p, c_float, c_int32, c_int64, c_size_t, c_uint64, c_void_p

import torch

from . import build as _build

HG_F32, HG_BF16 = 0, 1
HG_ACT_RELU, HG_ACT_GELU_TANH, HG_ACT_NONE = 0, 1, 2
DTYPES = {"f32": HG_F32, "bf16": HG_BF16}
TORCH_DTYPES = {HG_F32: torch.float32, HG_BF16: torch.bfloat16}
ACTS = {"relu": HG_ACT_RELU, "gelu_tanh": HG_ACT_GELU_TANH, "none": HG_ACT_NONE}


class hg_rel_desc(Structure):
    _fields_ = [("src_type", c_int32), ("dst_type", c_int32)]


class hg_graph_arrays(Structure):
    _fields_ = [("n_dst", c_int64), ("n_src", c_int64), ("num_edges", c_int64), ("row_ptr", c_void_p),
                ("col", c_void_p), ("eid", c_void_p), ("csc_ptr", c_void_p), ("csc_col", c_void_p),
                ("csc_eid", c_void_p), ("csc_coef", c_void_p)]


class hg_node_order(Structure):
    _fields_ = [("n", c_int64), ("tiles", c_int64), ("tile_rows", c_int32), ("perm", c_void_p),
                ("tile_mask", c_void_p)]


class hg_layer_params(Structure):
    _fields_ = [("d", c_int32), ("dtype", c_int32), ("act", c_int32), ("layernorm", c_int32), ("ln_eps", c_float),
                ("W_rel", c_void_p), ("W_agg", c_void_p), ("b_agg", c_void_p), ("ln_gamma", c_void_p),
                ("ln_beta", c_void_p), ("fused", c_int32)]


class hg_layer_grads(Structure):
    _fields_ = [("dW_rel", c_void_p), ("dW_agg", c_void_p), ("db_agg", c_void_p), ("dln_gamma", c_void_p),
                ("dln_beta", c_void_p)]


class hg_hgt_params(Structure):
    _fields_ = [("d", c_int32), ("heads", c_int32), ("dtype", c_int32), ("act", c_int32), ("layernorm", c_int32),
                ("ln_eps", c_float), ("W_K", c_void_p), ("W_Q", c_void_p), ("W_V", c_void_p), ("b_K", c_void_p),
                ("b_Q", c_void_p), ("b_V", c_void_p), ("W_att", c_void_p), ("W_msg", c_void_p), ("mu", c_void_p),
                ("W_agg", c_void_p), ("b_agg", c_void_p), ("ln_gamma", c_void_p), ("ln_beta", c_void_p)]


HGT_KEYS = ("W_K", "W_Q", "W_V", "b_K", "b_Q", "b_V", "W_att", "W_msg", "mu", "W_agg", "b_agg", "ln_gamma", "ln_beta")


class hg_hgt_grads(Structure):
    _fields_ = [("d" + k, c_void_p) for k in HGT_KEYS]


class hg_head_params(Structure):
    _fields_ = [("d", c_int32), ("dtype", c_int32), ("W1", c_void_p), ("b1", c_void_p), ("w2", c_void_p),
                ("b2", c_void_p)]


class hg_head_grads(Structure):
    _fields_ = [("dW1", c_void_p), ("db1", c_void_p), ("dw2", c_void_p), ("db2", c_void_p)]


class hg_temporal_params(Structure):
    _fields_ = [("d", c_int32), ("w", c_int32), ("dtype", c_int32), ("Wa", c_void_p), ("r", c_void_p),
                ("W_i", c_void_p), ("W_h", c_void_p), ("b_i", c_void_p), ("b_h", c_void_p)]


class hg_temporal_grads(Structure):
    _fields_ = [("dWa", c_void_p), ("dr", c_void_p), ("dW_i", c_void_p), ("dW_h", c_void_p), ("db_i", c_void_p),
                ("db_h", c_void_p)]


EXPORTS = {
    # name: (restype, argtypes)
    "hg_status_string": (c_char_p, [c_int32]),
    "hg_last_error": (c_char_p, []),
    "hg_abi_version": (c_int32, []),
    "hg_device_status": (c_int32, [POINTER(c_int32)]),
    "hg_bind_device": (c_int32, [c_int32]),
    "hg_selftest_bounded_wait": (c_int32, [ctypes.c_uint32, c_void_p]),
    "hg_graph_workspace_size": (c_int32, [c_int64, POINTER(c_int64), c_int32, POINTER(hg_rel_desc), c_int32,
                                          POINTER(c_size_t)]),
    "hg_build_csr": (c_int32, [c_void_p, c_void_p, c_void_p, c_int64, POINTER(c_int64), c_int32,
                               POINTER(hg_rel_desc), c_int32, c_void_p, c_size_t, c_void_p, POINTER(c_void_p)]),
    "hg_graph_destroy": (c_int32, [c_void_p]),
    "hg_graph_check": (c_int32, [c_void_p, POINTER(c_int64)]),
    "hg_graph_view": (c_int32, [c_void_p, c_int32, POINTER(hg_graph_arrays)]),
    "hg_graph_node_order": (c_int32, [c_void_p, c_int32, POINTER(hg_node_order)]),
    "hg_layer_workspace_size": (c_int32, [c_void_p, POINTER(hg_layer_params), POINTER(c_size_t), POINTER(c_size_t)]),
    "hg_layer_fwd": (c_int32, [c_void_p, POINTER(hg_layer_params), c_void_p, c_void_p, c_void_p, c_void_p, c_void_p]),
    "hg_layer_bwd": (c_int32, [c_void_p, POINTER(hg_layer_params), c_void_p, c_void_p, c_void_p, c_void_p,
                               POINTER(hg_layer_grads), c_void_p, c_void_p]),
    "hg_overlap_intersect_workspace_size": (c_int32, [c_int64, c_int64, POINTER(c_size_t)]),
    "hg_overlap_intersect": (c_int32, [c_void_p, c_int64, c_void_p, c_int64, c_void_p, c_void_p, c_void_p, c_void_p,
                                       c_size_t, c_void_p]),
    "hg_overlap_align_workspace_size": (c_int32, [c_int64, c_int32, POINTER(c_size_t), POINTER(c_size_t)]),
    "hg_overlap_align_loss": (c_int32, [c_void_p, c_int64, c_void_p, c_void_p, c_int64, c_void_p, c_int64, c_void_p,
                                        c_int32, c_int32, c_float, c_float, c_void_p, c_void_p, c_void_p, c_void_p]),
    "hg_overlap_align_bwd": (c_int32, [c_void_p, c_int64, c_void_p, c_void_p, c_int64, c_void_p, c_int64, c_void_p,
                                       c_int32, c_int32, c_float, c_float, c_float, c_void_p, c_void_p, c_void_p,
                                       c_void_p, c_void_p]),
    "hg_overlap_align_loss_static": (c_int32, [c_void_p, c_int64, c_void_p, c_void_p, c_int64, c_void_p, c_int64,
                                               c_void_p, c_int32, c_int32, c_float, c_float, c_void_p, c_void_p,
                                               c_void_p]),
    "hg_overlap_build_workspace_size": (c_int32, [c_int64, c_int64, POINTER(c_size_t)]),
    "hg_overlap_build": (c_int32, [c_void_p, c_void_p, c_void_p, c_int64, c_int64, POINTER(c_int64), c_int32, c_int32,
                                   c_int32, c_int32, c_int64, c_uint64, c_uint64, c_void_p, c_void_p, c_void_p,
                                   c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_size_t, c_void_p]),
    "hg_head_workspace_size": (c_int32, [c_int64, c_int64, c_int32, c_int32, POINTER(c_size_t), POINTER(c_size_t)]),
    "hg_head_loss": (c_int32, [POINTER(hg_head_params), c_void_p, c_int64, c_void_p, c_int64, c_void_p, c_void_p,
                               c_int64, c_void_p, c_void_p, c_void_p, c_int64, c_void_p, c_float, c_void_p, c_void_p,
                               c_void_p, c_void_p, c_void_p]),
    "hg_head_bwd": (c_int32, [POINTER(hg_head_params), c_void_p, c_int64, c_float, c_void_p, c_void_p, c_int64,
                              c_void_p, c_int64, c_int32,
                              POINTER(hg_head_grads), c_void_p, c_void_p]),
    "hg_temporal_workspace_size": (c_int32, [c_int64, c_int32, c_int32, c_int32, POINTER(c_size_t),
                                             POINTER(c_size_t)]),
    "hg_temporal_fwd": (c_int32, [POINTER(hg_temporal_params), c_void_p, c_void_p, c_int64, c_void_p, c_void_p,
                                  c_void_p, c_void_p]),
    "hg_temporal_bwd": (c_int32, [POINTER(hg_temporal_params), c_void_p, c_void_p, c_int64, c_void_p, c_void_p,
                                  c_void_p, POINTER(hg_temporal_grads), c_void_p, c_void_p]),
    "hg_hgt_workspace_size": (c_int32, [c_void_p, POINTER(hg_hgt_params), POINTER(c_size_t), POINTER(c_size_t)]),
    "hg_hgt_fwd": (c_int32, [c_void_p, POINTER(hg_hgt_params), c_void_p, c_void_p, c_void_p, c_void_p, c_void_p]),
    "hg_hgt_bwd": (c_int32, [c_void_p, POINTER(hg_hgt_params), c_void_p, c_void_p, c_void_p, c_void_p,
                             POINTER(hg_hgt_grads), c_void_p, c_void_p]),
    "hg_timing_enable": (c_int32, [c_int32]),
    "hg_timing_report": (c_int32, [c_char_p, c_size_t]),
}

_lib = None


class HGError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str):
        super().__init__(f"{where}: status {status} ({_lib.hg_status_string(status).decode()}): {detail}")
        self.status = status


def lib() -> ctypes.CDLL:
    """The loaded libhg.so (ImportError if it has not been built)."""
    global _lib
    if _lib is None:
        path = _build.library_path()
        if not os.path.exists(path):
            raise ImportError(f"{path} is missing: build it with __graft_entry__.build() or "
                              "`python -m paper_2608_02168_gb300.build`")
        so = ctypes.CDLL(path)
        for name, (res, args) in EXPORTS.items():
            fn = getattr(so, name)
            fn.restype = res
            fn.argtypes = args
        _lib = so
    return _lib


def _check(status: int, where: str):
    if status != 0:
        raise HGError(status, where, lib().hg_last_error().decode())


def _ptr(t) -> int | None:
    """Device address of a tensor argument (None passes NULL).  The library reads rows by address from
    device memory, so anything but a contiguous CUDA tensor is rejected here instead of being read
    wrongly (or faulting the GPU)."""
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError(f"libhg takes device memory; got a tensor on {t.device}")
    if not t.is_contiguous():
        raise ValueError(f"libhg reads rows by address; the tensor of shape {tuple(t.shape)} and strides "
                         f"{t.stride()} must be contiguous (call .contiguous())")
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


def _offsets(type_offsets):
    arr = (c_int64 * len(type_offsets))(*[int(x) for x in type_offsets])
    return arr


def _rels(rels):
    arr = (hg_rel_desc * len(rels))(*[hg_rel_desc(int(s), int(t)) for s, t in rels])
    return arr


# ------------------------------------------------------------------------------------------------
# graph
# ------------------------------------------------------------------------------------------------
def hg_graph_workspace_size(num_edges: int, type_offsets, rels) -> int:
    n = c_size_t(0)
    _check(lib().hg_graph_workspace_size(int(num_edges), _offsets(type_offsets), len(type_offsets) - 1, _rels(rels),
                                         len(rels), byref(n)), "hg_graph_workspace_size")
    return n.value


class Graph:
    """Host handle of a built graph; keeps the workspace tensor alive."""

    def __init__(self, handle: c_void_p, workspace: torch.Tensor, type_offsets, rels):
        self.handle = handle
        self.workspace = workspace
        self.type_offsets = [int(x) for x in type_offsets]
        self.rels = [tuple(r) for r in rels]

    @property
    def num_nodes(self) -> int:
        return self.type_offsets[-1]

    def __del__(self):
        if getattr(self, "handle", None) and _lib is not None:
            _lib.hg_graph_destroy(self.handle)
            self.handle = None


def hg_build_csr(src, dst, rel, type_offsets, rels, workspace: torch.Tensor | None = None, stream=None) -> Graph:
    E = int(src.numel())
    need = hg_graph_workspace_size(E, type_offsets, rels)
    if workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=src.device)
    h = c_void_p()
    _check(lib().hg_build_csr(_ptr(src), _ptr(dst), _ptr(rel), E, _offsets(type_offsets), len(type_offsets) - 1,
                              _rels(rels), len(rels), _ptr(workspace), workspace.numel(), _stream(stream), byref(h)),
           "hg_build_csr")
    return Graph(h, workspace, type_offsets, rels)


def hg_graph_destroy(g: Graph):
    if g.handle:
        _check(lib().hg_graph_destroy(g.handle), "hg_graph_destroy")
        g.handle = None


def hg_graph_check(g: Graph) -> int:
    """Synchronises the build stream; returns the number of dropped (invalid) edges."""
    n = c_int64(0)
    st = lib().hg_graph_check(g.handle, byref(n))
    if st not in (0, 5):
        _check(st, "hg_graph_check")
    return n.value


def hg_graph_view(g: Graph, rel: int) -> dict:
    """Device views (torch tensors sharing the workspace) of one relation's CSR / CSC arrays."""
    a = hg_graph_arrays()
    _check(lib().hg_graph_view(g.handle, int(rel), byref(a)), "hg_graph_view")
    ws = g.workspace
    base = ws.data_ptr()

    def view(ptr, n, dtype):
        off = ptr - base
        return ws[off:off + n * 4].view(dtype)

    E = a.num_edges
    return dict(n_dst=a.n_dst, n_src=a.n_src, row_ptr=view(a.row_ptr, a.n_dst + 1, torch.int32),
                col=view(a.col, E, torch.int32), eid=view(a.eid, E, torch.int32),
                csc_ptr=view(a.csc_ptr, a.n_src + 1, torch.int32), csc_col=view(a.csc_col, E, torch.int32),
                csc_eid=view(a.csc_eid, E, torch.int32), csc_coef=view(a.csc_coef, E, torch.float32))


def hg_graph_node_order(g: Graph, node_type: int) -> dict:
    """Device views of the forward projection's node order of one type: perm (position -> local id,
    sorted stably by relation mask) and tile_mask (OR of the masks of each tile of tile_rows rows)."""
    a = hg_node_order()
    _check(lib().hg_graph_node_order(g.handle, int(node_type), byref(a)), "hg_graph_node_order")
    ws = g.workspace
    base = ws.data_ptr()

    def view(ptr, n):
        off = ptr - base
        return ws[off:off + n * 4].view(torch.int32)

    return dict(n=a.n, tiles=a.tiles, tile_rows=a.tile_rows, perm=view(a.perm, a.n),
                tile_mask=view(a.tile_mask, a.tiles))


# ------------------------------------------------------------------------------------------------
# layer
# ------------------------------------------------------------------------------------------------
class LayerParams:
    """Packed device parameters of one layer (see hg_layer_params)."""

    def __init__(self, W_rel, W_agg, b_agg, ln_gamma=None, ln_beta=None, act: str = "relu", layernorm: bool = True,
                 ln_eps: float = 1e-5, fused: bool = False):
        self.W_rel, self.W_agg, self.b_agg = W_rel.contiguous(), W_agg.contiguous(), b_agg.contiguous()
        self.fused = bool(fused)
        self.ln_gamma = ln_gamma.contiguous() if ln_gamma is not None else None
        self.ln_beta = ln_beta.contiguous() if ln_beta is not None else None
        self.act, self.layernorm, self.ln_eps = act, layernorm, ln_eps
        self.d = int(W_rel.shape[-1])
        self.dtype = HG_F32 if W_rel.dtype == torch.float32 else HG_BF16

    def c(self) -> hg_layer_params:
        return hg_layer_params(self.d, self.dtype, ACTS[self.act], 1 if self.layernorm else 0, self.ln_eps,
                               _ptr(self.W_rel), _ptr(self.W_agg), _ptr(self.b_agg), _ptr(self.ln_gamma),
                               _ptr(self.ln_beta), 1 if self.fused else 0)


def hg_layer_workspace_size(g: Graph, params: LayerParams) -> tuple:
    s, k = c_size_t(0), c_size_t(0)
    p = params.c()
    _check(lib().hg_layer_workspace_size(g.handle, byref(p), byref(s), byref(k)), "hg_layer_workspace_size")
    return s.value, k.value


def hg_layer_fwd(g: Graph, params: LayerParams, H_in, H_out, saved, scratch, stream=None):
    p = params.c()
    _check(lib().hg_layer_fwd(g.handle, byref(p), _ptr(H_in), _ptr(H_out), _ptr(saved), _ptr(scratch),
                              _stream(stream)), "hg_layer_fwd")


def hg_layer_bwd(g: Graph, params: LayerParams, H_in, saved, dH_out, dH_in, grads: dict, scratch, stream=None):
    p = params.c()
    gr = hg_layer_grads(_ptr(grads["W_rel"]), _ptr(grads["W_agg"]), _ptr(grads["b_agg"]), _ptr(grads.get("ln_gamma")),
                        _ptr(grads.get("ln_beta")))
    _check(lib().hg_layer_bwd(g.handle, byref(p), _ptr(H_in), _ptr(saved), _ptr(dH_out), _ptr(dH_in), byref(gr),
                              _ptr(scratch), _stream(stream)), "hg_layer_bwd")


# ------------------------------------------------------------------------------------------------
# overlap + alignment
# ------------------------------------------------------------------------------------------------
def hg_overlap_intersect_workspace_size(n_a: int, n_b: int) -> int:
    n = c_size_t(0)
    _check(lib().hg_overlap_intersect_workspace_size(int(n_a), int(n_b), byref(n)), "hg_overlap_intersect_workspace_size")
    return n.value


def hg_overlap_intersect(gid_a, gid_b, idx_a, idx_b, n_out, scratch, stream=None):
    _check(lib().hg_overlap_intersect(_ptr(gid_a), gid_a.numel(), _ptr(gid_b), gid_b.numel(), _ptr(idx_a), _ptr(idx_b),
                                      _ptr(n_out), _ptr(scratch), scratch.numel(), _stream(stream)),
           "hg_overlap_intersect")


def hg_overlap_align_workspace_size(n_max: int, d: int) -> tuple:
    s, k = c_size_t(0), c_size_t(0)
    _check(lib().hg_overlap_align_workspace_size(int(n_max), int(d), byref(s), byref(k)),
           "hg_overlap_align_workspace_size")
    return s.value, k.value


def _dtype_of(t) -> int:
    return HG_F32 if t.dtype == torch.float32 else HG_BF16


def hg_overlap_align_loss(H_a, idx_a, H_b, idx_b, n_max: int, n_dev, lambda_n: float, var_eps: float, loss_out, saved,
                          scratch, stream=None):
    _check(lib().hg_overlap_align_loss(_ptr(H_a), H_a.shape[0], _ptr(idx_a), _ptr(H_b), H_b.shape[0], _ptr(idx_b),
                                       int(n_max), _ptr(n_dev),
                                       int(H_a.shape[-1]), _dtype_of(H_a), float(lambda_n), float(var_eps),
                                       _ptr(loss_out), _ptr(saved), _ptr(scratch), _stream(stream)),
           "hg_overlap_align_loss")


def hg_overlap_align_bwd(H_a, idx_a, H_b, idx_b, n_max: int, n_dev, lambda_n: float, var_eps: float, dloss: float,
                         saved, dH_a, dH_b, scratch, stream=None):
    _check(lib().hg_overlap_align_bwd(_ptr(H_a), H_a.shape[0], _ptr(idx_a), _ptr(H_b), H_b.shape[0], _ptr(idx_b),
                                      int(n_max), _ptr(n_dev),
                                      int(H_a.shape[-1]), _dtype_of(H_a), float(lambda_n), float(var_eps),
                                      float(dloss), _ptr(saved), _ptr(dH_a), _ptr(dH_b), _ptr(scratch),
                                      _stream(stream)), "hg_overlap_align_bwd")


def hg_device_status() -> int:
    """Synchronises; returns the device status flags (0 = no bounded wait gave up) and clears them."""
    f = c_int32(0)
    st = lib().hg_device_status(byref(f))
    if st not in (0, 6):
        _check(st, "hg_device_status")
    return f.value


def hg_selftest_bounded_wait(polls: int, stream=None):
    """One wait on an mbarrier nothing arrives at, giving up after `polls` polls (see hg.h)."""
    _check(lib().hg_selftest_bounded_wait(int(polls), _stream(stream)), "hg_selftest_bounded_wait")


def hg_overlap_align_loss_static(H_a, idx_a, H_b, idx_b, n_max: int, n_dev, lambda_n: float, var_eps: float,
                                 loss_out, saved, stream=None):
    """hg_overlap_align_loss without a scratch argument: the library's own static device array is
    used instead, for callers that cannot allocate (calls must not overlap on the GPU)."""
    _check(lib().hg_overlap_align_loss_static(_ptr(H_a), H_a.shape[0], _ptr(idx_a), _ptr(H_b), H_b.shape[0],
                                              _ptr(idx_b), int(n_max), _ptr(n_dev), int(H_a.shape[-1]),
                                              _dtype_of(H_a), float(lambda_n), float(var_eps), _ptr(loss_out),
                                              _ptr(saved), _stream(stream)), "hg_overlap_align_loss_static")


# ------------------------------------------------------------------------------------------------
# timing
# ------------------------------------------------------------------------------------------------
def hg_timing_enable(on: bool):
    _check(lib().hg_timing_enable(1 if on else 0), "hg_timing_enable")


def hg_timing_report() -> dict:
    """Synchronises; returns {kernel name: (launches, total ms)} since the last report."""
    buf = ctypes.create_string_buffer(1 << 16)
    _check(lib().hg_timing_report(buf, len(buf)), "hg_timing_report")
    out = {}
    for line in buf.value.decode().splitlines():
        name, n, ms = line.split()
        out[name] = (int(n), float(ms))
    return out


# -------------------------------------------------------------------------------------------------
# overlapping subgraph construction
# -------------------------------------------------------------------------------------------------
def hg_overlap_build_workspace_size(num_nodes: int, num_edges: int) -> int:
    n = c_size_t(0)
    _check(lib().hg_overlap_build_workspace_size(int(num_nodes), int(num_edges), byref(n)),
           "hg_overlap_build_workspace_size")
    return n.value


def hg_overlap_build(src, dst, rel, type_offsets, K: int, k: int, theta: int, M: int, part_seed: int,
                     sample_seed: int, workspace=None, with_h: bool = False, stream=None) -> dict:
    """Overlapping subgraph k of K of a global graph (device tensors src, dst, rel; host list
    type_offsets).  Returns device tensors trimmed to the counts (one synchronisation to read them):
    gid, src, dst, rel, eid, type_offsets, h (when with_h), and the counts as a dict."""
    import torch
    dev = src.device
    N, E = int(type_offsets[-1]), int(src.numel())
    T = len(type_offsets) - 1
    if workspace is None:
        workspace = torch.empty(hg_overlap_build_workspace_size(N, E), dtype=torch.uint8, device=dev)
    gid = torch.empty(max(N, 1), dtype=torch.int64, device=dev)
    out = {k2: torch.empty(max(E, 1), dtype=torch.int32, device=dev) for k2 in ("src", "dst", "rel", "eid")}
    toff = torch.empty(T + 1, dtype=torch.int64, device=dev)
    h = torch.empty(max(N, 1), dtype=torch.int32, device=dev) if with_h else None
    counts = torch.empty(6, dtype=torch.int64, device=dev)
    offs = (c_int64 * (T + 1))(*[int(x) for x in type_offsets])
    _check(lib().hg_overlap_build(_ptr(src), _ptr(dst), _ptr(rel), E, N, offs, T, int(K), int(k), int(theta), int(M),
                                  int(part_seed) & (2**64 - 1), int(sample_seed) & (2**64 - 1), _ptr(gid),
                                  _ptr(out["src"]), _ptr(out["dst"]), _ptr(out["rel"]), _ptr(out["eid"]), _ptr(toff),
                                  _ptr(h), _ptr(counts), _ptr(workspace), workspace.numel(), _stream(stream)),
           "hg_overlap_build")
    c = [int(x) for x in counts.cpu()]
    names = ("nodes", "base", "expanded", "edges", "candidates", "filtered")
    res = {"gid": gid[:c[0]], "type_offsets": toff, "counts": dict(zip(names, c))}
    res.update({k2: v[:c[3]] for k2, v in out.items()})
    if with_h:
        res["h"] = h[:N]
    return res



# ------------------------------------------------------------------------------------------------
# prediction head and joint objective
# ------------------------------------------------------------------------------------------------
class HeadParams:
    """Packed device parameters of the two-layer head (see hg_head_params)."""

    def __init__(self, W1, b1, w2, b2):
        self.W1, self.b1, self.w2, self.b2 = W1.contiguous(), b1.contiguous(), w2.contiguous(), b2.contiguous()
        self.d = int(W1.shape[-1])
        self.dtype = HG_F32 if W1.dtype == torch.float32 else HG_BF16

    def c(self) -> hg_head_params:
        return hg_head_params(self.d, self.dtype, _ptr(self.W1), _ptr(self.b1), _ptr(self.w2), _ptr(self.b2))


def hg_head_workspace_size(rows: int, n_lab: int, d: int, dtype) -> tuple:
    s, k = c_size_t(0), c_size_t(0)
    dt = dtype if isinstance(dtype, int) else (HG_F32 if dtype == torch.float32 else HG_BF16)
    _check(lib().hg_head_workspace_size(int(rows), int(n_lab), int(d), dt, byref(s), byref(k)),
           "hg_head_workspace_size")
    return s.value, k.value


def hg_head_loss(params: HeadParams, H, H_rep, idx_a, idx_b, n_rep_max: int, n_rep_dev, lab_idx, lab_y, cca_loss,
                 lambda_cca: float, loss_out, logits, saved, scratch, stream=None):
    p = params.c()
    _check(lib().hg_head_loss(byref(p), _ptr(H), H.shape[0], _ptr(H_rep), H_rep.shape[0] if H_rep is not None else 0,
                              _ptr(idx_a), _ptr(idx_b), int(n_rep_max), _ptr(n_rep_dev), _ptr(lab_idx), _ptr(lab_y),
                              lab_idx.numel(), _ptr(cca_loss), float(lambda_cca), _ptr(loss_out), _ptr(logits),
                              _ptr(saved), _ptr(scratch), _stream(stream)), "hg_head_loss")


def hg_head_bwd(params: HeadParams, lab_idx, dloss: float, saved, dH, dH_rep, grads: dict, scratch, stream=None,
                overwrite: bool = False):
    p = params.c()
    gr = hg_head_grads(_ptr(grads["W1"]), _ptr(grads["b1"]), _ptr(grads["w2"]), _ptr(grads["b2"]))
    _check(lib().hg_head_bwd(byref(p), _ptr(lab_idx), lab_idx.numel(), float(dloss), _ptr(saved), _ptr(dH),
                             dH.shape[0] if dH is not None else 0, _ptr(dH_rep),
                             dH_rep.shape[0] if dH_rep is not None else 0, 1 if overwrite else 0, byref(gr),
                             _ptr(scratch), _stream(stream)), "hg_head_bwd")


# ------------------------------------------------------------------------------------------------
# temporal module
# ------------------------------------------------------------------------------------------------
class TemporalParams:
    """Packed device parameters of the temporal module (see hg_temporal_params); w = context size."""

    def __init__(self, Wa, r, W_i, W_h, b_i, b_h, w: int):
        self.t = [x.contiguous() for x in (Wa, r, W_i, W_h, b_i, b_h)]
        self.d = int(Wa.shape[-1])
        self.w = int(w)
        self.dtype = HG_F32 if Wa.dtype == torch.float32 else HG_BF16

    def c(self) -> hg_temporal_params:
        return hg_temporal_params(self.d, self.w, self.dtype, *(_ptr(x) for x in self.t))


def hg_temporal_workspace_size(n: int, d: int, w: int, dtype) -> tuple:
    s, k = c_size_t(0), c_size_t(0)
    dt = dtype if isinstance(dtype, int) else (HG_F32 if dtype == torch.float32 else HG_BF16)
    _check(lib().hg_temporal_workspace_size(int(n), int(d), int(w), dt, byref(s), byref(k)),
           "hg_temporal_workspace_size")
    return s.value, k.value


def hg_temporal_fwd(params: TemporalParams, X, C, H_out, saved, scratch, stream=None):
    p = params.c()
    _check(lib().hg_temporal_fwd(byref(p), _ptr(X), _ptr(C), X.shape[0], _ptr(H_out), _ptr(saved), _ptr(scratch),
                                 _stream(stream)), "hg_temporal_fwd")


def hg_temporal_bwd(params: TemporalParams, X, C, saved, dH_out, dX, grads: dict, scratch, stream=None):
    p = params.c()
    gr = hg_temporal_grads(*(_ptr(grads[k]) for k in ("Wa", "r", "W_i", "W_h", "b_i", "b_h")))
    _check(lib().hg_temporal_bwd(byref(p), _ptr(X), _ptr(C), X.shape[0], _ptr(saved), _ptr(dH_out), _ptr(dX),
                                 byref(gr), _ptr(scratch), _stream(stream)), "hg_temporal_bwd")


# ------------------------------------------------------------------------------------------------
# attention layer (Heterogeneous Graph Transformer)
# ------------------------------------------------------------------------------------------------
class HgtParams:
    """Packed device parameters of one attention layer (see hg_hgt_params); mu is fp32."""

    def __init__(self, tensors: dict, heads: int, act: str = "relu", layernorm: bool = True, ln_eps: float = 1e-5):
        self.t = {k: (tensors[k].contiguous() if tensors.get(k) is not None else None) for k in HGT_KEYS}
        self.heads, self.act, self.layernorm, self.ln_eps = int(heads), act, layernorm, ln_eps
        self.d = int(self.t["W_K"].shape[-1])
        self.dtype = HG_F32 if self.t["W_K"].dtype == torch.float32 else HG_BF16

    def c(self) -> hg_hgt_params:
        return hg_hgt_params(self.d, self.heads, self.dtype, ACTS[self.act], 1 if self.layernorm else 0, self.ln_eps,
                             *(_ptr(self.t[k]) for k in HGT_KEYS))


def hg_hgt_workspace_size(g: Graph, params: HgtParams) -> tuple:
    s, k = c_size_t(0), c_size_t(0)
    p = params.c()
    _check(lib().hg_hgt_workspace_size(g.handle, byref(p), byref(s), byref(k)), "hg_hgt_workspace_size")
    return s.value, k.value


def hg_hgt_fwd(g: Graph, params: HgtParams, H_in, H_out, saved, scratch, stream=None):
    p = params.c()
    _check(lib().hg_hgt_fwd(g.handle, byref(p), _ptr(H_in), _ptr(H_out), _ptr(saved), _ptr(scratch), _stream(stream)),
           "hg_hgt_fwd")


def hg_hgt_bwd(g: Graph, params: HgtParams, H_in, saved, dH_out, dH_in, grads: dict, scratch, stream=None):
    p = params.c()
    gr = hg_hgt_grads(*(_ptr(grads.get(k)) for k in HGT_KEYS))
    _check(lib().hg_hgt_bwd(g.handle, byref(p), _ptr(H_in), _ptr(saved), _ptr(dH_out), _ptr(dH_in), byref(gr),
                            _ptr(scratch), _stream(stream)), "hg_hgt_bwd")
