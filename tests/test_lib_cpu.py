"""The C-ABI library loads, exports every entry point include/hg.h declares, and rejects bad
arguments on the host before touching the GPU (CPU only: no compute call is made)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def hg():
    from paper_2608_02168_gb300 import build
    build.build()
    from paper_2608_02168_gb300 import hg as binding
    return binding


def declared_functions():
    text = open(os.path.join(ROOT, "include", "hg.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\*?\s+(hg_\w+)\s*\(", text, flags=re.M)))


def test_every_declared_symbol_is_exported(hg):
    names = declared_functions()
    assert len(names) >= 17, names
    so = hg.lib()
    for n in names:
        assert hasattr(so, n), n
    assert set(names) == set(hg.EXPORTS), "binding and header disagree"


def test_status_strings_and_version(hg):
    so = hg.lib()
    assert so.hg_abi_version() == 2  # hg_layer_params gained `fused`
    assert so.hg_status_string(0) == b"ok"
    assert so.hg_status_string(3) == b"workspace too small"


def test_workspace_queries_are_host_only(hg):
    n = hg.hg_graph_workspace_size(1000, [0, 80, 100], [(0, 0), (0, 1), (1, 0)])
    assert n > 1000 * 4 * 7
    s, k = hg.hg_overlap_align_workspace_size(500, 64)
    assert s >= 4 * 64 * 4 + 2 * 64 * 64 * 4 and k > 2 * 500 * 64 * 4
    assert hg.hg_overlap_intersect_workspace_size(10, 20) > 0


def test_host_argument_checks(hg):
    so = hg.lib()
    offs = (ctypes.c_int64 * 3)(0, 8, 10)
    rels = (hg.hg_rel_desc * 1)(hg.hg_rel_desc(0, 1))
    out = ctypes.c_void_p()
    # null edge arrays with edges
    assert so.hg_build_csr(None, None, None, 5, offs, 2, rels, 1, 256, 1 << 20, None, ctypes.byref(out)) == 1
    # too many relation types
    assert so.hg_graph_workspace_size(5, offs, 2, rels, 9, ctypes.byref(ctypes.c_size_t())) == 2
    # edge count beyond int32
    assert so.hg_graph_workspace_size(1 << 31, offs, 2, rels, 1, ctypes.byref(ctypes.c_size_t())) == 2
    # bounded-wait self-test: poll count out of range
    assert so.hg_selftest_bounded_wait(0, None) == 1 and so.hg_selftest_bounded_wait((1 << 20) + 1, None) == 1
    # a relation pointing at a type that does not exist
    bad = (hg.hg_rel_desc * 1)(hg.hg_rel_desc(0, 2))
    assert so.hg_graph_workspace_size(5, offs, 2, bad, 1, ctypes.byref(ctypes.c_size_t())) == 1
    assert b"type out of range" in so.hg_last_error()
    # workspace smaller than the query (fake aligned address: rejected before any device access)
    assert so.hg_build_csr(256, 256, 256, 5, offs, 2, rels, 1, 256, 16, None, ctypes.byref(out)) == 3
    # unsupported feature width for the alignment
    assert so.hg_overlap_align_loss(256, 10, 256, 256, 10, 256, 4, None, 96, 0, 0.0, 0.0, 256, 256, 256, None) == 2
    # negative overlap size; empty tables with a non-empty overlap
    assert so.hg_overlap_align_loss(256, 10, 256, 256, 10, 256, -1, None, 64, 0, 0.0, 0.0, 256, 256, 256, None) == 1
    assert so.hg_overlap_align_bwd(256, 0, 256, 256, 10, 256, 4, None, 64, 0, 0.0, 0.0, 1.0, 256, 256, None, 256,
                                   None) == 1
    # unsorted ids are a device-side condition; a null n_out is a host one
    assert so.hg_overlap_intersect(256, 4, 256, 4, 256, 256, None, 256, 1 << 20, None) == 1


def test_timing_report_empty(hg):
    hg.hg_timing_enable(True)
    assert hg.hg_timing_report() == {}
    hg.hg_timing_enable(False)


def test_product_path_has_no_fallback():
    """The binding and step driver import neither the oracle nor any CPU implementation."""
    pkg = os.path.join(ROOT, "paper_2608_02168_gb300")
    for f in os.listdir(pkg):
        if f.endswith(".py"):
            src = open(os.path.join(pkg, f)).read()
            assert "oracle" not in src.replace("oracle.", ""), f
            assert "import numpy" not in src, f


def test_host_argument_checks_of_the_widened_rows(hg):
    """Head, temporal module, attention layer and subgraph construction reject bad arguments on
    the host (fake aligned addresses stand in for device buffers: nothing is dereferenced)."""
    so = hg.lib()
    A = 1 << 20  # a 256-byte-aligned stand-in address
    # head: unsupported width, misaligned weights, null loss output, negative sizes
    p = hg.hg_head_params(96, 1, A, A, A, A)
    assert so.hg_head_loss(ctypes.byref(p), A, 10, None, 0, None, None, 0, None, A, A, 4, None, 0.1, A, None, A, A,
                           None) == 2
    p = hg.hg_head_params(64, 1, A + 2, A, A, A)
    assert so.hg_head_loss(ctypes.byref(p), A, 10, None, 0, None, None, 0, None, A, A, 4, None, 0.1, A, None, A, A,
                           None) == 1
    p = hg.hg_head_params(64, 1, A, A, A, A)
    assert so.hg_head_loss(ctypes.byref(p), A, 10, None, 0, None, None, 0, None, A, A, 4, None, 0.1, None, None, A, A,
                           None) == 1
    assert so.hg_head_loss(ctypes.byref(p), A, 10, None, 0, None, None, 0, None, A, A, -1, None, 0.1, A, None, A, A,
                           None) == 1
    gr = hg.hg_head_grads(A, A, None, A)
    assert so.hg_head_bwd(ctypes.byref(p), A, 4, 1.0, A, A, 10, None, 0, 0, ctypes.byref(gr), A, None) == 1
    # temporal: window out of range, unsupported width, null pointers with rows
    t = hg.hg_temporal_params(64, 9, 1, A, A, A, A, A, A)
    assert so.hg_temporal_fwd(ctypes.byref(t), A, A, 10, A, A, A, None) == 1
    t = hg.hg_temporal_params(80, 3, 1, A, A, A, A, A, A)
    assert so.hg_temporal_fwd(ctypes.byref(t), A, A, 10, A, A, A, None) == 2
    t = hg.hg_temporal_params(64, 3, 1, A, A, A, A, A, A)
    assert so.hg_temporal_fwd(ctypes.byref(t), None, A, 10, A, A, A, None) == 1
    assert so.hg_temporal_workspace_size(10, 64, 0, 1, ctypes.byref(ctypes.c_size_t()),
                                         ctypes.byref(ctypes.c_size_t())) == 1
    # attention layer: heads not a power of two, null graph
    h = hg.hg_hgt_params(128, 3, 1, 0, 1, 1e-5, *([A] * 13))
    assert so.hg_hgt_workspace_size(A, ctypes.byref(h), ctypes.byref(ctypes.c_size_t()),
                                    ctypes.byref(ctypes.c_size_t())) == 1
    h = hg.hg_hgt_params(128, 4, 1, 0, 1, 1e-5, *([A] * 13))
    assert so.hg_hgt_fwd(None, ctypes.byref(h), A, A, A, A, None) == 1
    # construction: partition index out of range
    offs = (ctypes.c_int64 * 3)(0, 8, 10)
    assert so.hg_overlap_build(A, A, A, 5, 10, offs, 2, 4, 4, 2, 3, 1, 2, A, A, A, A, A, A, None, A, A, 1 << 30,
                               None) == 1


def test_widened_workspace_queries_are_host_only(hg):
    import torch
    s, k = hg.hg_head_workspace_size(1000, 100, 128, torch.bfloat16)
    assert s >= 2 * 100 * 128 * 2 and k >= 1000 * 4
    s, k = hg.hg_temporal_workspace_size(1000, 128, 3, torch.bfloat16)
    assert s >= 1000 * 128 * 2 + 1000 * 3 * 4 and k >= 4 * 1000 * 128 * 2
    s2, k2 = hg.hg_temporal_workspace_size(1000, 256, 3, torch.bfloat16)  # CUDA-core path: fp32 scratch
    assert k2 > k
    assert hg.hg_overlap_build_workspace_size(1000, 5000) > 5000 * 4


def test_binding_rejects_host_tensors_before_any_call(hg):
    """The binding passes device addresses only: a host tensor is refused on the host, before the
    library sees it (a host address handed to a kernel would fault or read the wrong memory)."""
    import torch
    a = torch.arange(8, dtype=torch.int64)
    out = torch.empty(8, dtype=torch.int32)
    with pytest.raises(ValueError, match="device memory"):
        hg.hg_overlap_intersect(a, a, out, out, torch.empty(1, dtype=torch.int64), torch.empty(64, dtype=torch.uint8))
    assert hg._ptr(None) is None


def test_device_binding_is_first_come_and_exclusive(hg):
    """hg_bind_device makes no CUDA call: it is checked here without a GPU, in a fresh process whose
    library state is unbound."""
    import subprocess
    import sys
    child = (f"import ctypes; so = ctypes.CDLL({hg.lib()._name!r}); "
             "assert so.hg_bind_device(3) == 0; assert so.hg_bind_device(3) == 0; "
             "assert so.hg_bind_device(1) == 2; assert so.hg_bind_device(-1) == 1; print('ok')")
    r = subprocess.run([sys.executable, "-c", child], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0 and r.stdout.strip() == "ok", r.stdout + r.stderr


def test_binding_structs_match_the_header(hg, tmp_path):
    """Every ctypes struct of the binding has the size and field offsets the C compiler gives the
    struct of the same name in include/hg.h (the argument structs cross the ABI by pointer)."""
    import shutil
    import subprocess
    if shutil.which("gcc") is None:
        pytest.skip("no C compiler")
    structs = [c for c in vars(hg).values()
               if isinstance(c, type) and issubclass(c, ctypes.Structure) and c.__name__.startswith("hg_")]
    assert any(c.__name__ == "hg_layer_params" for c in structs)
    lines = ['#include <stddef.h>', '#include <stdio.h>', '#include "hg.h"', "int main(void) {"]
    for c in structs:
        lines.append(f'  printf("{c.__name__} size %zu\\n", sizeof({c.__name__}));')
        for f in c._fields_:
            lines.append(f'  printf("{c.__name__} {f[0]} %zu\\n", offsetof({c.__name__}, {f[0]}));')
    lines.append("  return 0;\n}")
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True)
    got = {}
    for line in subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.splitlines():
        name, field, val = line.split()
        got[(name, field)] = int(val)
    for c in structs:
        assert got[(c.__name__, "size")] == ctypes.sizeof(c), c.__name__
        for f in c._fields_:
            assert got[(c.__name__, f[0])] == getattr(c, f[0]).offset, (c.__name__, f[0])
