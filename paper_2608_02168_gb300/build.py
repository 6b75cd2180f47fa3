"""Build libhg.so, the C-ABI library of the hot path, for sm_103a (GB300) with nvcc.

Each csrc/*.cu file is compiled in parallel to an object file, then linked into
paper_2608_02168_gb300/_build/libhg.so (in-tree, git-ignored).  Objects are rebuilt when their
source or any header is newer.  Run as `python -m paper_2608_02168_gb300.build`.
Set HG_PTXAS_VERBOSE=1 to print register / shared-memory usage per kernel.
"""
from __future__ import annotations

import concurrent.futures
import glob
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "csrc")
OUT = os.path.join(HERE, "_build")
INCLUDE = os.path.join(os.path.dirname(HERE), "include")
LIB = os.path.join(OUT, "libhg.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
CFLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
          "-I" + INCLUDE, "-I" + SRC]


def nvcc() -> str:
    path = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(path):
        raise RuntimeError("nvcc not found (CUDA toolkit required to build libhg.so)")
    return path


def library_path() -> str:
    return LIB


def _headers_mtime() -> float:
    hs = glob.glob(os.path.join(SRC, "*.cuh")) + glob.glob(os.path.join(INCLUDE, "*.h"))
    return max((os.path.getmtime(h) for h in hs), default=0.0)


def _compile(src: str, obj: str, verbose: bool) -> str:
    cmd = [nvcc(), *ARCH, *CFLAGS, "-c", src, "-o", obj]
    if verbose:
        cmd += ["-Xptxas", "-v"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {os.path.basename(src)}:\n{r.stdout}\n{r.stderr}")
    return r.stderr


def build(force: bool = False, verbose: bool | None = None) -> str:
    """Compile and link libhg.so if anything changed; returns the library path."""
    if verbose is None:
        verbose = os.environ.get("HG_PTXAS_VERBOSE", "0") == "1"
    os.makedirs(OUT, exist_ok=True)
    hdr = _headers_mtime()
    jobs = []
    for src in sorted(glob.glob(os.path.join(SRC, "*.cu"))):
        obj = os.path.join(OUT, os.path.basename(src)[:-3] + ".o")
        stale = force or verbose or not os.path.exists(obj) or os.path.getmtime(obj) < max(os.path.getmtime(src), hdr)
        jobs.append((src, obj, stale))
    todo = [(s, o) for s, o, st in jobs if st]
    if todo:
        with concurrent.futures.ThreadPoolExecutor(max_workers=min(len(todo), os.cpu_count() or 4)) as ex:
            for (s, _), log in zip(todo, ex.map(lambda so: _compile(so[0], so[1], verbose), todo)):
                if verbose and log:
                    sys.stderr.write(f"== {os.path.basename(s)}\n{log}")
    objs = [o for _, o, _ in jobs]
    if todo or not os.path.exists(LIB) or os.path.getmtime(LIB) < max(os.path.getmtime(o) for o in objs):
        tmp = LIB + ".tmp"
        r = subprocess.run([nvcc(), *ARCH, "-shared", "-o", tmp, *objs], capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link of libhg.so failed:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
