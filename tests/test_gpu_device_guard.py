"""The library binds itself to one device per process: a call made with another device current is
refused (HG_ERR_UNSUPPORTED) before any kernel is launched.  A single-GPU machine cannot make another
device current, so the test binds the library to an ordinal other than the current one (in a fresh
process, whose library state is not yet bound) and checks that kernel-launching entry points then
refuse to run and launch nothing."""
import os
import subprocess
import sys

import pytest

from tests.gpu_util import need_gpu

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import ctypes, sys
import torch
sys.path.insert(0, ROOT)
from paper_2608_02168_gb300 import hg
so = hg.lib()
cur = torch.cuda.current_device()
assert so.hg_bind_device(cur + 1) == 0
assert so.hg_bind_device(cur + 1) == 0        # the same device again: accepted
assert so.hg_bind_device(cur) == 2            # another one: refused
hg.hg_timing_enable(True)
x = torch.zeros(64, 64, dtype=torch.float32, device="cuda")
i = torch.zeros(2, dtype=torch.int32, device="cuda")
loss = torch.zeros(3, dtype=torch.float32, device="cuda")
s, k = hg.hg_overlap_align_workspace_size(2, 64)
saved = torch.empty(s, dtype=torch.uint8, device="cuda")
scratch = torch.empty(k, dtype=torch.uint8, device="cuda")
p = lambda t: ctypes.c_void_p(t.data_ptr())
st = so.hg_overlap_align_loss(p(x), 64, p(i), p(x), 64, p(i), 2, None, 64, 0, ctypes.c_float(2e-4),
                              ctypes.c_float(1e-8), p(loss), p(saved), p(scratch), None)
assert st == 2, st
assert b"bound to device" in so.hg_last_error()
st = so.hg_overlap_align_loss_static(p(x), 64, p(i), p(x), 64, p(i), 2, None, 64, 0, ctypes.c_float(2e-4),
                                     ctypes.c_float(1e-8), p(loss), p(saved), None)
assert st == 2, st
flags = ctypes.c_int32(0)
assert so.hg_device_status(ctypes.byref(flags)) == 2
torch.cuda.synchronize()
assert hg.hg_timing_report() == {}, "a refused call launched a kernel"
print("ok")
"""


def test_calls_on_another_device_are_refused_before_any_launch():
    need_gpu()
    from tests.gpu_util import lib
    lib()  # built in this process; the child loads the same library
    r = subprocess.run([sys.executable, "-c", CHILD.replace("ROOT", repr(ROOT))], capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0 and r.stdout.strip().endswith("ok"), r.stdout + r.stderr
