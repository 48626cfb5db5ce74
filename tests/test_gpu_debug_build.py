"""The debug library (-DSADMM_DEBUG, loaded when SADMM_DEBUG=1): every global
load and store of the forward, sparse and backward kernels checks its index
against the buffer's extent; a failed check skips the access and raises
SADMM_EBOUNDS.

Each test runs in a child process, since a process loads one library.  The
first runs the parity suites of those kernels on the debug library (their own
status checks must stay clear).  The second corrupts one gather-table entry of
a packed plan so that column 0 addresses past the end of x: x is the first half
of a buffer twice its size, so even an unchecked load would stay inside the
allocation; the debug library must skip those loads and report SADMM_EBOUNDS,
and the context must stay usable for the next forward.
"""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
TESTS = os.path.join(ROOT, "tests")


def _env():
    env = dict(os.environ)
    env["SADMM_DEBUG"] = "1"
    env["PYTHONPATH"] = os.pathsep.join([ROOT, TESTS, env.get("PYTHONPATH", "")])
    return env


def test_parity_suites_pass_on_the_debug_library():
    files = ["test_gpu_conv.py", "test_gpu_slab.py", "test_gpu_sparse.py", "test_gpu_backward.py",
             "test_gpu_splitk.py"]
    cmd = [sys.executable, "-m", "pytest", "-q", "-x", "-m", "gpu", "-p", "no:cacheprovider"]
    cmd += [os.path.join(TESTS, f) for f in files]
    r = subprocess.run(cmd, cwd=ROOT, env=_env(), capture_output=True, text=True, timeout=1800)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-2000:]


_BAD_OFFSET = r"""
import numpy as np, torch
import workloads as wl
from workloads import ConvShape
from paper_1807_11091_gb300 import sadmm
assert sadmm.library_path().endswith(("debug/libsadmm.so", "debug\\libsadmm.so")), sadmm.library_path()
dev = torch.device("cuda", 0)
s = ConvShape(n=2, c=8, h=12, w=11, f=24, kh=3, kw=3, ph=1, pw=1)
t = wl.gen_tensors(s, seed=41)
W = t["W"].to(dev)
nx = t["x"].numel()
big = torch.zeros(2 * nx + 4096, dtype=torch.bfloat16, device=dev)
x = big[:nx].view(t["x"].shape)
x.copy_(t["x"].to(dev))
bias = t["bias"].to(dev)
fi, ci, _ = sadmm.project_groups(s.desc16(), W, s.f, wl.COL_SHAPE, wl.retained(0.5, s.k))
pc = sadmm.PrunedConv(s.desc16(), W, None, wl.COL_SHAPE, ci, s.f, wl.retained(0.5, s.k))
assert pc.plan.xs_mode == 0
y0 = pc.forward(x, bias)
assert sadmm.device_status() == sadmm.SADMM_OK
entry = pc.buf[pc.plan.off_gather:pc.plan.off_gather + 8].view(torch.int32)
good = entry.clone()
entry[0] += nx  # column 0 now addresses x + nx .. (inside big, outside x)
y1 = pc.forward(x, bias)
st = sadmm.device_status()
assert st == sadmm.SADMM_EBOUNDS, st
entry.copy_(good)
y2 = pc.forward(x, bias)
assert sadmm.device_status() == sadmm.SADMM_OK
assert torch.equal(y0, y2)
print("OK")
"""


def test_debug_library_reports_an_index_past_x():
    r = subprocess.run([sys.executable, "-c", _BAD_OFFSET], cwd=ROOT, env=_env(), capture_output=True, text=True,
                       timeout=900)
    assert r.returncode == 0 and r.stdout.strip().endswith("OK"), r.stdout[-3000:] + r.stderr[-3000:]
