"""The checks build: every index a bandwidth kernel reads from device data is
range-checked before use (a stand-in for a memory checker, which this pool
does not offer).

1. The split, pack, unpack and row-size parity tests run again in a child
   process on the checks build (HILO_LIBRARY); the autouse fixture of
   conftest reads the check word after each test, so any failed check fails
   the run.
2. A planted out-of-range token row is caught: the kernel records the check
   and skips the row. The output buffer carries spare rows past the row
   capacity, so even an unguarded read would stay inside its allocation.
"""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_parity_tests_pass_on_checks_build():
    from paper_2606_13898_gb300 import build
    lib = build.build(variant="checks")
    env = dict(os.environ, HILO_LIBRARY=lib)
    cmd = [sys.executable, "-m", "pytest", "-q", "-x", "-m", "gpu", "-p", "no:cacheprovider",
           "tests/test_gpu_kernels.py", "tests/test_gpu_regions.py", "tests/test_gpu_lf.py",
           "-k", "(score or split or pack or unpack or row_sizes or regions or delta or lf) and not block"]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=1800)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-2000:]
    assert " passed" in r.stdout


CHILD = r"""
import numpy as np, torch
from paper_2606_13898_gb300 import hilo as H
assert H.library_path().endswith("_build_checks/libhilo.so"), H.library_path()
H.lib()
sh = H.Shape(B=1, H=8, W=8, d=128)
sp = H.SplitBuffers.alloc(sh)
rows = H.hilo_row_capacity(sh)
out = torch.zeros((rows + 16) * 128, dtype=torch.float32, device="cuda")
out[: rows * 128] = 1.0
tok = torch.arange(64, dtype=torch.int32, device="cuda") % rows
tok[5] = rows  # one past the row capacity
sp.tok_row.copy_(tok)
y = torch.full((64 * 128,), -1.0, dtype=torch.float32, device="cuda")
H.hilo_unpack(sh, out, sp, y)
try:
    H.hilo_sync_status()
    raise SystemExit("no check fired")
except H.HiloError as e:
    assert e.status == H.HILO_ERR_CHECK and "check 4" in str(e), str(e)
yy = y.view(64, 128).cpu().numpy()
assert np.all(yy[5] == -1.0)  # the bad row was skipped
assert np.all(np.delete(yy, 5, axis=0) == 1.0)
H.hilo_sync_status()  # cleared
print("planted check ok")
"""


def test_planted_bad_token_row_is_caught():
    from paper_2606_13898_gb300 import build
    lib = build.build(variant="checks")
    env = dict(os.environ, HILO_LIBRARY=lib)
    r = subprocess.run([sys.executable, "-c", CHILD], cwd=ROOT, env=env, capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0 and "planted check ok" in r.stdout, r.stdout[-3000:] + r.stderr[-3000:]
