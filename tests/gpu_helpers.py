"""Shared helpers of the GPU parity tests (device setup, comparisons)."""
from __future__ import annotations

import numpy as np
import torch

# Block-output tolerance: bf16 tensor-core compute against the fp64 oracle.
MAX_ABS = 2e-2
REL_L2 = 1e-2


def lib_ready():
    """Build (if stale) and load libhilo; GPU tests fail loudly without it."""
    from paper_2606_13898_gb300 import build
    from paper_2606_13898_gb300 import hilo as H

    build.build()
    H.lib()
    n, is103 = H.hilo_device_info()
    assert is103 == 1, "libhilo needs an sm_103 device"
    return H


def close_report(got, ref):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    err = got - ref
    max_abs = float(np.abs(err).max()) if err.size else 0.0
    den = float(np.linalg.norm(ref))
    rel = float(np.linalg.norm(err) / den) if den > 0 else float(np.linalg.norm(err))
    return max_abs, rel


def assert_block_close(got, ref, what=""):
    max_abs, rel = close_report(got, ref)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    assert max_abs <= MAX_ABS and rel <= REL_L2, f"{what}: max_abs={max_abs:.3e} rel_l2={rel:.3e}"
    return max_abs, rel


def to_dev_u8(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def to_dev_i32(a):
    return torch.from_numpy(np.ascontiguousarray(np.asarray(a, dtype=np.int32))).cuda()


def to_dev_f32(a):
    return torch.from_numpy(np.ascontiguousarray(np.asarray(a, dtype=np.float32))).cuda()
