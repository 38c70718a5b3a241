"""The device-side failure path: a bounded wait that runs out is reported, not hung.

The probe kernel waits, with the bounded mbarrier wait the tcgen05 kernels
use, on an mbarrier that nothing arrives at. After the 1 s device limit the
wait latches its code and the kernel returns; hilo_sync_status reports
HILO_ERR_TIMEOUT once and clears the word, and the context keeps working.
Nothing here faults, traps or hangs the GPU.
"""
import time

import numpy as np
import pytest
import torch

from oracle import hilo_oracle as O
from paper_2606_13898_gb300 import inputs as I

from .gpu_helpers import lib_ready

pytestmark = pytest.mark.gpu


def test_wait_timeout_is_reported_and_context_survives():
    H = lib_ready()
    H.hilo_sync_status()  # no stale code from earlier tests
    t0 = time.perf_counter()
    H.hilo_debug_wait_timeout()
    with pytest.raises(H.HiloError) as ei:
        H.hilo_sync_status()
    dt = time.perf_counter() - t0
    assert ei.value.status == -5  # HILO_ERR_TIMEOUT
    assert "probe=3" in str(ei.value)
    assert 0.9 < dt < 30.0  # the 1 s device limit, not an immediate or endless wait
    # the word was cleared, and the context still runs and gets results right
    H.hilo_sync_status()
    rng = np.random.default_rng(7)
    x = I.f32_to_bf16_bits(rng.standard_normal((1, 8, 8, 256)).astype(np.float32))
    sh = H.Shape(B=1, H=8, W=8, d=256)
    s = torch.empty(64, dtype=torch.float32, device="cuda")
    H.hilo_score(sh, H.bf16_from_bits(x), s)
    H.hilo_sync_status()
    ref = O.score(x)
    assert np.array_equal(s.cpu().numpy().reshape(ref.shape).view(np.uint32), ref.view(np.uint32))
