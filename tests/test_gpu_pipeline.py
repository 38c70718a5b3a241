"""PipelinedHotPath: host batches through the hot path with overlapped copies.

Each result copied back to the host must equal y from HotPath.run on the
same inputs, batch by batch, whatever the overlap of copies and kernels.
The 32x32 layer (no stream-K accumulation) is deterministic, so y is
compared bit for bit.
"""
import numpy as np
import pytest
import torch

from paper_2606_13898_gb300 import inputs as I

from .gpu_helpers import lib_ready

pytestmark = pytest.mark.gpu


def _host(batch):
    return (torch.from_numpy(batch.x.view(np.int16)).view(torch.bfloat16).pin_memory(),
            torch.from_numpy(batch.text.view(np.int16)).view(torch.bfloat16).pin_memory(),
            torch.from_numpy(batch.mask).pin_memory(),
            torch.from_numpy(batch.k_keep).pin_memory(),
            torch.from_numpy(batch.k_mid).pin_memory())


def test_pipeline_matches_hot_path_per_batch():
    H = lib_ready()
    wl = I.tiny_layer()
    w = I.make_weights(wl.d, wl.mlp, seed=I.weight_seed(wl))
    dw = H.DeviceWeights.from_host(w)
    sh = H.Shape(B=wl.B, H=wl.H, W=wl.W, d=wl.d, T=wl.T, heads=wl.heads, mlp=int(wl.mlp), levels=wl.levels)
    batches = [_host(I.make_batch(wl, seed_offset=s)) for s in range(5)]
    ys = [torch.empty(wl.B, wl.H, wl.W, wl.d, dtype=torch.float32).pin_memory() for _ in batches]
    pipe = H.PipelinedHotPath(sh, [dw], batches[0])
    for hin, yh in zip(batches, ys):
        pipe.submit(hin, yh)
    pipe.drain()
    torch.cuda.synchronize()
    H.hilo_sync_status()
    hp = H.HotPath(sh, [dw])
    for hin, yh in zip(batches, ys):
        dev = [t.cuda() for t in hin]
        hp.run(*dev)
        torch.cuda.synchronize()
        assert torch.equal(hp.y.cpu(), yh)
    assert not torch.equal(ys[0], ys[1])
