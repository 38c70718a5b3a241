"""The multi-GPU arrangement (independent replicas, sharded by image) on the CPU.

Two gloo ranks split a global batch of four images with `image_slice`, each
runs the oracle's hot path on its own slice, and rank 0 gathers the outputs:
they equal, bit for bit, one process running the whole batch, which is what
makes the path shard with no exchange step. The timing helpers
(max-over-ranks, whole-job throughput) run under the same process group.
"""
import dataclasses
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2606_13898_gb300 import inputs as I
from paper_2606_13898_gb300 import replicas as R

WL = I.Workload(name="gloo_4x8x8", B=4, H=8, W=8, d=128, T=8, heads=1, mlp=True, levels=1, mask_lo=0.1,
                mask_hi=0.3, keep_ratio="1/4")


def _oracle_run(wl, seed_offset):
    from oracle import hilo_oracle as O
    b = I.make_batch(wl, seed_offset=seed_offset)
    w = I.make_weights(wl.d, wl.mlp, seed=I.weight_seed(wl))
    sp, packed, (ut, ui), y = O.hot_path(b.x, b.text, b.mask, b.k_keep, b.k_mid, wl.levels, [w], wl.heads,
                                         wl.mlp)
    return np.asarray(y, dtype=np.float64).reshape(wl.B, -1), np.asarray(ut, dtype=np.float64).reshape(wl.B, -1)


def _worker(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        b0, b1 = R.image_slice(WL.B, rank, world)
        y, txt = _oracle_run(dataclasses.replace(WL, B=b1 - b0), seed_offset=b0)
        gy = [torch.empty(b1 - b0, y.shape[1], dtype=torch.float64) for _ in range(world)]
        gt = [torch.empty(b1 - b0, txt.shape[1], dtype=torch.float64) for _ in range(world)]
        dist.all_gather(gy, torch.from_numpy(y))
        dist.all_gather(gt, torch.from_numpy(txt))
        slowest = R.max_over_ranks(10.0 + rank, device="cpu")
        thr = R.whole_job_throughput((b1 - b0) * WL.N, dist.get_world_size(), slowest)
        if rank == 0:
            np.save(out + "_y.npy", torch.cat(gy).numpy())
            np.save(out + "_t.npy", torch.cat(gt).numpy())
            np.save(out + "_m.npy", np.array([slowest, thr]))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_image_slices_cover_the_batch():
    for n in (0, 1, 4, 7, 8):
        for world in (1, 2, 3, 8):
            sl = [R.image_slice(n, r, world) for r in range(world)]
            assert sl[0][0] == 0 and sl[-1][1] == n
            assert all(sl[r][1] == sl[r + 1][0] for r in range(world - 1))
            sizes = [b1 - b0 for b0, b1 in sl]
            assert max(sizes) - min(sizes) <= 1
    with pytest.raises(ValueError):
        R.image_slice(4, 2, 2)


def test_throughput_helpers_single_process():
    assert R.max_over_ranks(3.5) == 3.5  # no process group: the value itself
    assert R.whole_job_throughput(4096, 2, 0.5) == pytest.approx(4096 * 2 / 0.5e-3)


def test_two_gloo_ranks_equal_one_process(tmp_path):
    out = str(tmp_path / "r")
    mp.spawn(_worker, args=(2, _free_port(), out), nprocs=2, join=True)
    y_ref, t_ref = _oracle_run(WL, seed_offset=0)
    y = np.load(out + "_y.npy")
    t = np.load(out + "_t.npy")
    assert np.array_equal(y, y_ref) and np.array_equal(t, t_ref)
    slowest, thr = np.load(out + "_m.npy")
    assert slowest == 11.0
    assert thr == pytest.approx(2 * 2 * WL.N / 11.0e-3)
