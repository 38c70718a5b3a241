"""Every row of the block output at the d=3072 workloads against the oracle.

The configuration tests compare sampled rows at d=3072; here the oracle
computes the whole block (fp64, all text and packed image rows of every
image) and each output row of the GPU path is compared with it, element by
element, within the block tolerance (max-abs 2e-2, rel-L2 1e-2). The GPU
runs exactly as bench.py launches it (HotPath: score -> split -> pack ->
block -> unpack), so the GEMMs' stream-K tail tiles (out-projection and MLP2),
the ragged last 256-row tile of each weight group and the ragged attention
tiles are all inside the compared range.

Workloads: the 64x64 grid (512 text tokens, d=3072, 24 heads of 128, 4x MLP)
at keep ratios 1/4 and 1/10, the batch of four 64x64 images with varying
keep ratios, and the 128x128 grid with two-level pooling.
"""
import numpy as np
import pytest

from oracle import hilo_oracle as O
from paper_2606_13898_gb300 import inputs as I

from .gpu_helpers import assert_block_close, lib_ready
from .test_gpu_configs import check_split_pack, run_path

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def H():
    return lib_ready()


def check_all_rows(H, wl):
    batch = I.make_batch(wl)
    w = I.make_weights(wl.d, wl.mlp, seed=I.weight_seed(wl))
    hp = run_path(H, wl, batch, [H.DeviceWeights.from_host(w)])
    sp, packed = check_split_pack(H, hp, wl, batch)
    rows = int(sp.cu_img[-1])
    BT = wl.B * wl.T
    got = hp.out.cpu().numpy()
    ot, oi = O.block(batch.text.reshape(BT, wl.d), packed, sp.cu_img, wl.T, O.weights_f64(w), wl.heads, wl.mlp)
    for b in range(wl.B):
        t0, t1 = b * wl.T, (b + 1) * wl.T
        i0, i1 = int(sp.cu_img[b]), int(sp.cu_img[b + 1])
        assert_block_close(got[t0:t1], ot[t0:t1], f"{wl.name} image {b}: all {wl.T} text rows")
        assert_block_close(got[BT + i0:BT + i1], oi[i0:i1], f"{wl.name} image {b}: all {i1 - i0} image rows")
    # the unpacked grid is the gather of these rows
    y = hp.y.cpu().numpy().reshape(wl.B, wl.N, wl.d)
    assert np.array_equal(y, got[BT:BT + rows][sp.tok_row])
    return rows


@pytest.mark.parametrize("ratio", ["1/4", "1/10"])
def test_block64_every_row(H, ratio):
    rows = check_all_rows(H, I.block_64(keep_ratio=ratio))
    assert rows > 256 * 4   # several 256-row tiles plus a ragged one


def test_block64_batch4_every_row(H):
    check_all_rows(H, I.block_64_batch4())


def test_block128_two_level_every_row(H):
    check_all_rows(H, I.block_128_two_level())
