"""The paper's Sobel selector on the GPU against the oracle (Sec. 2.3).

The keep map must equal the oracle's bit for bit: every step of the
magnitude, the token maxima, the normalising division and the strict
threshold comparison are defined as correctly rounded fp32 operations on
both sides. Sizes cover partial pixel tiles, both patch sizes, 1 to 4
channels and the 64 x 64-token (1024 x 1024 pixel) image of the timed
workload; the whole hot path is then run with the selector's keep map in
place of the top-k budget.
"""
import numpy as np
import pytest
import torch

from oracle import hilo_oracle as O
from paper_2606_13898_gb300 import inputs as I

from .gpu_helpers import assert_block_close, lib_ready

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def H():
    return lib_ready()


def run_select(H, img, mask, Hh, W, patch, radius, thr):
    B, C = img.shape[0], img.shape[3]
    sh = H.Shape(B=B, H=Hh, W=W, d=128)
    ws_bytes = H.hilo_sobel_workspace_bytes(sh)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    keep = torch.full((B, Hh * W), 7, dtype=torch.uint8, device="cuda")
    H.hilo_sobel_select(sh, torch.from_numpy(img).cuda(), C, patch, torch.from_numpy(mask).cuda(), radius, thr,
                        keep, ws, ws_bytes)
    H.hilo_sync_status()
    return keep.cpu().numpy()


@pytest.mark.parametrize("B,Hh,W,patch,C,radius,thr", [
    (1, 8, 8, 16, 3, 1, 0.1),
    (2, 10, 6, 8, 1, 0, 0.3),    # partial 32 x 64 pixel tiles (80 x 48 pixels)
    (3, 6, 10, 16, 4, 3, 0.05),
    (1, 64, 64, 16, 3, 2, 0.1),  # the timed workload's image
])
def test_sobel_select_bitexact(H, B, Hh, W, patch, C, radius, thr):
    img = I.make_image(B, Hh, W, patch, C, seed=10 * Hh + W)
    rng = np.random.default_rng(Hh + W)
    mask = (rng.random((B, Hh * W)) < 0.05).astype(np.uint8)
    got = run_select(H, img, mask, Hh, W, patch, radius, thr)
    ref = O.sobel_select(img, mask, Hh, W, patch, radius, thr)
    assert np.array_equal(got, ref)
    assert 0 < ref.sum() < ref.size


def test_sobel_select_unaligned_image(H):
    """An image that starts 4 bytes past a 16-byte boundary takes the scalar
    load path of every tile; the keep map is unchanged in definition."""
    B, Hh, W, patch, C = 2, 8, 12, 16, 3
    img = I.make_image(B, Hh, W, patch, C, seed=5)
    rng = np.random.default_rng(9)
    mask = (rng.random((B, Hh * W)) < 0.05).astype(np.uint8)
    buf = torch.empty(img.size + 1, dtype=torch.float32, device="cuda")
    view = buf[1:].view(img.shape)
    view.copy_(torch.from_numpy(img))
    assert view.data_ptr() % 16 != 0
    sh = H.Shape(B=B, H=Hh, W=W, d=128)
    ws_bytes = H.hilo_sobel_workspace_bytes(sh)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    keep = torch.full((B, Hh * W), 7, dtype=torch.uint8, device="cuda")
    H.hilo_sobel_select(sh, view, C, patch, torch.from_numpy(mask).cuda(), 1, 0.1, keep, ws, ws_bytes)
    H.hilo_sync_status()
    ref = O.sobel_select(img, mask, Hh, W, patch, 1, 0.1)
    assert np.array_equal(keep.cpu().numpy(), ref)
    assert 0 < ref.sum() < ref.size


def test_sobel_select_constant_and_step_images(H):
    Hh, W, patch = 4, 6, 16
    const = np.full((1, Hh * patch, W * patch, 3), 0.25, dtype=np.float32)
    mask = np.zeros((1, Hh * W), dtype=np.uint8)
    mask[0, 9] = 1
    got = run_select(H, const, mask, Hh, W, patch, 1, 0.1)
    assert np.array_equal(got, O.dilate_mask(mask, Hh, W, 1))
    step = np.zeros((2, Hh * patch, W * patch, 1), dtype=np.float32)
    step[0, :, 40:] = 1.0
    step[1, 30:, :] = 0.5
    z = np.zeros((2, Hh * W), dtype=np.uint8)
    got = run_select(H, step, z, Hh, W, patch, 0, 0.1).reshape(2, Hh, W)
    assert np.array_equal(got, O.sobel_select(step, z, Hh, W, patch, 0, 0.1).reshape(2, Hh, W))
    assert got[0].sum() == Hh and got[0][:, 2].all()   # pixel columns 39 and 40: token column 2 only
    assert got[1].sum() == W and got[1][1].all()       # pixel rows 29 and 30: token row 1 only


def test_hot_path_with_sobel_selection(H):
    """Selector -> split (mask = keep map, k_keep = 0) -> pack -> block ->
    unpack at the 32 x 32 layer: index sets and packed rows bit for bit, block
    output within tolerance, against the oracle fed the oracle's keep map."""
    wl = I.tiny_layer()
    batch = I.make_batch(wl)
    img = I.make_image(wl.B, wl.H, wl.W, 16, 3, seed=3)
    w = I.make_weights(wl.d, wl.mlp, seed=I.weight_seed(wl))
    sh = H.Shape(B=wl.B, H=wl.H, W=wl.W, d=wl.d, T=wl.T, heads=wl.heads, mlp=int(wl.mlp), levels=1)
    keep_ref = O.sobel_select(img, batch.mask, wl.H, wl.W, 16, 1, 0.1)
    keep = torch.from_numpy(run_select(H, img, batch.mask, wl.H, wl.W, 16, 1, 0.1)).cuda()
    hp = H.HotPath(sh, [H.DeviceWeights.from_host(w)])
    x = H.bf16_from_bits(batch.x)
    text = H.bf16_from_bits(batch.text)
    zeros = torch.zeros(wl.B, dtype=torch.int32, device="cuda")
    hp.run(x, text, keep, zeros, zeros)
    H.hilo_sync_status()
    s_ref = O.score(batch.x)
    sp = O.split(s_ref, keep_ref, np.zeros(wl.B, np.int32), np.zeros(wl.B, np.int32), wl.H, wl.W, 1)
    cu = hp.split.cu_img.cpu().numpy()
    assert np.array_equal(cu, sp.cu_img)
    assert np.array_equal(hp.split.labels.cpu().numpy().reshape(wl.B, wl.N), sp.labels)
    assert np.array_equal(sp.labels == O.KEEP, keep_ref != 0)
    rows = int(cu[-1])
    packed = O.pack(batch.x, sp)
    assert np.array_equal(H.bits_from_bf16(hp.packed[:rows]), packed)
    ot, oi = O.block(batch.text.reshape(wl.B * wl.T, wl.d), packed, sp.cu_img, wl.T, w, wl.heads, wl.mlp)
    got = hp.out.cpu().numpy()
    assert_block_close(got[:wl.B * wl.T], ot, "text")
    assert_block_close(got[wl.B * wl.T:wl.B * wl.T + rows], oi, "image")
