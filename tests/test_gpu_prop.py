"""Proportional attention for pooled tokens on the GPU against the oracle.

A packed row standing for n grid tokens adds ln n to its logits as a key
(the oracle's definition); the kernel multiplies each probability by n before
the row sum and the bf16 rounding of P. Row sizes are integers and must match
bit for bit; block outputs within max-abs 2e-2 and rel-L2 1e-2 over shapes
with ragged text and image tiles, both head widths, several images and no
text, and the whole hot path in this mode at the 32 x 32 layer.
"""
import numpy as np
import pytest
import torch

from oracle import hilo_oracle as O
from paper_2606_13898_gb300 import inputs as I

from .gpu_helpers import assert_block_close, close_report, lib_ready, to_dev_f32, to_dev_i32, to_dev_u8
from .test_gpu_kernels import bits, scaled_weights

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def H():
    return lib_ready()


@pytest.mark.parametrize("granular", [False, True])
@pytest.mark.parametrize("levels", [1, 2])
@pytest.mark.parametrize("B", [1, 3])
def test_row_sizes_bitexact(H, B, levels, granular):
    rng = np.random.default_rng(70 + B + 2 * levels + int(granular))
    Hh, W = 16, 24
    N = Hh * W
    s = (rng.integers(0, 9, size=(B, N)) * 0.5).astype(np.float32)
    mask = (rng.random((B, N)) < 0.05).astype(np.uint8)
    kk = rng.integers(0, N // 3, size=B).astype(np.int32)
    km = rng.integers(0, N // 2, size=B).astype(np.int32)
    sh = H.Shape(B=B, H=Hh, W=W, d=128, levels=levels)
    sp = H.SplitBuffers.alloc(sh)
    (H.hilo_split_regions if granular else H.hilo_split)(sh, to_dev_f32(s), to_dev_u8(mask), to_dev_i32(kk),
                                                         to_dev_i32(km), sp)
    cap = B * N
    n = torch.full((cap,), float("nan"), dtype=torch.float32, device="cuda")
    H.hilo_row_sizes(sh, sp, n, cap)
    H.hilo_sync_status()
    ref = O.split(s, mask, kk, km, Hh, W, levels, granular=granular)
    rows = int(ref.cu_img[-1])
    assert np.array_equal(n.cpu().numpy()[:rows], O.row_sizes(ref))


@pytest.mark.parametrize("d,heads,T,lens,mlp", [
    (128, 1, 64, [200], 0),          # head_dim 128, ragged text and image tiles
    (128, 2, 64, [256, 77], 1),      # head_dim 64, two images of different length
    (256, 2, 0, [130, 300, 5], 1),   # no text, three images
    (512, 8, 200, [384], 1),         # several 256-wide GEMM column tiles
])
def test_block_forward_prop_matches_oracle(H, d, heads, T, lens, mlp):
    rng = np.random.default_rng(d + T + 7 * len(lens))
    B = len(lens)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    rows = int(cu[-1])
    cap = rows + 37
    ut = bits(rng.standard_normal((B * T, d)))
    ui = bits(rng.standard_normal((rows, d)))
    w = scaled_weights(rng, d, mlp, std=1.0 / np.sqrt(d))
    # row weights as the splits produce them (1, 2..4, 16), and larger ones
    n = rng.choice(np.array([1, 1, 1, 2, 3, 4, 16, 40], np.float32), size=rows)
    grid = int(np.ceil(np.sqrt(cap)))
    sh = H.Shape(B=B, H=2 * grid, W=2 * grid, d=d, T=T, heads=heads, mlp=mlp)
    dw = H.DeviceWeights.from_host(w)
    in_txt = H.bf16_from_bits(ut) if T else None
    in_img = torch.full((cap, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    in_img[:rows] = H.bf16_from_bits(ui)
    n_dev = torch.full((cap,), float("nan"), dtype=torch.float32, device="cuda")
    n_dev[:rows] = torch.from_numpy(n).cuda()
    out = torch.empty(B * T + cap, d, dtype=torch.float32, device="cuda")
    wsb = H.hilo_block_workspace_bytes(sh, cap)
    ws = torch.full((wsb,), 0xFF, dtype=torch.uint8, device="cuda")   # NaN-filled scratch
    H.hilo_block_forward_prop(sh, dw, to_dev_i32(cu), cap, in_txt, in_img, H.HILO_BF16, n_dev, out, ws, wsb)
    H.hilo_sync_status()
    ot, oi = O.block(ut, ui, cu, T, w, heads, bool(mlp), n_img=n)
    got = out.cpu().numpy()
    assert_block_close(got[:B * T], ot, "text rows")
    assert_block_close(got[B * T:B * T + rows], oi, "image rows")
    # the weighting is really applied: the unweighted block is far off
    pt, pi = O.block(ut, ui, cu, T, w, heads, bool(mlp))
    assert close_report(got[B * T:B * T + rows], pi)[0] > 10 * close_report(got[B * T:B * T + rows], oi)[0]


def test_hot_path_prop_mode(H):
    """score -> split -> pack -> row sizes -> block with proportional
    attention -> unpack at the 32 x 32 layer, both split modes."""
    wl = I.tiny_layer()
    batch = I.make_batch(wl)
    w = I.make_weights(wl.d, wl.mlp, seed=I.weight_seed(wl))
    sh = H.Shape(B=wl.B, H=wl.H, W=wl.W, d=wl.d, T=wl.T, heads=wl.heads, mlp=int(wl.mlp), levels=1)
    hp = H.HotPath(sh, [H.DeviceWeights.from_host(w)])
    x = H.bf16_from_bits(batch.x)
    text = H.bf16_from_bits(batch.text)
    for regions in (False, True):
        hp.run(x, text, to_dev_u8(batch.mask), to_dev_i32(batch.k_keep), to_dev_i32(batch.k_mid), regions=regions,
               prop=True)
        H.hilo_sync_status()
        sp, packed, (ot, oi), y = O.hot_path(batch.x, batch.text, batch.mask, batch.k_keep, batch.k_mid, 1, [w],
                                             wl.heads, wl.mlp, regions=regions, prop=True)
        rows = int(sp.cu_img[-1])
        assert np.array_equal(hp.n_img.cpu().numpy()[:rows], O.row_sizes(sp))
        got = hp.out.cpu().numpy()
        assert_block_close(got[:wl.B * wl.T], ot, "text")
        assert_block_close(got[wl.B * wl.T:wl.B * wl.T + rows], oi, "image")
        assert_block_close(hp.y.cpu().numpy().reshape(wl.B, wl.N, wl.d), np.reshape(y, (wl.B, wl.N, wl.d)), "grid")
