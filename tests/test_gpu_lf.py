"""The separate low-frequency token set (shape.lf > 0) on the GPU against the
oracle: the kept tokens followed by every lf x lf window mean of the grid
(Sec. 2.3's downsampled-image tokens in token space).

Labels, offsets, row sources, the token -> row map, packed rows, row sizes
and the delta-unpooled grid match bit for bit, for one image (one kernel)
and batches (two kernels), lf = 2, 4, 8, including every token kept (the
largest row count, N + N/lf^2 per image) and nothing kept. The hot path in
this mode is checked at the 32 x 32 layer within the block tolerance, and a
block called with more image rows than its capacity computes the clamped
sequence instead of reading or writing past its buffers.
"""
import numpy as np
import pytest
import torch

from oracle import hilo_oracle as O
from paper_2606_13898_gb300 import inputs as I

from .gpu_helpers import assert_block_close, lib_ready, to_dev_f32, to_dev_i32, to_dev_u8
from .test_gpu_kernels import bits, scaled_weights

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def H():
    return lib_ready()


def check_split(sp, ref, B, N):
    cu = sp.cu_img.cpu().numpy()
    assert np.array_equal(cu, ref.cu_img)
    rows = int(cu[-1])
    assert np.array_equal(sp.labels.cpu().numpy().reshape(B, N), ref.labels)
    assert np.array_equal(sp.counts.cpu().numpy().reshape(B, 3), ref.counts)
    assert np.array_equal(sp.row_src.cpu().numpy()[:rows], ref.row_src)
    assert np.array_equal(sp.tok_row.cpu().numpy().reshape(B, N), ref.tok_row)


@pytest.mark.parametrize("B", [1, 3])
@pytest.mark.parametrize("lf", [2, 4, 8])
@pytest.mark.parametrize("case", ["random", "keep_all", "keep_none"])
def test_lf_split_pack_sizes_unpack_bitexact(H, B, lf, case):
    rng = np.random.default_rng(80 + 3 * lf + B)
    Hh, W, d = 32, 48, 128
    N = Hh * W
    x = I.f32_to_bf16_bits(rng.standard_normal((B, Hh, W, d)).astype(np.float32))
    s = O.score(x)
    mask = (rng.random((B, N)) < 0.1).astype(np.uint8)
    kk = rng.integers(0, N // 3, size=B).astype(np.int32)
    if case == "keep_all":
        kk[:] = N
    elif case == "keep_none":
        kk[:] = 0
        mask[:] = 0
    km = np.zeros(B, np.int32)
    sh = H.Shape(B=B, H=Hh, W=W, d=d, lf=lf)
    cap = H.hilo_row_capacity(sh)
    assert cap == B * (N + N // (lf * lf))
    sp = H.SplitBuffers.alloc(sh)
    H.hilo_split(sh, to_dev_f32(s), to_dev_u8(mask), to_dev_i32(kk), to_dev_i32(km), sp)
    packed = torch.full((cap, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    xd = H.bf16_from_bits(x)
    H.hilo_pack(sh, xd, sp, packed, cap)
    n = torch.full((cap,), float("nan"), dtype=torch.float32, device="cuda")
    H.hilo_row_sizes(sh, sp, n, cap)
    H.hilo_sync_status()
    ref = O.split(s, mask, kk, km, Hh, W, 1, lf=lf)
    check_split(sp, ref, B, N)
    rows = int(ref.cu_img[-1])
    if case == "keep_all":
        assert rows == cap
    pref = O.pack(x, ref, lf)
    assert np.array_equal(H.bits_from_bf16(packed[:rows]), pref)
    assert np.array_equal(n.cpu().numpy()[:rows], O.row_sizes(ref))
    out = torch.from_numpy(rng.standard_normal((cap, d)).astype(np.float32)).cuda()
    y = torch.full((B, Hh, W, d), float("nan"), dtype=torch.float32, device="cuda")
    H.hilo_unpack_delta(sh, out, packed, xd, sp, y)
    H.hilo_sync_status()
    assert np.array_equal(y.cpu().numpy(), O.unpack_delta(out.cpu().numpy()[:rows], pref, x, ref))


@pytest.mark.parametrize("prop", [False, True])
def test_hot_path_lf_mode(H, prop):
    wl = I.tiny_layer()
    batch = I.make_batch(wl)
    w = I.make_weights(wl.d, wl.mlp, seed=I.weight_seed(wl))
    sh = H.Shape(B=wl.B, H=wl.H, W=wl.W, d=wl.d, T=wl.T, heads=wl.heads, mlp=int(wl.mlp), levels=1, lf=4)
    hp = H.HotPath(sh, [H.DeviceWeights.from_host(w)])
    x = H.bf16_from_bits(batch.x)
    text = H.bf16_from_bits(batch.text)
    hp.run(x, text, to_dev_u8(batch.mask), to_dev_i32(batch.k_keep), to_dev_i32(batch.k_mid), prop=prop)
    H.hilo_sync_status()
    sp, packed, (ot, oi), y = O.hot_path(batch.x, batch.text, batch.mask, batch.k_keep, batch.k_mid, 1, [w],
                                         wl.heads, wl.mlp, prop=prop, lf=4)
    cu = hp.split.cu_img.cpu().numpy()
    assert np.array_equal(cu, sp.cu_img)
    rows = int(cu[-1])
    assert np.array_equal(H.bits_from_bf16(hp.packed[:rows]), packed)
    got = hp.out.cpu().numpy()
    assert_block_close(got[:wl.B * wl.T], ot, "text")
    assert_block_close(got[wl.B * wl.T:wl.B * wl.T + rows], oi, "image")
    assert_block_close(hp.y.cpu().numpy(), y, "grid")


def test_block_rows_clamped_to_capacity(H):
    """cu_img says 300 image rows, the capacity is 200: every kernel of the
    block stops at the capacity, and the result is the block over the first
    200 rows."""
    rng = np.random.default_rng(91)
    d, heads, T, cap = 256, 2, 64, 200
    ut = bits(rng.standard_normal((T, d)))
    ui = bits(rng.standard_normal((cap, d)))
    w = scaled_weights(rng, d, 1, std=1.0 / np.sqrt(d))
    sh = H.Shape(B=1, H=16, W=16, d=d, T=T, heads=heads, mlp=1)
    dw = H.DeviceWeights.from_host(w)
    in_img = H.bf16_from_bits(ui)
    out = torch.full((T + cap, d), float("nan"), dtype=torch.float32, device="cuda")
    wsb = H.hilo_block_workspace_bytes(sh, cap)
    ws = torch.full((wsb,), 0xFF, dtype=torch.uint8, device="cuda")
    H.hilo_block_forward(sh, dw, to_dev_i32([0, 300]), cap, H.bf16_from_bits(ut), in_img, H.HILO_BF16, out, ws,
                         wsb)
    H.hilo_sync_status()
    ot, oi = O.block(ut, ui, [0, cap], T, w, heads, True)
    got = out.cpu().numpy()
    assert_block_close(got[:T], ot, "text rows")
    assert_block_close(got[T:], oi, "image rows")
