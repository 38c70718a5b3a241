"""The window-granular split and the delta unpool on the GPU against the
oracle (Sec. 2.3's coherent, region-level selection read in token space).

Labels, offsets, row sources and the token -> row map must match bit for
bit, for one image (the single-kernel path) and for batches (two kernels),
with one and two pooling levels; packed rows and the delta-unpooled grid are
bit-exact as well (fp32 subtract then add on both sides). The whole hot path
in this mode is then checked at the 32 x 32 layer: index sets and packed
rows exactly, block output and unpooled grid within the block tolerance.
"""
import numpy as np
import pytest
import torch

from oracle import hilo_oracle as O
from paper_2606_13898_gb300 import inputs as I

from .gpu_helpers import assert_block_close, lib_ready, to_dev_f32, to_dev_i32, to_dev_u8

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def H():
    return lib_ready()


def run_split_regions(H, s, mask, kk, km, Hh, W, levels):
    B = s.shape[0]
    sh = H.Shape(B=B, H=Hh, W=W, d=128, levels=levels)
    sp = H.SplitBuffers.alloc(sh)
    H.hilo_split_regions(sh, to_dev_f32(s), to_dev_u8(mask), to_dev_i32(kk), to_dev_i32(km), sp)
    H.hilo_sync_status()
    return sp


def check_split(sp, ref, B, N):
    cu = sp.cu_img.cpu().numpy()
    assert np.array_equal(cu, ref.cu_img)
    rows = int(cu[-1])
    assert np.array_equal(sp.labels.cpu().numpy().reshape(B, N), ref.labels)
    assert np.array_equal(sp.counts.cpu().numpy().reshape(B, 3), ref.counts)
    assert np.array_equal(sp.row_src.cpu().numpy()[:rows], ref.row_src)
    assert np.array_equal(sp.tok_row.cpu().numpy().reshape(B, N), ref.tok_row)


@pytest.mark.parametrize("B", [1, 3])
@pytest.mark.parametrize("levels", [1, 2])
@pytest.mark.parametrize("seed", range(4))
def test_split_regions_bitexact_random_ties(H, seed, levels, B):
    rng = np.random.default_rng(40 + seed)
    Hh, W = [(8, 8), (16, 12), (64, 64), (128, 128)][seed]
    N = Hh * W
    s = (rng.integers(0, 7, size=(B, N)) * 0.25).astype(np.float32)
    mask = (rng.random((B, N)) < 0.05).astype(np.uint8)
    kk = rng.integers(0, N // 4 + 1, size=B).astype(np.int32)
    km = rng.integers(0, N // 2 + 1, size=B).astype(np.int32)
    sp = run_split_regions(H, s, mask, kk, km, Hh, W, levels)
    ref = O.split(s, mask, kk, km, Hh, W, levels, granular=True)
    check_split(sp, ref, B, N)
    # the mode changes the result on these inputs
    assert not np.array_equal(ref.labels, O.split(s, mask, kk, km, Hh, W, levels).labels)


@pytest.mark.parametrize("B", [1, 2])
@pytest.mark.parametrize("case", ["k0", "kN", "all_mask", "no_mask", "all_equal"])
def test_split_regions_edge_cases(H, case, B):
    rng = np.random.default_rng(8)
    Hh, W = 32, 32
    N = Hh * W
    s = rng.random((B, N)).astype(np.float32)
    mask = (rng.random((B, N)) < 0.03).astype(np.uint8)
    kk = np.array([N // 8, 3][:B], dtype=np.int32)
    km = np.array([N // 4, 0][:B], dtype=np.int32)
    if case == "k0":
        kk[:] = 0
    elif case == "kN":
        kk[:] = N
    elif case == "all_mask":
        mask[:] = 1
    elif case == "no_mask":
        mask[:] = 0
    elif case == "all_equal":
        s[:] = 1.5
    for levels in (1, 2):
        sp = run_split_regions(H, s, mask, kk, km, Hh, W, levels)
        check_split(sp, O.split(s, mask, kk, km, Hh, W, levels, granular=True), B, N)


@pytest.mark.parametrize("levels", [1, 2])
def test_pack_and_unpack_delta_bitexact(H, levels):
    rng = np.random.default_rng(60 + levels)
    B, Hh, W, d = 3, 16, 24, 256
    N = Hh * W
    x = I.f32_to_bf16_bits(rng.standard_normal((B, Hh, W, d)).astype(np.float32))
    s = O.score(x)
    mask = (rng.random((B, N)) < 0.05).astype(np.uint8)
    kk = np.array([0, N // 8, N], dtype=np.int32)
    km = np.array([N // 3, N // 5, 0], dtype=np.int32)
    ref = O.split(s, mask, kk, km, Hh, W, levels, granular=True)
    sh = H.Shape(B=B, H=Hh, W=W, d=d, levels=levels)
    sp = H.SplitBuffers.alloc(sh)
    H.hilo_split_regions(sh, to_dev_f32(s), to_dev_u8(mask), to_dev_i32(kk), to_dev_i32(km), sp)
    cap = B * N
    packed = torch.full((cap, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    xd = H.bf16_from_bits(x)
    H.hilo_pack(sh, xd, sp, packed, cap)
    H.hilo_sync_status()
    check_split(sp, ref, B, N)
    rows = int(ref.cu_img[-1])
    pref = O.pack(x, ref)
    assert np.array_equal(H.bits_from_bf16(packed[:rows]), pref)
    out = torch.from_numpy(rng.standard_normal((cap, d)).astype(np.float32)).cuda()
    y = torch.full((B, Hh, W, d), float("nan"), dtype=torch.float32, device="cuda")
    H.hilo_unpack_delta(sh, out, packed, xd, sp, y)
    H.hilo_sync_status()
    yref = O.unpack_delta(out.cpu().numpy()[:rows], pref, x, ref)
    assert np.array_equal(y.cpu().numpy(), yref)


def test_hot_path_regions_mode(H):
    """score -> window-granular split -> pack -> block -> delta unpool at the
    32 x 32 layer against the oracle's hot path in the same mode."""
    wl = I.tiny_layer()
    batch = I.make_batch(wl)
    w = I.make_weights(wl.d, wl.mlp, seed=I.weight_seed(wl))
    sh = H.Shape(B=wl.B, H=wl.H, W=wl.W, d=wl.d, T=wl.T, heads=wl.heads, mlp=int(wl.mlp), levels=1)
    hp = H.HotPath(sh, [H.DeviceWeights.from_host(w)])
    x = H.bf16_from_bits(batch.x)
    text = H.bf16_from_bits(batch.text)
    hp.run(x, text, to_dev_u8(batch.mask), to_dev_i32(batch.k_keep), to_dev_i32(batch.k_mid), regions=True)
    H.hilo_sync_status()
    sp, packed, (ot, oi), y = O.hot_path(batch.x, batch.text, batch.mask, batch.k_keep, batch.k_mid, 1, [w],
                                         wl.heads, wl.mlp, regions=True)
    cu = hp.split.cu_img.cpu().numpy()
    assert np.array_equal(cu, sp.cu_img)
    assert np.array_equal(hp.split.labels.cpu().numpy().reshape(wl.B, wl.N), sp.labels)
    rows = int(cu[-1])
    assert np.array_equal(H.bits_from_bf16(hp.packed[:rows]), packed)
    got = hp.out.cpu().numpy()
    assert_block_close(got[:wl.B * wl.T], ot, "text")
    assert_block_close(got[wl.B * wl.T:wl.B * wl.T + rows], oi, "image")
    assert_block_close(hp.y.cpu().numpy(), y, "delta-unpooled grid")
