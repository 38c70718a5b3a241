"""The hot path's other modes at the timed workload's size (64 x 64 grid,
d = 3072, 512 text tokens, keep ratio 1/4), run through the C ABI exactly
as bench.py runs them, against the oracle on the same seeded inputs:

  * window-granular split + delta unpool, and the separate low-frequency set
    (lf = 4): labels, offsets, row sources, token map and packed rows bit for
    bit; the delta-unpooled grid bit for bit from the GPU's own block output;
  * proportional attention: row sizes bit for bit;
  * block outputs on sampled rows (keys and values over the whole joint
    sequence in the oracle) within max-abs 2e-2 and rel-L2 1e-2;
  * the FP8 block on sampled rows: within 3% of the rows' update (out - u)
    of the oracle's FP8 emulation, and within the e4m3 error model (under
    10%) of the exact block.
"""
import numpy as np
import pytest
import torch

from oracle import hilo_oracle as O
from paper_2606_13898_gb300 import inputs as I

from .gpu_helpers import assert_block_close, lib_ready
from .test_gpu_configs import sample_rows

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def H():
    return lib_ready()


@pytest.fixture(scope="module")
def setup():
    wl = I.block_64("1/4")
    batch = I.make_batch(wl)
    w = I.make_weights(wl.d, wl.mlp, seed=I.weight_seed(wl))
    return wl, batch, w


def run(H, wl, batch, weights, lf=0, **kw):
    sh = H.Shape(B=wl.B, H=wl.H, W=wl.W, d=wl.d, T=wl.T, heads=wl.heads, mlp=int(wl.mlp), levels=wl.levels, lf=lf)
    hp = H.HotPath(sh, weights)
    return hp, sh


def inputs(H, batch):
    return (H.bf16_from_bits(batch.x), H.bf16_from_bits(batch.text), torch.from_numpy(batch.mask).cuda(),
            torch.from_numpy(batch.k_keep).cuda(), torch.from_numpy(batch.k_mid).cuda())


def check_split(hp, sp, wl):
    cu = hp.split.cu_img.cpu().numpy()
    assert np.array_equal(cu, sp.cu_img)
    rows = int(cu[-1])
    assert np.array_equal(hp.split.labels.cpu().numpy().reshape(wl.B, wl.N), sp.labels)
    assert np.array_equal(hp.split.counts.cpu().numpy().reshape(wl.B, 3), sp.counts)
    assert np.array_equal(hp.split.row_src.cpu().numpy()[:rows], sp.row_src)
    assert np.array_equal(hp.split.tok_row.cpu().numpy().reshape(wl.B, wl.N), sp.tok_row)
    return rows


def sampled(wl, cu, seed, n=24):
    rng = np.random.default_rng(seed)
    return sample_rows(rng, 0, wl.T, n // 3), sample_rows(rng, int(cu[0]), int(cu[1]), n)


@pytest.mark.parametrize("mode", ["regions", "lf"])
def test_regions_and_low_frequency_modes_full_size(H, setup, mode):
    wl, batch, w = setup
    lf = 4 if mode == "lf" else 0
    hp, sh = run(H, wl, batch, [H.DeviceWeights.from_host(w)], lf=lf)
    hp.run(*inputs(H, batch), regions=mode == "regions")
    H.hilo_sync_status()
    s = O.score(batch.x)
    sp = O.split(s, batch.mask, batch.k_keep, batch.k_mid, wl.H, wl.W, wl.levels, granular=mode == "regions", lf=lf)
    rows = check_split(hp, sp, wl)
    packed = O.pack(batch.x, sp, lf)
    assert np.array_equal(H.bits_from_bf16(hp.packed[:rows]), packed)
    got = hp.out.cpu().numpy()
    tr, ir = sampled(wl, sp.cu_img, 31 + lf)
    ot, oi = O.block_rows(batch.text.reshape(-1, wl.d), packed, sp.cu_img, wl.T, O.weights_f64(w), wl.heads,
                          wl.mlp, 0, tr, ir)
    assert_block_close(got[tr], ot, f"{mode} text rows")
    assert_block_close(got[wl.T + ir], oi, f"{mode} image rows")
    y_ref = O.unpack_delta(got[wl.T:wl.T + rows], packed, batch.x, sp)
    assert np.array_equal(hp.y.cpu().numpy(), y_ref)


def test_proportional_attention_full_size(H, setup):
    wl, batch, w = setup
    hp, sh = run(H, wl, batch, [H.DeviceWeights.from_host(w)])
    hp.run(*inputs(H, batch), prop=True)
    H.hilo_sync_status()
    sp = O.split(O.score(batch.x), batch.mask, batch.k_keep, batch.k_mid, wl.H, wl.W, wl.levels)
    rows = check_split(hp, sp, wl)
    n = O.row_sizes(sp)
    assert np.array_equal(hp.n_img.cpu().numpy()[:rows], n)
    packed = O.pack(batch.x, sp)
    got = hp.out.cpu().numpy()
    tr, ir = sampled(wl, sp.cu_img, 41)
    ot, oi = O.block_rows(batch.text.reshape(-1, wl.d), packed, sp.cu_img, wl.T, O.weights_f64(w), wl.heads,
                          wl.mlp, 0, tr, ir, n_img=n)
    assert_block_close(got[tr], ot, "prop text rows")
    assert_block_close(got[wl.T + ir], oi, "prop image rows")


def test_fp8_block_full_size(H, setup):
    wl, batch, w = setup
    hp, sh = run(H, wl, batch, [H.DeviceWeights.from_host(w)])
    hp.enable_fp8([H.DeviceWeightsFP8.from_host(w)])
    hp.run(*inputs(H, batch), fp8=True)
    H.hilo_sync_status()
    sp = O.split(O.score(batch.x), batch.mask, batch.k_keep, batch.k_mid, wl.H, wl.W, wl.levels)
    check_split(hp, sp, wl)
    packed = O.pack(batch.x, sp)
    got = hp.out.cpu().numpy()
    tr, ir = sampled(wl, sp.cu_img, 51, n=30)
    txt = batch.text.reshape(-1, wl.d)
    qt, qi = O.block_rows_fp8(txt, packed, sp.cu_img, wl.T, O.quantize_weights(w), wl.heads, wl.mlp, 0, tr, ir)
    et, ei = O.block_rows(txt, packed, sp.cu_img, wl.T, O.weights_f64(w), wl.heads, wl.mlp, 0, tr, ir)
    u = np.concatenate([O.bf16_to_f32(txt[tr]), O.bf16_to_f32(packed[ir])]).astype(np.float64)
    g = np.concatenate([got[tr], got[wl.T + ir]])
    emu = np.concatenate([qt, qi])
    ex = np.concatenate([et, ei])
    assert np.all(np.isfinite(g))
    delta = np.linalg.norm(ex - u)
    e_emu = np.linalg.norm(g - emu) / delta
    e_ex = np.linalg.norm(g - ex) / delta
    assert e_emu < 0.03, e_emu
    assert 0.005 < e_ex < 0.1, e_ex


def test_fp8_block_proportional_attention_full_size(H, setup):
    """The FP8 block with proportional attention (row sizes from the GPU's
    own split, bit-exact against the oracle's) at the timed workload's size:
    sampled rows against the oracle's FP8 emulation with the same weights,
    and against the exact proportional block within the e4m3 model."""
    wl, batch, w = setup
    hp, sh = run(H, wl, batch, [H.DeviceWeights.from_host(w)])
    hp.enable_fp8([H.DeviceWeightsFP8.from_host(w)])
    hp.run(*inputs(H, batch), fp8=True, prop=True)
    H.hilo_sync_status()
    sp = O.split(O.score(batch.x), batch.mask, batch.k_keep, batch.k_mid, wl.H, wl.W, wl.levels)
    check_split(hp, sp, wl)
    n = O.row_sizes(sp)
    rows = int(sp.cu_img[-1])
    assert np.array_equal(hp.n_img[:rows].cpu().numpy(), n.astype(np.float32))
    packed = O.pack(batch.x, sp)
    got = hp.out.cpu().numpy()
    tr, ir = sampled(wl, sp.cu_img, 53, n=30)
    txt = batch.text.reshape(-1, wl.d)
    qt, qi = O.block_rows_fp8(txt, packed, sp.cu_img, wl.T, O.quantize_weights(w), wl.heads, wl.mlp, 0, tr, ir,
                              n_img=n)
    et, ei = O.block_rows(txt, packed, sp.cu_img, wl.T, O.weights_f64(w), wl.heads, wl.mlp, 0, tr, ir, n_img=n)
    u = np.concatenate([O.bf16_to_f32(txt[tr]), O.bf16_to_f32(packed[ir])]).astype(np.float64)
    g = np.concatenate([got[tr], got[wl.T + ir]])
    emu = np.concatenate([qt, qi])
    ex = np.concatenate([et, ei])
    assert np.all(np.isfinite(g))
    delta = np.linalg.norm(ex - u)
    e_emu = np.linalg.norm(g - emu) / delta
    e_ex = np.linalg.norm(g - ex) / delta
    assert e_emu < 0.03, e_emu
    assert 0.005 < e_ex < 0.1, e_ex
