"""Parity of the whole hot path at the five workload configurations.

Every configuration runs through the C ABI exactly as bench.py launches it
(HotPath: score -> split -> pack -> block(s) -> unpack, buffers sized to the
upper bound). Checked against the CPU oracle on the same seeded inputs:
  * scores, labels, row sources, counts, cu_img, token->row map and packed
    rows bit for bit;
  * block outputs within max-abs 2e-2 and rel-L2 1e-2 -- on every row for
    the 32x32 layer, on sampled rows (the oracle computes them one by one,
    keys/values over the whole joint sequence) at the d=3072 sizes;
  * unpack bit for bit (a gather of the GPU's own block output).
The 8-block x 28-step denoising loop is checked teacher-forced: at steps 0,
13 and 27 the oracle takes the GPU's bf16 latents, must reproduce the split
exactly, and blocks 0 and 7 are checked on sampled rows from the GPU's own
input to that block.
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


def run_path(H, wl, batch, weights_dev, keep_block_inputs=False):
    sh = H.Shape(B=wl.B, H=wl.H, W=wl.W, d=wl.d, T=wl.T, heads=wl.heads, mlp=int(wl.mlp), levels=wl.levels)
    hp = H.HotPath(sh, weights_dev)
    x = H.bf16_from_bits(batch.x)
    text = H.bf16_from_bits(batch.text)
    mask = torch.from_numpy(batch.mask).cuda()
    kk = torch.from_numpy(batch.k_keep).cuda()
    km = torch.from_numpy(batch.k_mid).cuda()
    hp.run(x, text, mask, kk, km)
    H.hilo_sync_status()
    return hp


def check_split_pack(H, hp, wl, batch):
    s_ref = O.score(batch.x)
    got_s = hp.score.cpu().numpy().reshape(s_ref.shape)
    assert np.array_equal(got_s.view(np.uint32), s_ref.view(np.uint32)), "score"
    sp = O.split(s_ref, batch.mask, batch.k_keep, batch.k_mid, wl.H, wl.W, wl.levels)
    cu = hp.split.cu_img.cpu().numpy()
    assert np.array_equal(cu, sp.cu_img), "cu_img"
    rows = int(cu[-1])
    assert np.array_equal(hp.split.labels.cpu().numpy().reshape(wl.B, wl.N), sp.labels), "labels"
    assert np.array_equal(hp.split.counts.cpu().numpy().reshape(wl.B, 3), sp.counts), "counts"
    assert np.array_equal(hp.split.row_src.cpu().numpy()[:rows], sp.row_src), "row_src"
    assert np.array_equal(hp.split.tok_row.cpu().numpy().reshape(wl.B, wl.N), sp.tok_row), "tok_row"
    packed = O.pack(batch.x, sp)
    assert np.array_equal(H.bits_from_bf16(hp.packed[:rows]), packed), "packed rows"
    return sp, packed


def sample_rows(rng, lo, hi, n):
    n = min(n, hi - lo)
    return np.sort(rng.choice(np.arange(lo, hi), size=n, replace=False)) if n > 0 else np.zeros(0, int)


def check_block_sampled(got_out, u_txt, u_img, cu, wl, w, rng, n_per_image=24, label=""):
    """Oracle rows of the block, image by image, against the GPU output rows."""
    T = wl.T
    for b in range(wl.B):
        tr = sample_rows(rng, b * T, (b + 1) * T, n_per_image // 3)
        ir = sample_rows(rng, int(cu[b]), int(cu[b + 1]), n_per_image)
        ot, oi = O.block_rows(u_txt, u_img, cu, T, w, wl.heads, wl.mlp, b, tr, ir)
        assert_block_close(got_out[tr], ot, f"{label} image {b} text rows")
        assert_block_close(got_out[wl.B * T + ir], oi, f"{label} image {b} image rows")


def test_tiny_layer_full_compare(H):
    wl = I.tiny_layer()
    batch = I.make_batch(wl)
    w = I.make_weights(wl.d, wl.mlp, seed=I.weight_seed(wl))
    hp = run_path(H, wl, batch, [H.DeviceWeights.from_host(w)])
    sp, packed = check_split_pack(H, hp, wl, batch)
    rows = int(sp.cu_img[-1])
    ot, oi = O.block(batch.text.reshape(wl.B * wl.T, wl.d), packed, sp.cu_img, wl.T, w, wl.heads, wl.mlp)
    got = hp.out.cpu().numpy()
    assert_block_close(got[:wl.B * wl.T], ot, "text")
    assert_block_close(got[wl.B * wl.T:wl.B * wl.T + rows], oi, "image")
    y = hp.y.cpu().numpy().reshape(wl.B, wl.N, wl.d)
    assert np.array_equal(y, hp.out_img[:rows].cpu().numpy()[sp.tok_row])


@pytest.mark.parametrize("ratio", ["1/10", "1/4", "1/2", "1"])
def test_block64_keep_ratio_sweep(H, ratio):
    wl = I.block_64(keep_ratio=ratio)
    batch = I.make_batch(wl)
    w = I.make_weights(wl.d, wl.mlp, seed=I.weight_seed(wl))
    hp = run_path(H, wl, batch, [H.DeviceWeights.from_host(w)])
    sp, packed = check_split_pack(H, hp, wl, batch)
    if ratio == "1":
        assert np.all(sp.labels == O.KEEP) and np.array_equal(packed, batch.x.reshape(wl.N, wl.d))
    got = hp.out.cpu().numpy()
    rng = np.random.default_rng(1)
    check_block_sampled(got, batch.text.reshape(-1, wl.d), packed, sp.cu_img, wl, O.weights_f64(w), rng,
                        label=f"r={ratio}")
    rows = int(sp.cu_img[-1])
    y = hp.y.cpu().numpy().reshape(wl.B, wl.N, wl.d)
    assert np.array_equal(y, got[wl.B * wl.T:wl.B * wl.T + rows][sp.tok_row])


def test_block64_batch4_varlen(H):
    wl = I.block_64_batch4()
    batch = I.make_batch(wl)
    assert len(set(batch.k_keep.tolist())) > 1
    w = I.make_weights(wl.d, wl.mlp, seed=I.weight_seed(wl))
    hp = run_path(H, wl, batch, [H.DeviceWeights.from_host(w)])
    sp, packed = check_split_pack(H, hp, wl, batch)
    lens = np.diff(sp.cu_img)
    assert len(set(lens.tolist())) == wl.B, lens
    got = hp.out.cpu().numpy()
    check_block_sampled(got, batch.text.reshape(-1, wl.d), packed, sp.cu_img, wl, O.weights_f64(w),
                        np.random.default_rng(2), n_per_image=16, label="b4")


def test_block128_two_level(H):
    wl = I.block_128_two_level()
    batch = I.make_batch(wl)
    w = I.make_weights(wl.d, wl.mlp, seed=I.weight_seed(wl))
    hp = run_path(H, wl, batch, [H.DeviceWeights.from_host(w)])
    sp, packed = check_split_pack(H, hp, wl, batch)
    assert sp.counts[0, 2] > 0 and sp.counts[0, 1] > 0
    got = hp.out.cpu().numpy()
    check_block_sampled(got, batch.text.reshape(-1, wl.d), packed, sp.cu_img, wl, O.weights_f64(w),
                        np.random.default_rng(3), label="two-level")


def test_denoise_loop_teacher_forced(H):
    wl = I.denoise_loop()
    batch = I.make_batch(wl)
    n_layers, n_steps, alpha = 8, 28, 0.035
    ws = [I.make_weights(wl.d, wl.mlp, seed=I.weight_seed(wl, i)) for i in range(n_layers)]
    dws = [H.DeviceWeights.from_host(w) for w in ws]
    sh = H.Shape(B=wl.B, H=wl.H, W=wl.W, d=wl.d, T=wl.T, heads=wl.heads, mlp=1, levels=wl.levels)
    hp = H.HotPath(sh, dws[:1])
    x = H.bf16_from_bits(batch.x)
    text = H.bf16_from_bits(batch.text)
    mask = torch.from_numpy(batch.mask).cuda()
    kk = torch.from_numpy(batch.k_keep).cuda()
    km = torch.from_numpy(batch.k_mid).cuda()
    rng = np.random.default_rng(4)
    BT = wl.B * wl.T
    for step in range(n_steps):
        check = step in (0, 13, 27)
        x_bits = H.bits_from_bf16(x) if check else None
        H.hilo_score(sh, x, hp.score)
        H.hilo_split(sh, hp.score, mask, kk, km, hp.split)
        H.hilo_pack(sh, x, hp.split, hp.packed, hp.cap)
        if check:
            H.hilo_sync_status()
            sp, packed = check_split_pack(H, hp, wl, type(batch)(wl, x_bits, batch.text, batch.mask,
                                                                  batch.k_keep, batch.k_mid))
        for li in range(n_layers):
            if li == 0:
                in_t, in_i, dt = text, hp.packed, H.HILO_BF16
            else:
                in_t, in_i, dt = hp.out, hp.out_img, H.HILO_F32
            snap = None
            if check and li in (0, n_layers - 1):
                H.hilo_sync_status()
                if li == 0:
                    snap = (batch.text.reshape(-1, wl.d), packed)
                else:
                    o = hp.out.cpu().numpy()
                    snap = (o[:BT], o[BT:BT + int(sp.cu_img[-1])])
            H.hilo_block_forward(sh, dws[li], hp.split.cu_img, hp.cap, in_t, in_i, dt, hp.out, hp.ws, hp.ws_bytes)
            if snap is not None:
                H.hilo_sync_status()
                check_block_sampled(hp.out.cpu().numpy(), snap[0], snap[1], sp.cu_img, wl,
                                    O.weights_f64(ws[li]), rng, n_per_image=12, label=f"step {step} layer {li}")
        H.hilo_unpack_update(sh, hp.out_img, hp.split, x, alpha)
        if check:
            H.hilo_sync_status()
            rows = int(sp.cu_img[-1])
            yref = hp.out.cpu().numpy()[BT:BT + rows][sp.tok_row].reshape(x.shape)
            assert np.array_equal(H.bits_from_bf16(x), O.update(x_bits, yref, alpha)), f"update at step {step}"
    H.hilo_sync_status()
    assert torch.isfinite(x.float()).all()
