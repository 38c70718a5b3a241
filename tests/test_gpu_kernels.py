"""GPU-vs-oracle parity of each C entry point on small shapes.

Sizes span several tiles (128-row GEMM / attention tiles, 256-column GEMM
tiles) and ragged tails, with the oracle finishing in seconds. Integer and
bf16-coded outputs (scores, labels, offsets, packed rows, unpacked rows) must
match bit for bit; block outputs within max-abs 2e-2 and rel-L2 1e-2.
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


def bits(a):
    return I.f32_to_bf16_bits(np.asarray(a, dtype=np.float32))


# ------------------------------------------------------------------ score --

@pytest.mark.parametrize("B,Hh,W,d", [(1, 32, 32, 512), (2, 6, 10, 128), (1, 2, 2, 3072), (3, 8, 4, 384)])
def test_score_bitexact(H, B, Hh, W, d):
    rng = np.random.default_rng(B * 100 + Hh + d)
    x = bits(rng.standard_normal((B, Hh, W, d)) * rng.uniform(0.1, 10, size=(B, Hh, W, 1)))
    sh = H.Shape(B=B, H=Hh, W=W, d=d)
    s = torch.empty(B * Hh * W, dtype=torch.float32, device="cuda")
    H.hilo_score(sh, H.bf16_from_bits(x), s)
    torch.cuda.synchronize()
    ref = O.score(x)
    got = s.cpu().numpy().reshape(ref.shape)
    assert np.array_equal(got.view(np.uint32), ref.view(np.uint32))


def test_score_closed_forms_on_gpu(H):
    # checkerboard +-a -> d*a^2 everywhere; constant -> 0
    d = 256
    p = np.arange(8)[:, None]
    q = np.arange(8)[None, :]
    cb = np.where((p + q) % 2 == 0, 0.75, -0.75)[None, :, :, None] * np.ones(d)
    x = np.concatenate([cb, np.full((1, 8, 8, d), 3.0)], axis=0)
    sh = H.Shape(B=2, H=8, W=8, d=d)
    s = torch.empty(2 * 64, dtype=torch.float32, device="cuda")
    H.hilo_score(sh, H.bf16_from_bits(bits(x)), s)
    got = s.cpu().numpy().reshape(2, 64)
    assert np.all(got[0] == np.float32(d * 0.5625)) and np.all(got[1] == 0.0)


# ------------------------------------------------------------------ split --

def run_split(H, s, mask, kk, km, Hh, W, levels):
    B = s.shape[0]
    sh = H.Shape(B=B, H=Hh, W=W, d=128, levels=levels)
    sp = H.SplitBuffers.alloc(sh)
    H.hilo_split(sh, to_dev_f32(s), to_dev_u8(mask), to_dev_i32(kk), to_dev_i32(km), sp)
    torch.cuda.synchronize()
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
def test_split_bitexact_random_ties(H, seed, levels, B):
    """B = 1 runs the single-kernel path (selection and compaction in one
    CTA), B = 3 the two-kernel path with offsets across images."""
    rng = np.random.default_rng(seed)
    Hh, W = [(8, 8), (16, 12), (64, 64), (128, 128)][seed]
    N = Hh * W
    # coarse scores: many exact ties decided by the token index
    s = (rng.integers(0, 7, size=(B, N)) * 0.25).astype(np.float32)
    mask = (rng.random((B, N)) < 0.2).astype(np.uint8)
    kk = rng.integers(0, N + 1, size=B).astype(np.int32)
    km = rng.integers(0, N + 1, size=B).astype(np.int32)
    sp = run_split(H, s, mask, kk, km, Hh, W, levels)
    check_split(sp, O.split(s, mask, kk, km, Hh, W, levels), B, N)


@pytest.mark.parametrize("B", [1, 2])
@pytest.mark.parametrize("case", ["k0", "kN", "all_mask", "no_mask", "all_equal", "wide_range"])
def test_split_edge_cases(H, case, B):
    rng = np.random.default_rng(7)
    Hh, W = 32, 32
    N = Hh * W
    s = rng.random((B, N)).astype(np.float32)
    mask = (rng.random((B, N)) < 0.15).astype(np.uint8)
    kk = np.array([N // 4, 3][:B], dtype=np.int32)
    km = np.array([N // 3, 0][:B], dtype=np.int32)
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
    elif case == "wide_range":
        s = (rng.random((B, N)) * 1e30).astype(np.float32)
        s[:, ::7] = 0.0
        s[:, 3::11] = 1e-40   # subnormal scores order correctly by their bits
    for levels in (1, 2):
        sp = run_split(H, s, mask, kk, km, Hh, W, levels)
        check_split(sp, O.split(s, mask, kk, km, Hh, W, levels), B, N)


@pytest.mark.parametrize("levels", [1, 2])
def test_split_largest_image(H, levels):
    """The largest image the ABI accepts (32768 tokens): the selection CTA's
    shared memory is 7 bytes per token, just inside the per-CTA limit."""
    rng = np.random.default_rng(11 + levels)
    Hh, W, B = 128, 256, 1
    N = Hh * W
    s = (rng.integers(0, 50, size=(B, N)) * 0.125).astype(np.float32)
    mask = (rng.random((B, N)) < 0.05).astype(np.uint8)
    kk = np.array([N // 4], dtype=np.int32)
    km = np.array([N // 4], dtype=np.int32)
    sp = run_split(H, s, mask, kk, km, Hh, W, levels)
    check_split(sp, O.split(s, mask, kk, km, Hh, W, levels), B, N)


# ------------------------------------------------------------ pack/unpack --

@pytest.mark.parametrize("levels", [1, 2])
def test_pack_unpack_bitexact(H, levels):
    rng = np.random.default_rng(20 + levels)
    B, Hh, W, d = 3, 16, 24, 256
    N = Hh * W
    x = bits(rng.standard_normal((B, Hh, W, d)))
    s = O.score(x)
    mask = (rng.random((B, N)) < 0.1).astype(np.uint8)
    kk = np.array([0, N // 5, N], dtype=np.int32)
    km = np.array([N // 2, N // 3, 0], dtype=np.int32)
    ref = O.split(s, mask, kk, km, Hh, W, levels)
    sh = H.Shape(B=B, H=Hh, W=W, d=d, levels=levels)
    sp = H.SplitBuffers.alloc(sh)
    H.hilo_split(sh, to_dev_f32(s), to_dev_u8(mask), to_dev_i32(kk), to_dev_i32(km), sp)
    cap = B * N
    packed = torch.full((cap, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    xd = H.bf16_from_bits(x)
    H.hilo_pack(sh, xd, sp, packed, cap)
    torch.cuda.synchronize()
    rows = int(ref.cu_img[-1])
    assert np.array_equal(H.bits_from_bf16(packed[:rows]), O.pack(x, ref))
    # unpack of an arbitrary fp32 block output
    out = torch.from_numpy(rng.standard_normal((cap, d)).astype(np.float32)).cuda()
    y = torch.empty(B, Hh, W, d, dtype=torch.float32, device="cuda")
    H.hilo_unpack(sh, out, sp, y)
    torch.cuda.synchronize()
    assert np.array_equal(y.cpu().numpy().reshape(B, N, d), O.unpack(out.cpu().numpy(), ref))
    # fused update x <- bf16(x - alpha * y)
    H.hilo_unpack_update(sh, out, sp, xd, 0.035)
    torch.cuda.synchronize()
    yref = O.unpack(out.cpu().numpy(), ref).reshape(B, Hh, W, d)
    assert np.array_equal(H.bits_from_bf16(xd), O.update(x, yref, 0.035))


# ------------------------------------------------------------------ block --

def scaled_weights(rng, d, mlp, std):
    def one():
        s = I.StreamWeights(w_qkv=bits(rng.normal(0, std, (3 * d, d))), b_qkv=bits(rng.normal(0, std, 3 * d)),
                            w_o=bits(rng.normal(0, std, (d, d))), b_o=bits(rng.normal(0, std, d)))
        if mlp:
            s.w_1 = bits(rng.normal(0, std, (4 * d, d)))
            s.b_1 = bits(rng.normal(0, std, 4 * d))
            s.w_2 = bits(rng.normal(0, std / 2, (d, 4 * d)))
            s.b_2 = bits(rng.normal(0, std, d))
        return s
    return I.BlockWeights(txt=one(), img=one())


@pytest.mark.parametrize("d,heads,T,lens,mlp,sharp", [
    (128, 1, 64, [200], 0, 1.0),          # head_dim 128, ragged text and image tiles
    (128, 2, 64, [256, 77], 1, 1.0),      # head_dim 64, two images of different length
    (256, 2, 0, [130, 300, 5], 1, 1.0),   # no text, three images
    (128, 1, 64, [0, 50], 1, 1.0),        # an image with no image rows: text-only joint sequence
    (512, 8, 200, [384], 1, 1.0),         # several 256-wide GEMM column tiles
    (1024, 8, 256, [4800], 1, 1.0),       # > 76 pair tiles: out-proj / MLP2 tiles split across SM pairs
])
def test_block_forward_matches_oracle(H, d, heads, T, lens, mlp, sharp):
    rng = np.random.default_rng(d + T + len(lens) + int(sharp))
    B = len(lens)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    rows = int(cu[-1])
    cap = rows + 37   # capacity above the used rows: the tail must not matter
    ut = bits(rng.standard_normal((B * T, d)))
    ui = bits(rng.standard_normal((rows, d)))
    w = scaled_weights(rng, d, mlp, std=1.0 / np.sqrt(d))
    grid = int(np.ceil(np.sqrt(cap)))
    sh = H.Shape(B=B, H=2 * grid, W=2 * grid, d=d, T=T, heads=heads, mlp=mlp)
    dw = H.DeviceWeights.from_host(w)
    in_txt = H.bf16_from_bits(ut) if T else torch.empty(0, dtype=torch.bfloat16, device="cuda")
    in_img = torch.full((cap, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    in_img[:rows] = H.bf16_from_bits(ui)
    out = torch.empty(B * T + cap, d, dtype=torch.float32, device="cuda")
    wsb = H.hilo_block_workspace_bytes(sh, cap)
    ws = torch.full((wsb,), 0xFF, dtype=torch.uint8, device="cuda")   # NaN-filled scratch
    H.hilo_block_forward(sh, dw, to_dev_i32(cu), cap, in_txt if T else None, in_img, H.HILO_BF16, out, ws, wsb)
    H.hilo_sync_status()
    ot, oi = O.block(ut, ui, cu, T, w, heads, bool(mlp))
    got = out.cpu().numpy()
    assert_block_close(got[:B * T], ot, "text rows")
    assert_block_close(got[B * T:B * T + rows], oi, "image rows")


def _ws_regions(sh, cap, ws):
    """Views of the block workspace: LayerNorm rows, q|k|v rows, attention rows
    (the layout hilo_block_forward uses: each region 256-byte aligned)."""
    R, d = sh.B * sh.T + cap, sh.d
    a256 = lambda v: (v + 255) // 256 * 256
    o_qkv = a256(R * d * 2)
    o_att = o_qkv + a256(R * 3 * d * 2)
    qkv = ws[o_qkv:o_qkv + R * 3 * d * 2].view(torch.bfloat16).view(R, 3 * d)
    att = ws[o_att:o_att + R * d * 2].view(torch.bfloat16).view(R, d)
    return qkv, att


@pytest.mark.parametrize("d,heads,T,lens,sharp", [
    (256, 2, 128, [1500], 4.0),        # head_dim 128
    (256, 4, 64, [900, 333], 5.0),     # head_dim 64, two images
])
def test_attention_rescale_against_own_qkv(H, d, heads, T, lens, sharp):
    # Large q/k projections spread the logits over tens of units, so the
    # running row maxima jump by more than 2^8 at different key tiles for
    # different rows of one warp. The kernel's attention output is compared
    # with fp64 softmax attention over the same bf16 q, k, v it consumed.
    rng = np.random.default_rng(77 + heads)
    B = len(lens)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    rows = int(cu[-1])
    cap = rows
    w = scaled_weights(rng, d, False, std=1.0 / np.sqrt(d))
    for sw in (w.txt, w.img):
        sw.w_qkv = bits(I.bf16_bits_to_f32(sw.w_qkv) * sharp)
    sh = H.Shape(B=B, H=64, W=64, d=d, T=T, heads=heads, mlp=0)
    ut = bits(rng.standard_normal((B * T, d)))
    ui = bits(rng.standard_normal((rows, d)))
    out = torch.empty(B * T + cap, d, dtype=torch.float32, device="cuda")
    wsb = H.hilo_block_workspace_bytes(sh, cap)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    H.hilo_block_forward(sh, H.DeviceWeights.from_host(w), to_dev_i32(cu), cap, H.bf16_from_bits(ut),
                         H.bf16_from_bits(ui), H.HILO_BF16, out, ws, wsb)
    H.hilo_sync_status()
    qkv_t, att_t = _ws_regions(sh, cap, ws)
    qkv = qkv_t.float().cpu().numpy().astype(np.float64)
    att = att_t.float().cpu().numpy().astype(np.float64)
    hd = d // heads
    n_rescaled_rows = 0
    for b in range(B):
        idx = np.r_[b * T:(b + 1) * T, B * T + cu[b]:B * T + cu[b + 1]]
        for h in range(heads):
            q = qkv[idx, h * hd:(h + 1) * hd]
            k = qkv[idx, d + h * hd:d + (h + 1) * hd]
            v = qkv[idx, 2 * d + h * hd:2 * d + (h + 1) * hd]
            ref = O.softmax_attention(q, k, v)
            # rows whose maximum logit grows by > 8 (log2 units) after the first key tile
            lg = (q @ k.T) / np.sqrt(hd) * np.log2(np.e)
            first = lg[:, :128].max(axis=1) if T >= 128 else lg[:, :T].max(axis=1)
            n_rescaled_rows += int(np.sum(lg.max(axis=1) > first + 8))
            got = att[idx, h * hd:(h + 1) * hd]
            err = np.abs(got - ref)
            # bf16 probabilities and bf16 output: a few 2^-8 relative of the value range
            assert err.max() <= 1.5e-2 * max(1.0, np.abs(ref).max()), (b, h, err.max())
    assert n_rescaled_rows > 0


def test_block_forward_fp32_in_place_chain(H):
    # two blocks chained on the fp32 residual stream, in place
    rng = np.random.default_rng(99)
    d, heads, T = 256, 2, 32
    lens = [150, 64]
    B = len(lens)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    rows = int(cu[-1])
    cap = rows
    ut = bits(rng.standard_normal((B * T, d)))
    ui = bits(rng.standard_normal((rows, d)))
    ws_ = [scaled_weights(rng, d, True, 1.0 / np.sqrt(d)) for _ in range(2)]
    sh = H.Shape(B=B, H=16, W=16, d=d, T=T, heads=heads, mlp=1)
    out = torch.empty(B * T + cap, d, dtype=torch.float32, device="cuda")
    wsb = H.hilo_block_workspace_bytes(sh, cap)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    cud = to_dev_i32(cu)
    H.hilo_block_forward(sh, H.DeviceWeights.from_host(ws_[0]), cud, cap, H.bf16_from_bits(ut),
                         H.bf16_from_bits(ui), H.HILO_BF16, out, ws, wsb)
    H.hilo_block_forward(sh, H.DeviceWeights.from_host(ws_[1]), cud, cap, out, out[B * T:], H.HILO_F32, out,
                         ws, wsb)
    H.hilo_sync_status()
    t1, i1 = O.block(ut, ui, cu, T, ws_[0], heads, True)
    t2, i2 = O.block(t1, i1, cu, T, ws_[1], heads, True)
    got = out.cpu().numpy()
    assert_block_close(got[:B * T], t2, "text rows")
    assert_block_close(got[B * T:], i2, "image rows")


def test_block_image_longer_than_grid(H):
    # cu_img is device data and may describe an image with more packed rows
    # than its H*W grid (anything up to the capacity): the attention's work
    # is derived from the device row counts, so every row is attended.
    rng = np.random.default_rng(5)
    d, heads, T = 128, 1, 0
    lens = [300, 20]                      # image 0: 300 rows on an 8x8 grid (64 tokens)
    B = len(lens)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    rows = int(cu[-1])
    cap = rows + 16
    sh = H.Shape(B=B, H=8, W=8, d=d, T=T, heads=heads, mlp=0)
    ui = bits(rng.standard_normal((cap, d)))
    w = scaled_weights(rng, d, False, 1.0 / np.sqrt(d))
    out = torch.empty(cap, d, dtype=torch.float32, device="cuda")
    wsb = H.hilo_block_workspace_bytes(sh, cap)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    H.hilo_block_forward(sh, H.DeviceWeights.from_host(w), to_dev_i32(cu), cap, None, H.bf16_from_bits(ui),
                         H.HILO_BF16, out, ws, wsb)
    H.hilo_sync_status()
    _, oi = O.block(np.zeros((0, d), np.uint16), ui[:rows], cu, T, w, heads, False)
    assert_block_close(out.cpu().numpy()[:rows], oi, "image rows")


def test_host_argument_errors(H):
    sh = H.Shape(B=1, H=8, W=8, d=128, T=0, heads=1, mlp=0)
    s = torch.empty(64, dtype=torch.float32, device="cuda")
    with pytest.raises(H.HiloError) as e:
        H.hilo_score(H.Shape(B=1, H=7, W=8, d=128), torch.empty(1, device="cuda"), s)
    assert e.value.status == -2
    with pytest.raises(H.HiloError) as e:
        H.hilo_score(sh, None, s)
    assert e.value.status == -1
    with pytest.raises(H.HiloError) as e:
        H.hilo_block_forward(sh, H.DeviceWeights.from_host(scaled_weights(np.random.default_rng(0), 128, False, 0.1)),
                             torch.zeros(2, dtype=torch.int32, device="cuda"), 64, None,
                             torch.empty(64, 128, dtype=torch.bfloat16, device="cuda"), H.HILO_BF16,
                             torch.empty(64, 128, device="cuda"), torch.empty(16, dtype=torch.uint8, device="cuda"), 16)
    assert e.value.status == -4


def test_convert_bf16_to_f16(H):
    rng = np.random.default_rng(31)
    v = np.concatenate([rng.standard_normal(4096) * 0.02, rng.standard_normal(4096) * 100,
                        [1e5, -1e6, 65504.0, 65520.0, 3e-5, 1e-9, 0.0, -0.0]]).astype(np.float32)
    v = np.concatenate([v, np.zeros((-len(v)) % 8, np.float32)])
    b = bits(v)
    src = H.bf16_from_bits(b)
    dst = torch.empty(len(v), dtype=torch.float16, device="cuda")
    H.hilo_convert_bf16_to_f16(src, dst, len(v))
    torch.cuda.synchronize()
    exact = I.bf16_bits_to_f32(b)
    ref = np.clip(exact, -65504, 65504).astype(np.float16)   # round to nearest even, saturate
    assert np.array_equal(dst.cpu().numpy().view(np.uint16), ref.view(np.uint16))
