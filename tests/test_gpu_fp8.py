"""FP8 (e4m3) GEMM operands on the GPU against the oracle.

Three levels. The per-row quantisation kernel must reproduce the oracle's
codes and scales bit for bit (same fp32 operations, round to nearest even,
saturation). The FP8 GEMM with its dequantising epilogue is isolated on an
attention-only block: its out-projection is recomputed from the GPU's own
e4m3 codes and scales (left in the workspace), leaving only the fp32
accumulation order (tolerance 1e-4 relative). The whole block is compared
with the oracle's FP8 emulation (the kernels' rounding points; codes can
flip where a bf16 intermediate rounds differently) and with the exact block,
whose distance follows the e4m3 error model (a few percent of the block's
update).
"""
import numpy as np
import pytest
import torch

from oracle import hilo_oracle as O
from paper_2606_13898_gb300 import inputs as I

from .gpu_helpers import lib_ready, to_dev_i32
from .test_gpu_kernels import bits, scaled_weights

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def H():
    return lib_ready()


@pytest.mark.parametrize("dtype", ["bf16", "f16", "f32"])
def test_quantize_rows_bitexact(H, dtype):
    rng = np.random.default_rng(5)
    rows, cols = 37, 1032
    x = (rng.standard_normal((rows, cols)) * np.exp(rng.uniform(-10, 10, (rows, 1)))).astype(np.float32)
    x[4] = 0.0
    x[5, :8] = [448.0, -1000.0, 2 ** -12, 1e-30, 0.0, -0.0, 3.0, -3.0]
    if dtype == "bf16":
        xb = bits(x)
        src, code = H.bf16_from_bits(xb), H.HILO_BF16
        xf = O.bf16_to_f32(xb)
    elif dtype == "f16":
        xf = np.clip(x, -60000, 60000).astype(np.float16).astype(np.float32)
        src, code = torch.from_numpy(xf.astype(np.float16)).cuda(), H.HILO_F16
    else:
        xf = x
        src, code = torch.from_numpy(x).cuda(), H.HILO_F32
    q = torch.empty(rows, cols, dtype=torch.uint8, device="cuda")
    sc = torch.empty(rows, dtype=torch.float32, device="cuda")
    H.hilo_quantize_rows_e4m3(src, code, rows, cols, q, sc)
    H.hilo_sync_status()
    cref, sref = O.quantize_rows(xf)
    assert np.array_equal(q.cpu().numpy(), cref)
    assert np.array_equal(sc.cpu().numpy(), sref)


def _ws8(H, sh, cap, ws):
    """Views of the FP8 block workspace (layout of hilo_block_forward_fp8:
    e4m3 rows, their scales, q|k|v, attention rows; 256-byte aligned)."""
    R, d = sh.B * sh.T + cap, sh.d
    a256 = lambda v: (v + 255) // 256 * 256
    o_qs = a256(R * (4 * d if sh.mlp else d))
    o_qkv = o_qs + a256(R * 4)
    o_att = o_qkv + a256(R * 3 * d * 2)
    q8 = ws[:R * d].view(R, d)
    qs = ws[o_qs:o_qs + R * 4].view(torch.float32)
    qkv = ws[o_qkv:o_qkv + R * 3 * d * 2].view(torch.bfloat16).view(R, 3 * d)
    att = ws[o_att:o_att + R * d * 2].view(torch.bfloat16).view(R, d)
    return q8, qs, qkv, att


def _run(H, d, heads, T, lens, mlp, seed):
    rng = np.random.default_rng(seed)
    B = len(lens)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    rows = int(cu[-1])
    cap = rows + 29
    ut = bits(rng.standard_normal((B * T, d)))
    ui = bits(rng.standard_normal((rows, d)))
    w = scaled_weights(rng, d, mlp, std=1.0 / np.sqrt(d))
    grid = int(np.ceil(np.sqrt(cap)))
    sh = H.Shape(B=B, H=2 * grid, W=2 * grid, d=d, T=T, heads=heads, mlp=mlp)
    w8 = H.DeviceWeightsFP8.from_host(w)
    in_img = torch.full((cap, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    in_img[:rows] = H.bf16_from_bits(ui)
    out = torch.empty(B * T + cap, d, dtype=torch.float32, device="cuda")
    wsb = H.hilo_block_fp8_workspace_bytes(sh, cap)
    ws = torch.full((wsb,), 0xFF, dtype=torch.uint8, device="cuda")
    H.hilo_block_forward_fp8(sh, w8, to_dev_i32(cu), cap, H.bf16_from_bits(ut) if T else None, in_img,
                             H.HILO_BF16, out, ws, wsb)
    H.hilo_sync_status()
    return dict(sh=sh, cu=cu, rows=rows, cap=cap, ut=ut, ui=ui, w=w, w8=w8, out=out.cpu().numpy(), ws=ws)


def test_device_weights_match_oracle_quantisation(H):
    rng = np.random.default_rng(3)
    w = scaled_weights(rng, 1024, 1, std=1.0 / 32)
    w8 = H.DeviceWeightsFP8.from_host(w)
    wq = O.quantize_weights(w)
    for s in ("txt", "img"):
        for m in ("qkv", "o", "1", "2"):
            codes, scale = getattr(getattr(wq, s), "w_" + m)
            assert np.array_equal(w8.tensors[(s, "w_" + m)].cpu().numpy(), codes)
            assert np.array_equal(w8.tensors[(s, "s_" + m)].cpu().numpy(), scale)


@pytest.mark.parametrize("lens,T", [([300, 77], 64), ([520], 0)])
def test_fp8_gemm_isolated_on_attention_only_block(H, lens, T):
    """Out-projection of an attention-only block: out = u + (codes_A codes_W^T)
    * scale_A * scale_W + b with the GPU's own quantised attention rows."""
    r = _run(H, 1024, 8, T, lens, 0, 11 + T)
    sh, cap, rows = r["sh"], r["cap"], r["rows"]
    BT = sh.B * sh.T
    q8, qs, qkv, att = _ws8(H, sh, cap, r["ws"])
    nr = BT + rows
    # the quantised attention rows are the oracle's quantisation of the GPU's bf16 attention rows
    codes, scale = O.quantize_rows(O.bf16_to_f32(H.bits_from_bf16(att[:nr])))
    assert np.array_equal(q8[:nr].cpu().numpy(), codes)
    assert np.array_equal(qs[:nr].cpu().numpy(), scale)
    wq = O.quantize_weights(r["w"])
    u = np.concatenate([O.bf16_to_f32(r["ut"]), O.bf16_to_f32(r["ui"])]).astype(np.float64)
    dq = O.e4m3_decode(codes)
    for lo, hi, s in ((0, BT, wq.txt), (BT, nr, wq.img)):
        if hi == lo:
            continue
        cw, sw = s.w_o
        ref = u[lo:hi] + (dq[lo:hi] @ O.e4m3_decode(cw).T) * scale[lo:hi, None].astype(np.float64) \
            * sw[None, :].astype(np.float64) + O.bf16_to_f32(s.b_o)
        got = r["out"][lo:hi]
        assert np.max(np.abs(got - ref)) <= 1e-4 * (1 + np.max(np.abs(ref)))


@pytest.mark.parametrize("d,heads,T,lens", [
    (1024, 8, 64, [300, 77]),
    (2048, 16, 128, [400]),
])
def test_block_forward_fp8_against_oracle(H, d, heads, T, lens):
    r = _run(H, d, heads, T, lens, 1, d + T)
    BT = r["sh"].B * T
    rows = r["rows"]
    got_t, got_i = r["out"][:BT], r["out"][BT:BT + rows]
    wq = O.quantize_weights(r["w"])
    qt, qi = O.block_fp8(r["ut"], r["ui"], r["cu"], T, wq, heads, True)
    et, ei = O.block(r["ut"], r["ui"], r["cu"], T, r["w"], heads, True)
    for got, emu, ex, u in ((got_i, qi, ei, r["ui"]), (got_t, qt, et, r["ut"])):
        assert np.all(np.isfinite(got))
        delta = np.linalg.norm(ex - O.bf16_to_f32(u).astype(np.float64))
        # against the emulation: code flips where a bf16 intermediate rounds
        # differently (mostly the attention output) stay well below the FP8 error
        e_emu = np.linalg.norm(got - emu) / delta
        # against the exact block: the e4m3 error model
        e_ex = np.linalg.norm(got - ex) / delta
        assert e_emu < 0.03, e_emu
        assert 0.005 < e_ex < 0.1, e_ex


@pytest.mark.parametrize("d,heads,T,lens", [
    (1024, 8, 64, [300, 77]),
    (2048, 16, 128, [400]),
])
def test_block_forward_fp8_prop_against_oracle(H, d, heads, T, lens):
    """Proportional attention in the FP8 block: each packed row weighted by a
    row size (1..16, as pooled windows give), against the oracle's FP8
    emulation with the same weights and the exact proportional block."""
    rng = np.random.default_rng(d + 7)
    B = len(lens)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    rows = int(cu[-1])
    cap = rows + 29
    ut = bits(rng.standard_normal((B * T, d)))
    ui = bits(rng.standard_normal((rows, d)))
    n = rng.choice([1.0, 1.0, 2.0, 3.0, 4.0, 16.0], size=rows).astype(np.float32)
    w = scaled_weights(rng, d, 1, std=1.0 / np.sqrt(d))
    grid = int(np.ceil(np.sqrt(cap)))
    sh = H.Shape(B=B, H=2 * grid, W=2 * grid, d=d, T=T, heads=heads, mlp=1)
    w8 = H.DeviceWeightsFP8.from_host(w)
    in_img = torch.full((cap, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    in_img[:rows] = H.bf16_from_bits(ui)
    n_dev = torch.ones(cap, dtype=torch.float32, device="cuda")
    n_dev[:rows] = torch.from_numpy(n).cuda()
    out = torch.empty(B * T + cap, d, dtype=torch.float32, device="cuda")
    wsb = H.hilo_block_fp8_workspace_bytes(sh, cap)
    ws = torch.full((wsb,), 0xFF, dtype=torch.uint8, device="cuda")
    H.hilo_block_forward_fp8_prop(sh, w8, to_dev_i32(cu), cap, H.bf16_from_bits(ut) if T else None, in_img,
                                  H.HILO_BF16, n_dev, out, ws, wsb)
    H.hilo_sync_status()
    o = out.cpu().numpy()
    BT = B * T
    wq = O.quantize_weights(w)
    qt, qi = O.block_fp8(ut, ui, cu, T, wq, heads, True, n_img=n)
    et, ei = O.block(ut, ui, cu, T, w, heads, True, n_img=n)
    pt, pi = O.block_fp8(ut, ui, cu, T, wq, heads, True)
    for got, emu, ex, plain, u in ((o[BT:BT + rows], qi, ei, pi, ui), (o[:BT], qt, et, pt, ut)):
        assert np.all(np.isfinite(got))
        delta = np.linalg.norm(ex - O.bf16_to_f32(u).astype(np.float64))
        e_emu = np.linalg.norm(got - emu) / delta
        e_ex = np.linalg.norm(got - ex) / delta
        assert e_emu < 0.03, e_emu
        assert 0.005 < e_ex < 0.1, e_ex
        # the weights are applied: the unweighted FP8 block is much further away
        assert np.linalg.norm(got - plain) / delta > 3 * e_emu
