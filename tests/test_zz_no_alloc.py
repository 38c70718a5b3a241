"""hilo_block_forward_static_ws: the block for callers that cannot allocate.

Such a caller passes no workspace; the call uses the library's built-in
device scratch array instead. It must give the same results as
hilo_block_forward with a caller workspace, also when called twice in a row
with different inputs (the shared scratch keeps the previous call's
contents), and must reject shapes whose scratch would not fit.

This file is collected last, so a run that stops at the first failure has
run every other test before it.
"""
import numpy as np
import pytest
import torch

from paper_2606_13898_gb300 import inputs as I

from .gpu_helpers import assert_block_close, lib_ready

pytestmark = pytest.mark.gpu


def _case(H, seed, lens, d=512, heads=8, T=64, mlp=1):
    rng = np.random.default_rng(seed)
    B = len(lens)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    cap = int(cu[-1]) + 40
    ut = I.f32_to_bf16_bits(rng.standard_normal((B * T, d)).astype(np.float32))
    ui = I.f32_to_bf16_bits(rng.standard_normal((cap, d)).astype(np.float32))
    w = I.make_weights(d, bool(mlp), seed=seed)
    sh = H.Shape(B=B, H=32, W=32, d=d, T=T, heads=heads, mlp=mlp)
    return sh, H.DeviceWeights.from_host(w), torch.from_numpy(cu).cuda(), cap, H.bf16_from_bits(ut), \
        H.bf16_from_bits(ui)


def test_static_scratch_matches_workspace_entry_twice():
    H = lib_ready()
    cases = [_case(H, 5, [700]), _case(H, 6, [300, 1000])]
    # First fill the shared array with NaN: a call whose inputs are all NaN
    # leaves NaN in every scratch region it writes. A kernel that read a
    # scratch value before writing it in the same call would then turn the
    # real cases below non-finite.
    sh, dw, cu, cap, t_in, i_in = cases[1]
    poison = torch.empty(sh.B * sh.T + cap, sh.d, dtype=torch.float32, device="cuda")
    H.hilo_block_forward_static_ws(sh, dw, cu, cap, torch.full_like(t_in, float("nan")),
                                   torch.full_like(i_in, float("nan")), H.HILO_BF16, poison)
    H.hilo_sync_status()
    assert torch.isnan(poison[:sh.B * sh.T + int(cu[-1].item())]).all()
    for sh, dw, cu, cap, t_in, i_in in cases:
        ws_bytes = H.hilo_block_workspace_bytes(sh, cap)
        assert ws_bytes <= 16 << 20
        ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
        ref = torch.empty(sh.B * sh.T + cap, sh.d, dtype=torch.float32, device="cuda")
        H.hilo_block_forward(sh, dw, cu, cap, t_in, i_in, H.HILO_BF16, ref, ws, ws_bytes)
        got = torch.full_like(ref, float("nan"))
        H.hilo_block_forward_static_ws(sh, dw, cu, cap, t_in, i_in, H.HILO_BF16, got)
        H.hilo_sync_status()
        rows = sh.B * sh.T + int(cu[-1].item())
        assert_block_close(got[:rows].cpu().numpy(), ref[:rows].cpu().numpy().astype(np.float64),
                           "static scratch vs caller workspace")


def test_static_scratch_rejects_oversized_shape():
    H = lib_ready()
    sh = H.Shape(B=1, H=64, W=64, d=3072, T=512, heads=24, mlp=1)
    dummy = torch.empty(16, dtype=torch.uint8, device="cuda")
    dw = H.DeviceWeights({(s, f): dummy for s in ("txt", "img")
                          for f in ("w_qkv", "b_qkv", "w_o", "b_o", "w_1", "b_1", "w_2", "b_2")})
    with pytest.raises(H.HiloError) as e:
        H.hilo_block_forward_static_ws(sh, dw, dummy, 4096, dummy, dummy, H.HILO_BF16, dummy)
    assert e.value.status == -4
    assert "scratch bytes" in H.lib().hilo_last_error().decode()
    # an invalid shape is reported as such, not as a scratch size
    bad = H.Shape(B=1, H=8, W=8, d=-128, T=8, heads=1, mlp=1)
    with pytest.raises(H.HiloError) as e:
        H.hilo_block_forward_static_ws(bad, dw, dummy, 64, dummy, dummy, H.HILO_BF16, dummy)
    assert e.value.status == -2
