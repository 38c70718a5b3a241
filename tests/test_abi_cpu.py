"""The C-ABI library builds, loads and exports every symbol of include/hilo.h.

No test here needs a GPU: calls are limited to pure host queries and to
argument/shape errors that the library rejects before touching the device.
"""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def H():
    from paper_2606_13898_gb300 import build
    from paper_2606_13898_gb300 import hilo

    build.build()
    hilo.lib()
    return hilo


def declared_functions():
    names = []
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            txt = open(os.path.join(ROOT, "include", f)).read()
            txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
            names += re.findall(r"\b(hilo_[a-z0-9_]+)\s*\(", txt)
    return sorted(set(names))


def test_exports_every_declared_symbol(H):
    L = H.lib()
    names = declared_functions()
    assert len(names) >= 12
    for n in names:
        assert hasattr(L, n), n
    assert set(H.EXPORTS) <= set(names)


def test_status_strings(H):
    L = H.lib()
    assert L.hilo_status_string(0) == b"HILO_OK"
    assert L.hilo_status_string(-5) == b"HILO_ERR_TIMEOUT"
    assert L.hilo_status_string(123) == b"HILO_ERR_UNKNOWN"


@pytest.mark.parametrize("bad,code", [
    (dict(H=7), -2), (dict(W=0), -2), (dict(d=100), -2), (dict(d=8192), -2), (dict(B=0), -2),
    (dict(levels=3), -2), (dict(levels=2, H=6), -2), (dict(H=256, W=256), -2),
    (dict(B=140000, H=128, W=128), -2),  # 2.3e9 rows: past the int32 row space
])
def test_shape_rejected_before_launch(H, bad, code):
    kw = dict(B=1, H=8, W=8, d=128, T=4, heads=1, mlp=0, levels=1)
    kw.update(bad)
    s = H.hilo_shape(*(kw[k] for k in ("B", "H", "W", "d", "T", "heads", "mlp", "levels")))
    L = H.lib()
    assert L.hilo_score(ctypes.byref(s), 1, 1, None) == code
    assert L.hilo_last_error() != b""


@pytest.mark.parametrize("bad", [dict(heads=3), dict(heads=4, d=128), dict(mlp=2), dict(T=-1)])
def test_block_shape_rejected(H, bad):
    kw = dict(B=1, H=8, W=8, d=256, T=4, heads=2, mlp=1, levels=1)
    kw.update(bad)
    s = H.hilo_shape(*(kw[k] for k in ("B", "H", "W", "d", "T", "heads", "mlp", "levels")))
    w = H.hilo_block_weights()
    rc = H.lib().hilo_block_forward(ctypes.byref(s), ctypes.byref(w), 1, 64, 1, 1, 0, 1, 1, 1 << 30, None)
    assert rc == -2


def test_null_pointers_rejected(H):
    s = H.hilo_shape(1, 8, 8, 128, 4, 1, 1, 1)
    L = H.lib()
    assert L.hilo_score(ctypes.byref(s), None, 1, None) == -1
    assert L.hilo_score(None, 1, 1, None) == -1
    sp = H.hilo_split_out()
    assert L.hilo_split(ctypes.byref(s), 1, 1, 1, 1, ctypes.byref(sp), None, 0, None) == -1
    w = H.hilo_block_weights()
    assert L.hilo_block_forward(ctypes.byref(s), ctypes.byref(w), 1, 64, 1, 1, 0, 1, 1, 1 << 30, None) == -1


def test_regions_entry_points_check_arguments(H):
    """hilo_split_regions validates like hilo_split; hilo_unpack_delta rejects
    NULL and unaligned pointers before any launch."""
    s = H.hilo_shape(1, 8, 8, 128, 4, 1, 1, 1)
    L = H.lib()
    sp = H.hilo_split_out()
    assert L.hilo_split_regions(ctypes.byref(s), 1, 1, 1, 1, ctypes.byref(sp), None, 0, None) == -1
    bad = H.hilo_shape(1, 7, 8, 128, 4, 1, 1, 1)
    for f in ("labels", "row_src", "counts", "cu_img", "tok_row"):
        setattr(sp, f, 256)
    assert L.hilo_split_regions(ctypes.byref(bad), 1, 1, 1, 1, ctypes.byref(sp), None, 0, None) == -2
    s2 = H.hilo_shape(1, 8, 8, 128, 4, 1, 1, 2)
    assert L.hilo_split_regions(ctypes.byref(s2), 1, 1, 1, None, ctypes.byref(sp), None, 0, None) == -1
    assert L.hilo_unpack_delta(ctypes.byref(s), 256, None, 256, ctypes.byref(sp), 256, None) == -1
    assert L.hilo_unpack_delta(ctypes.byref(s), 260, 256, 256, ctypes.byref(sp), 256, None) == -1
    assert L.hilo_unpack_delta(ctypes.byref(s), 256, 256, 264, ctypes.byref(sp), 256, None) == -1


def test_prop_entry_points_check_arguments(H):
    s = H.hilo_shape(1, 8, 8, 128, 4, 1, 1, 1)
    L = H.lib()
    w = H.hilo_block_weights()
    for f in ("txt", "img"):
        sw = getattr(w, f)
        for n in ("w_qkv", "b_qkv", "w_o", "b_o", "w_1", "b_1", "w_2", "b_2"):
            setattr(sw, n, 256)
    assert L.hilo_block_forward_prop(ctypes.byref(s), ctypes.byref(w), 256, 64, 256, 256, 0, None, 256, 256,
                                     1 << 30, None) == -1
    assert L.hilo_block_forward_prop(ctypes.byref(s), ctypes.byref(w), 256, 64, 256, 256, 0, 258, 256, 256,
                                     1 << 30, None) == -1
    sp = H.hilo_split_out()
    assert L.hilo_row_sizes(ctypes.byref(s), ctypes.byref(sp), 256, 64, None) == -1
    for f in ("labels", "row_src", "counts", "cu_img", "tok_row"):
        setattr(sp, f, 256)
    assert L.hilo_row_sizes(ctypes.byref(s), ctypes.byref(sp), None, 64, None) == -1
    assert L.hilo_row_sizes(ctypes.byref(s), ctypes.byref(sp), 256, -1, None) == -1


def test_lf_shape_checks_and_row_capacity(H):
    L = H.lib()
    ok = H.hilo_shape(2, 8, 12, 128, 4, 1, 1, 1, 4)
    assert L.hilo_row_capacity(ctypes.byref(ok)) == 2 * (96 + 96 // 16)
    assert L.hilo_row_capacity(ctypes.byref(H.hilo_shape(2, 8, 12, 128, 4, 1, 1, 1, 0))) == 2 * 96
    for bad in (H.hilo_shape(1, 8, 12, 128, 4, 1, 1, 1, 3), H.hilo_shape(1, 8, 12, 128, 4, 1, 1, 2, 4),
                H.hilo_shape(1, 8, 12, 128, 4, 1, 1, 1, 8)):
        assert L.hilo_row_capacity(ctypes.byref(bad)) == 0
        assert L.hilo_score(ctypes.byref(bad), 256, 256, None) == -2
    sp = H.hilo_split_out()
    for f in ("labels", "row_src", "counts", "cu_img", "tok_row"):
        setattr(sp, f, 256)
    assert L.hilo_split_regions(ctypes.byref(ok), 256, 256, 256, 256, ctypes.byref(sp), None, 0, None) == -1


def test_workspace_size_and_check(H):
    s = H.hilo_shape(2, 64, 64, 3072, 512, 24, 1, 1)
    cap = 2 * 4096
    nb = H.lib().hilo_block_workspace_bytes(ctypes.byref(s), cap)
    R = 2 * 512 + cap
    assert nb >= R * 3072 * 2 * (1 + 3 + 1 + 4)
    s0 = H.hilo_shape(2, 64, 64, 3072, 512, 24, 0, 1)
    assert H.lib().hilo_block_workspace_bytes(ctypes.byref(s0), cap) < nb
    w = H.hilo_block_weights()
    for f in ("txt", "img"):
        sw = getattr(w, f)
        for n in ("w_qkv", "b_qkv", "w_o", "b_o", "w_1", "b_1", "w_2", "b_2"):
            setattr(sw, n, 1)
    rc = H.lib().hilo_block_forward(ctypes.byref(s), ctypes.byref(w), 1, cap, 256, 256, 0, 256, 1, nb - 1, None)
    assert rc == -4
    # the rows are read with 16-byte copies: unaligned row buffers are refused
    for args in ((264, 256, 256), (256, 260, 256), (256, 256, 258)):
        rc = H.lib().hilo_block_forward(ctypes.byref(s), ctypes.byref(w), 1, cap, *args[:2], 0, args[2], 1, nb, None)
        assert rc == -1
        assert b"16-byte aligned" in H.lib().hilo_last_error()


@pytest.mark.parametrize("channels,patch,radius,thr,code", [
    (0, 16, 1, 0.1, -1), (5, 16, 1, 0.1, -1), (3, 12, 1, 0.1, -1), (3, 16, -1, 0.1, -1),
    (3, 16, 1, float("nan"), -1), (3, 16, 1, float("inf"), -1), (3, 16, 65, 0.1, -1),
])
def test_sobel_select_arguments_rejected_before_launch(H, channels, patch, radius, thr, code):
    s = H.hilo_shape(1, 8, 8, 128, 4, 1, 0, 1)
    L = H.lib()
    assert L.hilo_sobel_select(ctypes.byref(s), 1, channels, patch, 1, radius, ctypes.c_float(thr), 1, 16,
                               1 << 20, None) == code


def test_sobel_workspace_query(H):
    s = H.hilo_shape(2, 8, 8, 128, 4, 1, 0, 1)
    n = H.lib().hilo_sobel_workspace_bytes(ctypes.byref(s))
    assert n >= 2 * 64 * 4 + 2 * 4
    s0 = H.hilo_shape(2, 7, 8, 128, 4, 1, 0, 1)
    assert H.lib().hilo_sobel_workspace_bytes(ctypes.byref(s0)) == 0
