"""Host logic of the Python binding: the C structs it hands to libhilo.

Shape, SplitBuffers and DeviceWeights build their ctypes structs once per
object. These checks run on the CPU (torch CPU tensors stand in for device
buffers; no library call is made): the cached struct carries the tensors'
current addresses, a replaced split tensor gives a rebuilt struct, and equal
shapes stay equal and hash alike.
"""
import ctypes

import torch

from paper_2606_13898_gb300 import hilo as H


def test_shape_struct_is_built_once_and_matches_fields():
    sh = H.Shape(B=2, H=16, W=24, d=256, T=7, heads=4, mlp=1, levels=2, lf=0)
    c1, c2 = sh.c(), sh.c()
    assert c1 is c2
    assert (c1.B, c1.H, c1.W, c1.d, c1.T, c1.heads, c1.mlp, c1.levels, c1.lf) == (2, 16, 24, 256, 7, 4, 1, 2, 0)
    other = H.Shape(B=2, H=16, W=24, d=256, T=7, heads=4, mlp=1, levels=2, lf=0)
    assert sh == other and hash(sh) == hash(other)
    assert "_c" not in repr(sh)


def test_split_struct_follows_replaced_tensors():
    sp = H.SplitBuffers(*(torch.empty(8, dtype=torch.int32) for _ in range(5)))
    c = sp.c()
    assert sp.c() is c
    assert c.labels == sp.labels.data_ptr() and c.tok_row == sp.tok_row.data_ptr()
    sp.cu_img = torch.empty(3, dtype=torch.int32)
    c2 = sp.c()
    assert c2 is not c and c2.cu_img == sp.cu_img.data_ptr() and c2.labels == sp.labels.data_ptr()


def test_weights_struct_carries_every_pointer():
    names = ("w_qkv", "b_qkv", "w_o", "b_o", "w_1", "b_1", "w_2", "b_2")
    t = {(s, f): torch.empty(4) for s in ("txt", "img") for f in names}
    t[("txt", "w_1")] = None  # an absent MLP weight is a NULL pointer
    dw = H.DeviceWeights(t)
    c = dw.c()
    assert dw.c() is c
    for s, st in (("txt", c.txt), ("img", c.img)):
        for f in names:
            want = t[(s, f)].data_ptr() if t[(s, f)] is not None else None
            assert getattr(st, f) == want, (s, f)
    assert ctypes.sizeof(c) == 16 * ctypes.sizeof(ctypes.c_void_p)
