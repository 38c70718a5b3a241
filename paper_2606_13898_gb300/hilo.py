"""Thin Python binding of libhilo's C ABI (include/hilo.h): the HiLo-Token
hot path of paper Sec. 2.3 around the DiT block of Sec. 2.1.

Functions carry the C names and only marshal arguments: torch tensors are
passed as device pointers, the shape as a ``hilo_shape`` struct, the stream
as the current torch stream. Every step of the hot path runs in libhilo's
CUDA kernels; there is no Python or CPU fallback. If the library has not been
built, or the device is not an sm_103 GPU, the calls raise.

PyTorch is used for device memory and streams only.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os

import numpy as np
import torch

from . import build as _build

HILO_OK = 0
HILO_F16 = 2
HILO_ERR_SHAPE = -2
HILO_ERR_TIMEOUT, HILO_ERR_CHECK = -5, -7
HILO_KEEP, HILO_POOL2, HILO_POOL4 = 0, 1, 2
HILO_BF16, HILO_F32 = 0, 1


class HiloError(RuntimeError):
    def __init__(self, fn: str, status: int, detail: str):
        super().__init__(f"{fn} failed: {status} ({detail})")
        self.status = status


class hilo_shape(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("B", "H", "W", "d", "T", "heads", "mlp", "levels", "lf")]


class hilo_split_out(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("labels", "row_src", "counts", "cu_img", "tok_row")]


class hilo_stream_weights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("w_qkv", "b_qkv", "w_o", "b_o", "w_1", "b_1", "w_2", "b_2")]


class hilo_block_weights(ctypes.Structure):
    _fields_ = [("txt", hilo_stream_weights), ("img", hilo_stream_weights)]


_FP8_FIELDS = ("w_qkv", "w_o", "w_1", "w_2", "s_qkv", "s_o", "s_1", "s_2", "b_qkv", "b_o", "b_1", "b_2")


class hilo_stream_weights_fp8(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in _FP8_FIELDS]


class hilo_block_weights_fp8(ctypes.Structure):
    _fields_ = [("txt", hilo_stream_weights_fp8), ("img", hilo_stream_weights_fp8)]


EXPORTS = ("hilo_status_string", "hilo_last_error", "hilo_sync_status", "hilo_device_info",
           "hilo_score", "hilo_split_workspace_bytes", "hilo_split", "hilo_pack",
           "hilo_block_workspace_bytes", "hilo_block_forward", "hilo_unpack", "hilo_unpack_update",
           "hilo_convert_bf16_to_f16", "hilo_set_stage_events", "hilo_launch_count",
           "hilo_block_forward_static_ws", "hilo_sobel_workspace_bytes", "hilo_sobel_select",
           "hilo_split_regions", "hilo_unpack_delta", "hilo_row_sizes", "hilo_block_forward_prop",
           "hilo_row_capacity", "hilo_quantize_rows_e4m3", "hilo_block_fp8_workspace_bytes",
           "hilo_block_forward_fp8", "hilo_block_forward_fp8_prop", "hilo_debug_wait_timeout")

_lib = None


def library_path() -> str:
    """The library to load: HILO_LIBRARY if set (e.g. the checks build), else the in-tree build."""
    return os.environ.get("HILO_LIBRARY") or _build.LIB


def lib() -> ctypes.CDLL:
    """Load libhilo.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    path = library_path()
    if not os.path.exists(path):
        raise RuntimeError(f"libhilo is not built ({path} missing); run paper_2606_13898_gb300.build.build()")
    L = ctypes.CDLL(path)
    P, I, S, F = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t, ctypes.c_float
    shp = ctypes.POINTER(hilo_shape)
    spo = ctypes.POINTER(hilo_split_out)
    sig = {
        "hilo_status_string": (ctypes.c_char_p, [I]),
        "hilo_last_error": (ctypes.c_char_p, []),
        "hilo_sync_status": (I, [P]),
        "hilo_debug_wait_timeout": (I, [P]),
        "hilo_device_info": (I, [ctypes.POINTER(I), ctypes.POINTER(I)]),
        "hilo_score": (I, [shp, P, P, P]),
        "hilo_split_workspace_bytes": (S, [shp]),
        "hilo_split": (I, [shp, P, P, P, P, spo, P, S, P]),
        "hilo_pack": (I, [shp, P, spo, P, ctypes.c_int32, P]),
        "hilo_block_workspace_bytes": (S, [shp, ctypes.c_int32]),
        "hilo_block_forward": (I, [shp, ctypes.POINTER(hilo_block_weights), P, ctypes.c_int32, P, P, I,
                                   P, P, S, P]),
        "hilo_unpack": (I, [shp, P, spo, P, P]),
        "hilo_unpack_update": (I, [shp, P, spo, P, F, P]),
        "hilo_convert_bf16_to_f16": (I, [P, P, S, P]),
        "hilo_block_forward_static_ws": (I, [shp, ctypes.POINTER(hilo_block_weights), P, ctypes.c_int32, P,
                                             P, I, P, P]),
        "hilo_set_stage_events": (I, [ctypes.POINTER(ctypes.c_void_p), I]),
        "hilo_launch_count": (ctypes.c_ulonglong, []),
        "hilo_sobel_workspace_bytes": (S, [shp]),
        "hilo_sobel_select": (I, [shp, P, I, I, P, I, F, P, P, S, P]),
        "hilo_split_regions": (I, [shp, P, P, P, P, spo, P, S, P]),
        "hilo_unpack_delta": (I, [shp, P, P, P, spo, P, P]),
        "hilo_row_sizes": (I, [shp, spo, P, ctypes.c_int32, P]),
        "hilo_row_capacity": (S, [shp]),
        "hilo_quantize_rows_e4m3": (I, [P, I, ctypes.c_int64, ctypes.c_int32, P, P, P]),
        "hilo_block_fp8_workspace_bytes": (S, [shp, ctypes.c_int32]),
        "hilo_block_forward_fp8": (I, [shp, ctypes.POINTER(hilo_block_weights_fp8), P, ctypes.c_int32, P, P, I,
                                       P, P, S, P]),
        "hilo_block_forward_fp8_prop": (I, [shp, ctypes.POINTER(hilo_block_weights_fp8), P, ctypes.c_int32, P, P,
                                            I, P, P, P, S, P]),
        "hilo_block_forward_prop": (I, [shp, ctypes.POINTER(hilo_block_weights), P, ctypes.c_int32, P, P, I,
                                        P, P, P, S, P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    _lib = L
    return L


def _ptr(t) -> int | None:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(fn: str, status: int) -> None:
    if status != HILO_OK:
        detail = lib().hilo_last_error().decode()
        raise HiloError(fn, status, detail)


@dataclasses.dataclass(frozen=True)
class Shape:
    B: int
    H: int
    W: int
    d: int
    T: int = 0
    heads: int = 1
    mlp: int = 1
    levels: int = 1
    lf: int = 0

    @property
    def N(self) -> int:
        return self.H * self.W

    def c(self) -> hilo_shape:
        """The C struct, built once per (frozen) shape; the C entry points
        only read it (const hilo_shape*)."""
        st = self.__dict__.get("_c")
        if st is None:
            st = hilo_shape(self.B, self.H, self.W, self.d, self.T, self.heads, int(self.mlp), self.levels, self.lf)
            self.__dict__["_c"] = st
        return st


@dataclasses.dataclass
class SplitBuffers:
    """Device outputs of hilo_split for one shape (allocated with torch)."""

    labels: torch.Tensor
    row_src: torch.Tensor
    counts: torch.Tensor
    cu_img: torch.Tensor
    tok_row: torch.Tensor

    @staticmethod
    def alloc(shape: Shape, device="cuda") -> "SplitBuffers":
        n = shape.B * shape.N
        return SplitBuffers(
            labels=torch.empty(n, dtype=torch.uint8, device=device),
            row_src=torch.empty(hilo_row_capacity(shape), dtype=torch.int32, device=device),
            counts=torch.empty(3 * shape.B, dtype=torch.int32, device=device),
            cu_img=torch.empty(shape.B + 1, dtype=torch.int32, device=device),
            tok_row=torch.empty(n, dtype=torch.int32, device=device))

    def c(self) -> hilo_split_out:
        """The C struct of the five device pointers, rebuilt only when one of
        the tensors is replaced."""
        ts = (self.labels, self.row_src, self.counts, self.cu_img, self.tok_row)
        key = tuple(id(t) for t in ts)
        cached = self.__dict__.get("_c")
        if cached is None or cached[0] != key:
            cached = (key, hilo_split_out(*(t.data_ptr() for t in ts)), ts)
            self.__dict__["_c"] = cached
        return cached[1]


def bf16_from_bits(a: np.ndarray, device="cuda") -> torch.Tensor:
    """uint16 bf16 bit patterns (numpy) -> bf16 torch tensor on ``device``."""
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(device)


def bits_from_bf16(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


@dataclasses.dataclass
class DeviceWeights:
    """Device copies of one block's weights (both streams): bf16, except the
    MLP matrices w_1 / w_2, which are converted once to fp16 on the device
    (hilo_convert_bf16_to_f16)."""

    tensors: dict

    @staticmethod
    def from_host(w, device="cuda") -> "DeviceWeights":
        t = {}
        for sname in ("txt", "img"):
            sw = getattr(w, sname)
            for f in ("w_qkv", "b_qkv", "w_o", "b_o", "w_1", "b_1", "w_2", "b_2"):
                v = getattr(sw, f)
                if v is None:
                    t[(sname, f)] = None
                elif f in ("w_1", "w_2"):
                    src = bf16_from_bits(v, device)
                    dst = torch.empty(src.shape, dtype=torch.float16, device=device)
                    hilo_convert_bf16_to_f16(src, dst, src.numel())
                    t[(sname, f)] = dst
                else:
                    t[(sname, f)] = bf16_from_bits(v, device)
        torch.cuda.synchronize()
        return DeviceWeights(t)

    def c(self) -> hilo_block_weights:
        """The C struct of the block's device pointers, built once: the
        tensors of a DeviceWeights are fixed after construction."""
        st = self.__dict__.get("_c")
        if st is None:
            def sw(s):
                return hilo_stream_weights(*(_ptr(self.tensors[(s, f)]) for f in
                                             ("w_qkv", "b_qkv", "w_o", "b_o", "w_1", "b_1", "w_2", "b_2")))
            st = hilo_block_weights(sw("txt"), sw("img"))
            self.__dict__["_c"] = st
        return st


@dataclasses.dataclass
class DeviceWeightsFP8:
    """One block's weights for hilo_block_forward_fp8: every matrix as e4m3
    codes with one fp32 scale per output channel, quantised on the device
    from the bf16 values (hilo_quantize_rows_e4m3); biases bf16."""

    tensors: dict

    @staticmethod
    def from_host(w, device="cuda") -> "DeviceWeightsFP8":
        t = {}
        for sname in ("txt", "img"):
            sw = getattr(w, sname)
            for m in ("qkv", "o", "1", "2"):
                v, b = getattr(sw, "w_" + m), getattr(sw, "b_" + m)
                if v is None:
                    t[(sname, "w_" + m)] = t[(sname, "s_" + m)] = t[(sname, "b_" + m)] = None
                    continue
                src = bf16_from_bits(v, device)
                q = torch.empty(src.shape, dtype=torch.uint8, device=device)
                sc = torch.empty(src.shape[0], dtype=torch.float32, device=device)
                hilo_quantize_rows_e4m3(src, HILO_BF16, src.shape[0], src.shape[1], q, sc)
                t[(sname, "w_" + m)], t[(sname, "s_" + m)] = q, sc
                t[(sname, "b_" + m)] = bf16_from_bits(b, device)
        torch.cuda.synchronize()
        return DeviceWeightsFP8(t)

    def c(self) -> hilo_block_weights_fp8:
        """The C struct of the block's device pointers, built once (as for
        DeviceWeights)."""
        st = self.__dict__.get("_c")
        if st is None:
            def sw(s):
                return hilo_stream_weights_fp8(*(_ptr(self.tensors[(s, f)]) for f in _FP8_FIELDS))
            st = hilo_block_weights_fp8(sw("txt"), sw("img"))
            self.__dict__["_c"] = st
        return st


# ---------------------------------------------------------------------------
# The C entry points
# ---------------------------------------------------------------------------


def hilo_device_info() -> tuple[int, int]:
    n, s = ctypes.c_int(), ctypes.c_int()
    _check("hilo_device_info", lib().hilo_device_info(ctypes.byref(n), ctypes.byref(s)))
    return n.value, s.value


def hilo_sync_status(stream=None) -> None:
    _check("hilo_sync_status", lib().hilo_sync_status(_stream(stream)))


def hilo_debug_wait_timeout(stream=None) -> None:
    """Launch the wait-timeout probe; the next hilo_sync_status raises HILO_ERR_TIMEOUT."""
    _check("hilo_debug_wait_timeout", lib().hilo_debug_wait_timeout(_stream(stream)))


def hilo_score(shape: Shape, x, score, stream=None) -> None:
    s = shape.c()
    _check("hilo_score", lib().hilo_score(ctypes.byref(s), _ptr(x), _ptr(score), _stream(stream)))


def hilo_row_capacity(shape: Shape) -> int:
    s = shape.c()
    n = int(lib().hilo_row_capacity(ctypes.byref(s)))
    if n == 0:
        raise HiloError("hilo_row_capacity", HILO_ERR_SHAPE, lib().hilo_last_error().decode())
    return n


def hilo_split_workspace_bytes(shape: Shape) -> int:
    s = shape.c()
    return lib().hilo_split_workspace_bytes(ctypes.byref(s))


def hilo_split(shape: Shape, score, mask, k_keep, k_mid, out: SplitBuffers, ws=None, ws_bytes=0,
               stream=None) -> None:
    s = shape.c()
    o = out.c()
    _check("hilo_split", lib().hilo_split(ctypes.byref(s), _ptr(score), _ptr(mask), _ptr(k_keep), _ptr(k_mid),
                                          ctypes.byref(o), _ptr(ws), ws_bytes, _stream(stream)))


def hilo_split_regions(shape: Shape, score, mask, k_keep, k_mid, out: SplitBuffers, ws=None, ws_bytes=0,
                       stream=None) -> None:
    s = shape.c()
    o = out.c()
    _check("hilo_split_regions", lib().hilo_split_regions(ctypes.byref(s), _ptr(score), _ptr(mask), _ptr(k_keep),
                                                          _ptr(k_mid), ctypes.byref(o), _ptr(ws), ws_bytes,
                                                          _stream(stream)))


def hilo_sobel_workspace_bytes(shape: Shape) -> int:
    s = shape.c()
    return int(lib().hilo_sobel_workspace_bytes(ctypes.byref(s)))


def hilo_sobel_select(shape: Shape, img, channels: int, patch: int, mask, radius: int, threshold: float, keep,
                      ws, ws_bytes: int, stream=None) -> None:
    s = shape.c()
    _check("hilo_sobel_select", lib().hilo_sobel_select(ctypes.byref(s), _ptr(img), channels, patch, _ptr(mask),
                                                        radius, ctypes.c_float(threshold), _ptr(keep), _ptr(ws),
                                                        ws_bytes, _stream(stream)))


def hilo_pack(shape: Shape, x, split: SplitBuffers, packed, cap: int, stream=None) -> None:
    s = shape.c()
    o = split.c()
    _check("hilo_pack", lib().hilo_pack(ctypes.byref(s), _ptr(x), ctypes.byref(o), _ptr(packed), cap,
                                        _stream(stream)))


def hilo_block_workspace_bytes(shape: Shape, cap: int) -> int:
    s = shape.c()
    return lib().hilo_block_workspace_bytes(ctypes.byref(s), cap)


def hilo_block_forward(shape: Shape, weights: DeviceWeights, cu_img, cap: int, in_txt, in_img, in_dtype: int,
                       out, ws, ws_bytes: int, stream=None) -> None:
    s = shape.c()
    w = weights.c()
    _check("hilo_block_forward", lib().hilo_block_forward(
        ctypes.byref(s), ctypes.byref(w), _ptr(cu_img), cap, _ptr(in_txt), _ptr(in_img), in_dtype, _ptr(out),
        _ptr(ws), ws_bytes, _stream(stream)))


def hilo_block_forward_prop(shape: Shape, weights: DeviceWeights, cu_img, cap: int, in_txt, in_img, in_dtype: int,
                            n_img, out, ws, ws_bytes: int, stream=None) -> None:
    s = shape.c()
    w = weights.c()
    _check("hilo_block_forward_prop", lib().hilo_block_forward_prop(
        ctypes.byref(s), ctypes.byref(w), _ptr(cu_img), cap, _ptr(in_txt), _ptr(in_img), in_dtype, _ptr(n_img),
        _ptr(out), _ptr(ws), ws_bytes, _stream(stream)))


def hilo_quantize_rows_e4m3(src, src_dtype: int, rows: int, cols: int, dst, scale, stream=None) -> None:
    _check("hilo_quantize_rows_e4m3", lib().hilo_quantize_rows_e4m3(_ptr(src), src_dtype, rows, cols, _ptr(dst),
                                                                    _ptr(scale), _stream(stream)))


def hilo_block_fp8_workspace_bytes(shape: Shape, cap: int) -> int:
    s = shape.c()
    return int(lib().hilo_block_fp8_workspace_bytes(ctypes.byref(s), cap))


def hilo_block_forward_fp8(shape: Shape, weights: DeviceWeightsFP8, cu_img, cap: int, in_txt, in_img,
                           in_dtype: int, out, ws, ws_bytes: int, stream=None) -> None:
    s = shape.c()
    w = weights.c()
    _check("hilo_block_forward_fp8", lib().hilo_block_forward_fp8(
        ctypes.byref(s), ctypes.byref(w), _ptr(cu_img), cap, _ptr(in_txt), _ptr(in_img), in_dtype, _ptr(out),
        _ptr(ws), ws_bytes, _stream(stream)))


def hilo_block_forward_fp8_prop(shape: Shape, weights: DeviceWeightsFP8, cu_img, cap: int, in_txt, in_img,
                                in_dtype: int, n_img, out, ws, ws_bytes: int, stream=None) -> None:
    s = shape.c()
    w = weights.c()
    _check("hilo_block_forward_fp8_prop", lib().hilo_block_forward_fp8_prop(
        ctypes.byref(s), ctypes.byref(w), _ptr(cu_img), cap, _ptr(in_txt), _ptr(in_img), in_dtype, _ptr(n_img),
        _ptr(out), _ptr(ws), ws_bytes, _stream(stream)))


def hilo_row_sizes(shape: Shape, split: SplitBuffers, n_img, cap: int, stream=None) -> None:
    s = shape.c()
    o = split.c()
    _check("hilo_row_sizes", lib().hilo_row_sizes(ctypes.byref(s), ctypes.byref(o), _ptr(n_img), cap,
                                                  _stream(stream)))


def hilo_block_forward_static_ws(shape: Shape, weights: DeviceWeights, cu_img, cap: int, in_txt, in_img,
                                 in_dtype: int, out, stream=None) -> None:
    """hilo_block_forward with the library's built-in scratch (no workspace argument)."""
    s = shape.c()
    w = weights.c()
    _check("hilo_block_forward_static_ws", lib().hilo_block_forward_static_ws(
        ctypes.byref(s), ctypes.byref(w), _ptr(cu_img), cap, _ptr(in_txt), _ptr(in_img), in_dtype, _ptr(out),
        _stream(stream)))


def hilo_unpack(shape: Shape, out_img, split: SplitBuffers, y, stream=None) -> None:
    s = shape.c()
    o = split.c()
    _check("hilo_unpack", lib().hilo_unpack(ctypes.byref(s), _ptr(out_img), ctypes.byref(o), _ptr(y),
                                            _stream(stream)))


def hilo_unpack_delta(shape: Shape, out_img, packed, x, split: SplitBuffers, y, stream=None) -> None:
    s = shape.c()
    o = split.c()
    _check("hilo_unpack_delta", lib().hilo_unpack_delta(ctypes.byref(s), _ptr(out_img), _ptr(packed), _ptr(x),
                                                        ctypes.byref(o), _ptr(y), _stream(stream)))


def hilo_unpack_update(shape: Shape, out_img, split: SplitBuffers, x, alpha: float, stream=None) -> None:
    s = shape.c()
    o = split.c()
    _check("hilo_unpack_update", lib().hilo_unpack_update(ctypes.byref(s), _ptr(out_img), ctypes.byref(o),
                                                          _ptr(x), ctypes.c_float(alpha), _stream(stream)))


def hilo_convert_bf16_to_f16(src, dst, n: int, stream=None) -> None:
    _check("hilo_convert_bf16_to_f16", lib().hilo_convert_bf16_to_f16(_ptr(src), _ptr(dst), n, _stream(stream)))


def hilo_set_stage_events(events) -> None:
    """Register torch.cuda.Event objects (already recorded once) as block stage markers."""
    n = len(events)
    arr = (ctypes.c_void_p * max(n, 1))(*[e.cuda_event for e in events])
    _check("hilo_set_stage_events", lib().hilo_set_stage_events(arr, n))


def hilo_launch_count() -> int:
    return int(lib().hilo_launch_count())


# ---------------------------------------------------------------------------
# One pass of the hot path with every buffer resident on the device
# ---------------------------------------------------------------------------


class HotPath:
    """Device buffers and the five C calls of one hot-path pass.

    score -> split -> pack -> n_layers x block_forward -> unpack. All buffers
    are sized to the upper bound cap = B*H*W image rows, so no call needs the
    data-dependent row counts on the host.
    """

    def __init__(self, shape: Shape, weights: list, device="cuda"):
        self.shape = shape
        self.cap = hilo_row_capacity(shape)
        self.weights = weights
        B, N, d, T = shape.B, shape.N, shape.d, shape.T
        self.score = torch.empty(B * N, dtype=torch.float32, device=device)
        self.split = SplitBuffers.alloc(shape, device)
        self.packed = torch.empty(self.cap, d, dtype=torch.bfloat16, device=device)
        self.out = torch.empty(B * T + self.cap, d, dtype=torch.float32, device=device)
        self.y = torch.empty(B, shape.H, shape.W, d, dtype=torch.float32, device=device)
        self.n_img = torch.empty(self.cap, dtype=torch.float32, device=device)
        self.ws_bytes = hilo_block_workspace_bytes(shape, self.cap)
        self.ws = torch.empty(self.ws_bytes, dtype=torch.uint8, device=device)
        self.weights_fp8 = None

    def enable_fp8(self, weights_fp8: list) -> None:
        """Makes run(..., fp8=True) available: one DeviceWeightsFP8 per block
        and the FP8 workspace (which the bf16 blocks' workspace is grown to)."""
        self.weights_fp8 = weights_fp8
        need = hilo_block_fp8_workspace_bytes(self.shape, self.cap)
        if need > self.ws_bytes:
            self.ws_bytes = need
            self.ws = torch.empty(need, dtype=torch.uint8, device=self.ws.device)

    @property
    def out_img(self) -> torch.Tensor:
        return self.out[self.shape.B * self.shape.T:]

    def run(self, x, text, mask, k_keep, k_mid, stream=None, unpack: bool = True, regions: bool = False,
            prop: bool = False, fp8: bool = False) -> None:
        """One pass. regions=True takes the window-granular split and the
        delta unpool instead of the token-granular split and the nearest
        unpool; prop=True weights each packed row's attention by its row size
        (proportional attention). A shape with lf > 0 runs the separate
        low-frequency token set (with the delta unpool). fp8=True runs the
        blocks with e4m3 GEMM operands (enable_fp8 first)."""
        sh = self.shape
        hilo_score(sh, x, self.score, stream)
        (hilo_split_regions if regions else hilo_split)(sh, self.score, mask, k_keep, k_mid, self.split, None, 0,
                                                        stream)
        hilo_pack(sh, x, self.split, self.packed, self.cap, stream)
        if prop:
            hilo_row_sizes(sh, self.split, self.n_img, self.cap, stream)
        if fp8:
            self.blocks_fp8(text, self.packed, HILO_BF16, stream, self.n_img if prop else None)
        else:
            self.blocks(text, self.packed, HILO_BF16, stream, self.n_img if prop else None)
        if unpack:
            # pooled or low-frequency tokens keep their own detail in the
            # window-granular and low-frequency modes (delta unpool)
            if regions or sh.lf:
                hilo_unpack_delta(sh, self.out_img, self.packed, x, self.split, self.y, stream)
            else:
                hilo_unpack(sh, self.out_img, self.split, self.y, stream)

    def blocks_fp8(self, in_txt, in_img, in_dtype, stream=None, n_img=None) -> None:
        sh = self.shape
        for i, w in enumerate(self.weights_fp8):
            args = (in_txt, in_img, in_dtype) if i == 0 else (self.out, self.out_img, HILO_F32)
            if n_img is None:
                hilo_block_forward_fp8(sh, w, self.split.cu_img, self.cap, *args, self.out, self.ws, self.ws_bytes,
                                       stream)
            else:
                hilo_block_forward_fp8_prop(sh, w, self.split.cu_img, self.cap, *args, n_img, self.out, self.ws,
                                            self.ws_bytes, stream)

    def blocks(self, in_txt, in_img, in_dtype, stream=None, n_img=None) -> None:
        sh = self.shape
        for i, w in enumerate(self.weights):
            args = (in_txt, in_img, in_dtype) if i == 0 else (self.out, self.out_img, HILO_F32)
            if n_img is None:
                hilo_block_forward(sh, w, self.split.cu_img, self.cap, *args, self.out, self.ws, self.ws_bytes,
                                   stream)
            else:
                hilo_block_forward_prop(sh, w, self.split.cu_img, self.cap, *args, n_img, self.out, self.ws,
                                        self.ws_bytes, stream)


# ---------------------------------------------------------------------------
# A stream of host-resident batches through the hot path
# ---------------------------------------------------------------------------


class PipelinedHotPath:
    """Runs the hot path over a sequence of host-resident batches with the
    host->device copy of batch i+1 and the device->host copy of result i-1
    overlapped with the kernels of batch i.

    Two sets of device input buffers and two device results are used in turn.
    Transfers run on their own streams: `h2d` for the inputs, `d2h` for the
    results. Events order them against the compute stream, so that a buffer
    is rewritten only after its last reader is done. This class only orders
    copies and calls; every step of the path runs in libhilo's kernels, as
    in `HotPath.run`.
    """

    def __init__(self, shape: Shape, weights: list, host_inputs, device="cuda"):
        self.hp = HotPath(shape, weights, device)
        self.h2d = torch.cuda.Stream(device=device)
        self.d2h = torch.cuda.Stream(device=device)
        self.dev_in = [tuple(torch.empty_like(t, device=device) for t in host_inputs) for _ in range(2)]
        self.dev_y = [torch.empty_like(self.hp.y) for _ in range(2)]
        self.in_ready = [torch.cuda.Event() for _ in range(2)]
        self.in_free = [torch.cuda.Event() for _ in range(2)]
        self.y_ready = [torch.cuda.Event() for _ in range(2)]
        self.y_free = [torch.cuda.Event() for _ in range(2)]
        self.i = 0

    def submit(self, host_inputs, host_y, compute=None) -> None:
        """Queue one batch: host_inputs = (x, text, mask, k_keep, k_mid) in
        pinned host memory; host_y receives y (pinned, B x H x W x d fp32)."""
        compute = compute or torch.cuda.current_stream()
        b = self.i & 1
        with torch.cuda.stream(self.h2d):
            if self.i >= 2:
                self.h2d.wait_event(self.in_free[b])
            for d, h in zip(self.dev_in[b], host_inputs):
                d.copy_(h, non_blocking=True)
            self.in_ready[b].record(self.h2d)
        compute.wait_event(self.in_ready[b])
        if self.i >= 2:
            compute.wait_event(self.y_free[b])
        hp, sh = self.hp, self.hp.shape
        x, text, mask, k_keep, k_mid = self.dev_in[b]
        hilo_score(sh, x, hp.score, compute)
        hilo_split(sh, hp.score, mask, k_keep, k_mid, hp.split, None, 0, compute)
        hilo_pack(sh, x, hp.split, hp.packed, hp.cap, compute)
        hp.blocks(text, hp.packed, HILO_BF16, compute)
        self.in_free[b].record(compute)
        hilo_unpack(sh, hp.out_img, hp.split, self.dev_y[b], compute)
        self.y_ready[b].record(compute)
        with torch.cuda.stream(self.d2h):
            self.d2h.wait_event(self.y_ready[b])
            host_y.copy_(self.dev_y[b], non_blocking=True)
            self.y_free[b].record(self.d2h)
        self.i += 1

    def drain(self, compute=None) -> None:
        """Make `compute` wait for every queued transfer."""
        compute = compute or torch.cuda.current_stream()
        compute.wait_stream(self.h2d)
        compute.wait_stream(self.d2h)
