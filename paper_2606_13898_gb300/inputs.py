"""Seeded synthetic inputs for the HiLo-Token hot path.

This module only draws random numbers and rounds them to bf16; it holds none
of the method's arithmetic (no score, split, pooling or block math), so the
CUDA path and the oracle can both consume its arrays without sharing method
code.

The paper's workloads are private editing data (407,630 training pairs,
Sec. 3.1; 92 user cases, Sec. 3.3) and cannot be reproduced. The generators
below stand in for them:

* latent token grid: a smooth field, the sum of four random 2-D sinusoids with
  wavelength 8..32 tokens, per channel amplitude N(0, 0.5^2) and phase U[0,2pi);
* edit mask: an axis-aligned rectangle (or the union of three axis-aligned
  ellipses) whose area fraction lies in the workload's range; mask shapes are
  modelled on the paper's mask statistics (Sec. 2.3, "Mask Distribution":
  most masks small, scattered or elongated holes);
* masked tokens are overwritten with N(0,1) noise, text tokens are N(0,1);
* all linear weights and biases are N(0, 0.02^2);
* input image for the paper's Sobel selector (pixel space, P x P pixels per
  token): a smooth field (three sinusoids per channel, wavelengths of 4..16
  tokens) in [0.2, 0.8] with sharp-edged rectangles and discs of random
  colour painted over it, and a small N(0, 0.01^2) noise, fp32 in [0, 1]; the
  edges carry most of the gradient, as object boundaries do in photographs.

Every floating value is drawn in fp32 and rounded to bf16 (round to nearest
even); arrays of bf16 are carried as numpy ``uint16`` bit patterns. Small
draws (field parameters, masks, keep ratios) use numpy's default_rng; the
bulk normal draws use seeded torch CPU generators (faster).
"""
from __future__ import annotations

import dataclasses
import math
from fractions import Fraction

import numpy as np
import torch

# ---------------------------------------------------------------------------
# bf16 bit helpers (storage format only)
# ---------------------------------------------------------------------------


def f32_to_bf16_bits(a) -> np.ndarray:
    """Round fp32 values to bf16 (nearest even) and return the uint16 patterns."""
    t = a if isinstance(a, torch.Tensor) else torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))
    return t.to(torch.float32).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Widen uint16 bf16 patterns to fp32 (exact)."""
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def ceil_ratio(r, n: int) -> int:
    """ceil(r * n) in exact rational arithmetic (r given as a float or str)."""
    f = Fraction(r) if not isinstance(r, str) else Fraction(r)
    v = f * n
    return int(-((-v.numerator) // v.denominator))


# ---------------------------------------------------------------------------
# Workload descriptions
# ---------------------------------------------------------------------------


@dataclasses.dataclass(frozen=True)
class Workload:
    """Shape and selection parameters of one synthetic workload."""

    name: str
    B: int
    H: int
    W: int
    d: int
    T: int
    heads: int
    mlp: bool            # False: attention-only layer (no MLP)
    levels: int          # 1: 2x2 pooling only; 2: 2x2 and 4x4 pooling
    mask_lo: float
    mask_hi: float
    keep_ratio: object   # float / str ratio, or None (drawn per image), or int k
    k_mid_ratio: object = None
    mask_shape: str = "rect"   # "rect" or "rect_or_ellipses"
    seed_base: int = 0
    ratio_lo: float = 0.1
    ratio_hi: float = 0.5

    @property
    def N(self) -> int:
        return self.H * self.W

    @property
    def head_dim(self) -> int:
        return self.d // self.heads


def tiny_layer(**kw) -> Workload:
    """32x32 grid + 64 text tokens, d=512, 8 heads of 64, attention only, seed 0."""
    base = dict(name="tiny_layer_32x32_d512", B=1, H=32, W=32, d=512, T=64, heads=8,
                mlp=False, levels=1, mask_lo=0.10, mask_hi=0.25, keep_ratio="1/4",
                seed_base=0)
    base.update(kw)
    return Workload(**base)


def block_64(keep_ratio="1/4", **kw) -> Workload:
    """One MMDiT block: 64x64 grid (4096 image tokens) + 512 text, d=3072, 24x128 heads."""
    base = dict(name=f"block_64x64_d3072_r{keep_ratio}", B=1, H=64, W=64, d=3072, T=512,
                heads=24, mlp=True, levels=1, mask_lo=0.10, mask_hi=0.40,
                keep_ratio=keep_ratio, seed_base=1000)
    base.update(kw)
    return Workload(**base)


def block_64_batch4(**kw) -> Workload:
    """The 64x64 block at batch 4 with per-image keep ratio U[0.1,0.5] and mask shape."""
    base = dict(name="block_64x64_d3072_b4_varlen", B=4, H=64, W=64, d=3072, T=512,
                heads=24, mlp=True, levels=1, mask_lo=0.10, mask_hi=0.40,
                keep_ratio=None, mask_shape="rect_or_ellipses", seed_base=2000)
    base.update(kw)
    return Workload(**base)


def block_128_two_level(**kw) -> Workload:
    """128x128 grid (16384 image tokens) + 512 text, two-level pooling."""
    base = dict(name="block_128x128_d3072_two_level", B=1, H=128, W=128, d=3072, T=512,
                heads=24, mlp=True, levels=2, mask_lo=0.05, mask_hi=0.20,
                keep_ratio="1/4", k_mid_ratio="1/4", seed_base=3000)
    base.update(kw)
    return Workload(**base)


def denoise_loop(**kw) -> Workload:
    """Stack of 8 blocks as block_64 (r=1/4), run for 28 steps."""
    base = dict(name="denoise_8x28_64x64_d3072", B=1, H=64, W=64, d=3072, T=512,
                heads=24, mlp=True, levels=1, mask_lo=0.10, mask_hi=0.40,
                keep_ratio="1/4", seed_base=4000)
    base.update(kw)
    return Workload(**base)


# ---------------------------------------------------------------------------
# Generators
# ---------------------------------------------------------------------------


def _field(rng: np.random.Generator, H: int, W: int, d: int) -> torch.Tensor:
    """Sum of 4 random 2-D sinusoids per channel, wavelength U[8,32] tokens (fp32)."""
    p = torch.arange(H, dtype=torch.float64)[:, None]
    q = torch.arange(W, dtype=torch.float64)[None, :]
    out = torch.zeros((H, W, d), dtype=torch.float64)
    for _ in range(4):
        lam = rng.uniform(8.0, 32.0)
        theta = rng.uniform(0.0, math.pi)
        amp = torch.from_numpy(rng.normal(0.0, 0.5, size=d))
        phase = torch.from_numpy(rng.uniform(0.0, 2.0 * math.pi, size=d))
        arg = 2.0 * math.pi * (p * math.cos(theta) + q * math.sin(theta)) / lam   # [H,W]
        out += amp[None, None, :] * torch.sin(arg[:, :, None] + phase[None, None, :])
    return out.to(torch.float32)


def _normal(seed: int, shape, std: float = 1.0) -> torch.Tensor:
    """Seeded N(0, std^2) fp32 draws (torch CPU generator)."""
    g = torch.Generator().manual_seed(int(seed))
    t = torch.randn(shape, generator=g, dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    return t


def _rect_mask(rng: np.random.Generator, H: int, W: int, lo: float, hi: float) -> np.ndarray:
    N = H * W
    for _ in range(100000):
        h = int(rng.integers(1, H + 1))
        w = int(rng.integers(1, W + 1))
        if lo <= h * w / N <= hi:
            break
    else:  # pragma: no cover - the ranges used are always reachable
        raise RuntimeError("rectangle mask rejection sampling failed")
    top = int(rng.integers(0, H - h + 1))
    left = int(rng.integers(0, W - w + 1))
    m = np.zeros((H, W), dtype=np.uint8)
    m[top:top + h, left:left + w] = 1
    return m


def _ellipse_mask(rng: np.random.Generator, H: int, W: int, lo: float, hi: float) -> np.ndarray:
    pc = np.arange(H, dtype=np.float64)[:, None] + 0.5
    qc = np.arange(W, dtype=np.float64)[None, :] + 0.5
    for _ in range(100000):
        m = np.zeros((H, W), dtype=bool)
        for _e in range(3):
            cp, cq = rng.uniform(0, H), rng.uniform(0, W)
            ap, aq = rng.uniform(0.1, 0.3) * H, rng.uniform(0.1, 0.3) * W
            m |= ((pc - cp) / ap) ** 2 + ((qc - cq) / aq) ** 2 <= 1.0
        if lo <= m.mean() <= hi:
            return m.astype(np.uint8)
    raise RuntimeError("ellipse mask rejection sampling failed")  # pragma: no cover


def make_image(B: int, H: int, W: int, patch: int = 16, channels: int = 3, seed: int = 0,
               n_shapes: int = 16) -> np.ndarray:
    """Synthetic image [B, H*patch, W*patch, channels] fp32 (see the module
    header). Image b uses numpy default_rng(seed + b)."""
    Hp, Wp = H * patch, W * patch
    y = np.arange(Hp, dtype=np.float32)[:, None]
    x = np.arange(Wp, dtype=np.float32)[None, :]
    out = np.empty((B, Hp, Wp, channels), dtype=np.float32)
    for b in range(B):
        rng = np.random.default_rng(seed + b)
        img = np.zeros((Hp, Wp, channels), dtype=np.float32)
        for c in range(channels):
            f = np.zeros((Hp, Wp), dtype=np.float32)
            for _ in range(3):
                lam = np.float32(rng.uniform(4.0, 16.0) * patch)
                th = rng.uniform(0.0, math.pi)
                ph = rng.uniform(0.0, 2.0 * math.pi)
                f += np.sin(2.0 * np.pi * (x * np.float32(math.cos(th)) + y * np.float32(math.sin(th))) / lam
                            + np.float32(ph)).astype(np.float32)
            img[:, :, c] = 0.5 + 0.1 * f
        for _ in range(n_shapes):
            col = rng.uniform(0.0, 1.0, size=channels).astype(np.float32)
            if rng.random() < 0.5:
                h, w = int(rng.integers(Hp // 16, Hp // 4 + 1)), int(rng.integers(Wp // 16, Wp // 4 + 1))
                t0, l0 = int(rng.integers(0, Hp - h + 1)), int(rng.integers(0, Wp - w + 1))
                img[t0:t0 + h, l0:l0 + w] = col
            else:
                r = rng.uniform(Hp / 32, Hp / 8)
                cy, cx = rng.uniform(0, Hp), rng.uniform(0, Wp)
                img[(y - cy) ** 2 + (x - cx) ** 2 <= r * r] = col
        img += rng.normal(0.0, 0.01, size=img.shape).astype(np.float32)
        out[b] = np.clip(img, 0.0, 1.0)
    return out


@dataclasses.dataclass
class Batch:
    """One batch of synthetic inputs (bf16 as uint16 bit patterns)."""

    wl: Workload
    x: np.ndarray        # uint16 [B,H,W,d]
    text: np.ndarray     # uint16 [B,T,d]
    mask: np.ndarray     # uint8  [B,H*W]
    k_keep: np.ndarray   # int32  [B]
    k_mid: np.ndarray    # int32  [B]  (zeros when levels == 1)


def make_batch(wl: Workload, seed_offset: int = 0) -> Batch:
    """Latents, masks, text and integer keep counts for workload ``wl``.

    Image b of the workload uses ``numpy.random.default_rng(seed_base + b)``.
    """
    B, H, W, d, T, N = wl.B, wl.H, wl.W, wl.d, wl.T, wl.N
    xs = np.empty((B, H, W, d), dtype=np.uint16)
    ts = np.empty((B, T, d), dtype=np.uint16)
    ms = np.empty((B, N), dtype=np.uint8)
    kk = np.zeros(B, dtype=np.int32)
    km = np.zeros(B, dtype=np.int32)
    for b in range(B):
        rng = np.random.default_rng(wl.seed_base + seed_offset + b)
        f = _field(rng, H, W, d)
        if wl.mask_shape == "rect_or_ellipses" and rng.integers(0, 2) == 1:
            m = _ellipse_mask(rng, H, W, wl.mask_lo, wl.mask_hi)
        else:
            m = _rect_mask(rng, H, W, wl.mask_lo, wl.mask_hi)
        noise_seed, text_seed = (int(v) for v in rng.integers(0, 2 ** 62, size=2))
        noise = _normal(noise_seed, (H, W, d))
        f = torch.where(torch.from_numpy(m)[:, :, None] == 1, noise, f)
        xs[b] = f32_to_bf16_bits(f)
        ts[b] = f32_to_bf16_bits(_normal(text_seed, (T, d)))
        ms[b] = m.reshape(N)
        if wl.keep_ratio is None:
            r = rng.uniform(wl.ratio_lo, wl.ratio_hi)
            kk[b] = ceil_ratio(r, N)
        elif isinstance(wl.keep_ratio, int):
            kk[b] = wl.keep_ratio
        else:
            kk[b] = ceil_ratio(wl.keep_ratio, N)
        if wl.levels == 2:
            km[b] = ceil_ratio(wl.k_mid_ratio, N)
    return Batch(wl, xs, ts, ms, kk, km)


@dataclasses.dataclass
class StreamWeights:
    """Linear weights of one stream (text or image), PyTorch layout [out, in]."""

    w_qkv: np.ndarray  # uint16 [3d, d]
    b_qkv: np.ndarray  # uint16 [3d]
    w_o: np.ndarray    # uint16 [d, d]
    b_o: np.ndarray    # uint16 [d]
    w_1: np.ndarray | None = None   # uint16 [4d, d]
    b_1: np.ndarray | None = None   # uint16 [4d]
    w_2: np.ndarray | None = None   # uint16 [d, 4d]
    b_2: np.ndarray | None = None   # uint16 [d]


@dataclasses.dataclass
class BlockWeights:
    txt: StreamWeights
    img: StreamWeights


def make_weights(d: int, mlp: bool, seed: int, mlp_ratio: int = 4) -> BlockWeights:
    """N(0, 0.02^2) weights and biases for both streams of one block."""
    counter = [0]

    def draw(shape) -> np.ndarray:
        counter[0] += 1
        return f32_to_bf16_bits(_normal(seed * 1000 + counter[0], shape, 0.02))

    def stream() -> StreamWeights:
        s = StreamWeights(w_qkv=draw((3 * d, d)), b_qkv=draw((3 * d,)), w_o=draw((d, d)), b_o=draw((d,)))
        if mlp:
            s.w_1 = draw((mlp_ratio * d, d))
            s.b_1 = draw((mlp_ratio * d,))
            s.w_2 = draw((d, mlp_ratio * d))
            s.b_2 = draw((d,))
        return s

    return BlockWeights(txt=stream(), img=stream())


def weight_seed(wl: Workload, layer: int = 0) -> int:
    """Seed of the weights of layer ``layer`` of workload ``wl``."""
    return wl.seed_base + 500 + layer
