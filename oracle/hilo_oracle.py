"""CPU oracle for the HiLo-Token hot path -- TEST INFRASTRUCTURE ONLY.

Only the tests, the smoke check and the benchmark's CPU-baseline leg may
import this module. The product path never calls it: it shares no code with
the CUDA library (no kernels, headers, helpers, constants or tables) and
imports nothing from the package.

What it computes, step by step (paper: Sec. 2.3 "HiLo-Token Selection" and
the DiT it feeds; the concrete variant -- token-space score, top-k split,
2x2/4x4 pooling, MMDiT block -- is the one the hot path implements):

  score   per-token high-frequency energy  s_i = sum_c (x_ic - m_w(i),c)^2,
          m_w the mean of the aligned 2x2 window holding token i
          (the token-space stand-in for the Sobel frequency map + 16x
          regionalisation of Sec. 2.3).
  split   keep = top-k tokens by (score desc, index asc) united with the edit
          mask (Sec. 2.3: tokens inside the mask are always retained); the
          rest is pooled 2x2, or for two-level pooling the next k_mid tokens
          are pooled 2x2 and the remainder 4x4.
  pack    the packed image sequence per image: kept tokens in raster order,
          then one row per 2x2 window (mean of that window's 2x2-pooled
          members), then one row per 4x4 window (Sec. 2.3: selected tokens
          concatenated with the low-frequency tokens along the token axis).
  block   an MMDiT-style block on the joint [text ; packed image] sequence:
          pre-LayerNorm (no affine), two-stream QKV / out / MLP weights, joint
          softmax attention, tanh-GELU 4x MLP, residual adds.
  unpack  every grid token reads the output row of its kept token or of its
          window (nearest broadcast).
  split(lf=f), pack(lf=f)  the separate low-frequency token set (Sec. 2.3:
          the kept tokens are concatenated with all tokens of a downsampled
          image, here the grid average-pooled f-fold per side, without the
          VAE); the other tokens read their window's row back (delta unpool).
  e4m3_encode, quantize_rows, block_fp8  FP8 GEMM operands (Sec. 3.3 reports
          FP8 on top of HiLo-Token without a scheme): per-row e4m3 scaling
          of activations and weights, fp32 accumulation, the activations
          rounded where the kernels round them.
  row_sizes, block(n_img=...)  proportional attention for pooled tokens:
          a packed row standing for n grid tokens adds ln(n) to its logits as
          a key, i.e. it draws the attention of n identical copies (the
          paper is silent on how pooled tokens attend; this is the reading
          that keeps the attention mass of the uncompressed sequence).
  split(granular=True), unpack_delta  the window-granular (regionalised)
          split -- each pooling window takes the finest class of any member,
          so kept regions are whole 2x2 windows and every pooled window is
          full -- and the delta unpool, where a pooled member keeps its own
          value plus its window's update (Sec. 2.3's coherent, region-level
          selection read in token space).
  update  x <- bf16(x - alpha * y) for the denoising loop.
  sobel_select  the paper's own selector (Sec. 2.3): a Sobel frequency map
          of the input image, normalised by its maximum, thresholded, pooled
          onto the token grid (a token of P x P pixels is selected when any
          of its pixels exceeds the threshold), united with the user mask
          dilated by R tokens. It yields the keep map used with k_keep = 0.

Precision. Where a float decides an integer or a stored bf16 code (the score
decides the split; the pooled mean is stored as bf16; the loop update is
stored as bf16) the oracle computes in fp32 with one fixed order of
operations and no fused multiply-add, the precision the kernels use. The
block is computed in fp64 from the exact bf16 inputs and weights.

Fixed orders (readings where the paper is silent):
  * window mean for the score: ((x_a + x_b) + (x_c + x_d)) * 0.25 with
    members a,b,c,d in raster order;
  * channel sum: channels are taken in groups of 8 consecutive channels;
    group g is folded into partial sum p[g mod 128] (groups ascending, the 8
    channels of a group ascending); the 128 partials are then combined by the
    halving tree p[j] += p[j + h] for h = 64, 32, 16, 8, 4, 2, 1;
  * pooled mean: fp32 sum of the class members in raster order starting from
    the first member, one correctly rounded division by the member count,
    then bf16 round-to-nearest-even.

  * Sobel map (readings: the paper names the operator, not the border rule,
    the channel combination or the norm): replicate borders; per channel
    gx = ((P(y-1,x+1) + 2P(y,x+1)) + P(y+1,x+1)) - ((P(y-1,x-1) + 2P(y,x-1))
    + P(y+1,x-1)) and gy likewise with rows; g = sqrt(sum over channels in
    ascending order of (gx*gx + gy*gy)), fp32, correctly rounded sqrt; the
    map is normalised by its per-image maximum with one fp32 division per
    token maximum, and the comparison with the threshold is strict.

Bit patterns of bf16 arrays are carried as numpy uint16.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

KEEP = 0
POOL2 = 1
POOL4 = 2
LF = 3

# ---------------------------------------------------------------------------
# bf16 conversion (own implementation; pinned against torch in the tests)
# ---------------------------------------------------------------------------


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to fp32. Numeric helper (bf16 storage of activations and weights); no
    paper passage."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def f32_to_bf16(a: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit pattern, round to nearest, ties to even (finite inputs). Numeric helper; no paper passage."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    keep_lsb = (u >> np.uint64(16)) & np.uint64(1)
    rounded = (u + np.uint64(0x7FFF) + keep_lsb) >> np.uint64(16)
    return rounded.astype(np.uint16)


# ---------------------------------------------------------------------------
# Step 1: frequency score (fp32, fixed order)
# ---------------------------------------------------------------------------


def score(x_bits: np.ndarray) -> np.ndarray:
    """Per-token energy of x minus its 2x2 average-pooled-then-upsampled value.

    x_bits: uint16 [B,H,W,d] (bf16); H, W even; d a multiple of 8.
    Returns fp32 [B, H*W].

    Paper: Sec. 2.3, HiLo-Token Selection (the frequency map, token-space form).
    """
    B, H, W, d = x_bits.shape
    assert H % 2 == 0 and W % 2 == 0 and d % 8 == 0
    x = bf16_to_f32(x_bits)
    a = x[:, 0::2, 0::2, :]
    b = x[:, 0::2, 1::2, :]
    c = x[:, 1::2, 0::2, :]
    e = x[:, 1::2, 1::2, :]
    m = ((a + b) + (c + e)) * np.float32(0.25)                 # [B,H/2,W/2,d]
    up = np.repeat(np.repeat(m, 2, axis=1), 2, axis=2)          # nearest upsample
    diff = x - up
    sq = diff * diff                                            # fp32, no FMA
    sq = sq.reshape(B, H * W, d)
    partial = np.zeros((B, H * W, 128), dtype=np.float32)
    for g in range(d // 8):
        j = g % 128
        for u in range(8):
            partial[:, :, j] = partial[:, :, j] + sq[:, :, 8 * g + u]
    for h in (64, 32, 16, 8, 4, 2, 1):
        partial[:, :, :h] = partial[:, :, :h] + partial[:, :, h:2 * h]
    return np.ascontiguousarray(partial[:, :, 0])


def score_f64(x_bits: np.ndarray) -> np.ndarray:
    """The same energy in fp64, summed plainly (a sanity reference). Paper: Sec. 2.3, as score."""
    B, H, W, d = x_bits.shape
    x = bf16_to_f32(x_bits).astype(np.float64)
    m = x.reshape(B, H // 2, 2, W // 2, 2, d).mean(axis=(2, 4))
    up = np.repeat(np.repeat(m, 2, axis=1), 2, axis=2)
    return ((x - up) ** 2).sum(axis=-1).reshape(B, H * W)


# ---------------------------------------------------------------------------
# Step 2: keep / pool split
# ---------------------------------------------------------------------------


@dataclasses.dataclass
class Split:
    labels: np.ndarray    # uint8 [B,N]   KEEP / POOL2 / POOL4
    row_src: np.ndarray   # int32 [rows]  token id (kept rows) or window id (pooled rows)
    counts: np.ndarray    # int32 [B,3]   kept tokens, 2x2 windows, 4x4 windows
    cu_img: np.ndarray    # int32 [B+1]   packed image-row offsets
    tok_row: np.ndarray   # int32 [B,N]   packed row each grid token reads back


def ranking(s: np.ndarray) -> np.ndarray:
    """Token ids ordered by (score descending, token index ascending). Paper: Sec. 2.3, HiLo-Token Selection
    (high-frequency tokens are selected)."""
    idx = np.arange(s.shape[0])
    return np.lexsort((idx, -s.astype(np.float64)))


def split(s: np.ndarray, mask: np.ndarray, k_keep, k_mid, H: int, W: int, levels: int,
          granular: bool = False, lf: int = 0) -> Split:
    """Deterministic keep/pool split of each image (see module docstring).

    granular=True is the window-granular (regionalised) variant, the token-
    space reading of the coherent region-level selection of Sec. 2.3: every
    pooling window takes the finest class any of its members has. An aligned
    2x2 window with a member in top-k_keep or the mask is kept whole; with two
    levels, an aligned 4x4 block is pooled 4x4 only when all 16 of its members
    rank below the k_mid cut, otherwise its (whole, non-kept) 2x2 windows are
    pooled 2x2. Every pooled window is then full.

    lf > 0 is the separate low-frequency token set of Sec. 2.3 in token
    space: the kept tokens (top-k_keep united with the mask) are followed by
    one row per aligned lf x lf window of the whole grid (every window, kept
    members included: the grid downsampled lf-fold per side); the other
    tokens are labelled LF and read their output from their window's row.
    counts = (kept, windows, 0); levels must be 1."""
    if lf:
        return _split_lf(s, mask, k_keep, H, W, lf)
    B, N = s.shape
    assert N == H * W and levels in (1, 2)
    labels = np.empty((B, N), dtype=np.uint8)
    counts = np.zeros((B, 3), dtype=np.int32)
    cu = np.zeros(B + 1, dtype=np.int32)
    tok_row = np.empty((B, N), dtype=np.int32)
    rows = []
    p = np.arange(N) // W
    q = np.arange(N) % W
    win2_of = (p // 2) * (W // 2) + (q // 2)
    win4_of = (p // 4) * (W // 4) + (q // 4) if levels == 2 else None
    for b in range(B):
        order = ranking(s[b])
        keep = mask[b].astype(bool).copy()
        keep[order[:int(k_keep[b])]] = True
        if granular:
            keep = np.isin(win2_of, win2_of[keep])
        lab = np.full(N, POOL2, dtype=np.uint8)
        lab[keep] = KEEP
        if levels == 2:
            rest = order[~keep[order]]
            lab[rest[int(k_mid[b]):]] = POOL4
            if granular:
                whole4 = np.ones((H // 4) * (W // 4), dtype=bool)
                np.logical_and.at(whole4, win4_of, lab == POOL4)
                lab[(lab == POOL4) & ~whole4[win4_of]] = POOL2
        labels[b] = lab
        kept = np.nonzero(lab == KEEP)[0]
        w2 = np.unique(win2_of[lab == POOL2])
        w4 = np.unique(win4_of[lab == POOL4]) if levels == 2 else np.zeros(0, dtype=np.int64)
        counts[b] = (len(kept), len(w2), len(w4))
        cu[b + 1] = cu[b] + len(kept) + len(w2) + len(w4)
        rows += [kept, w2, w4]
        base = int(cu[b])
        tok_row[b, kept] = base + np.arange(len(kept))
        r2 = {int(w): base + len(kept) + i for i, w in enumerate(w2)}
        r4 = {int(w): base + len(kept) + len(w2) + i for i, w in enumerate(w4)}
        for i in np.nonzero(lab == POOL2)[0]:
            tok_row[b, i] = r2[int(win2_of[i])]
        for i in np.nonzero(lab == POOL4)[0]:
            tok_row[b, i] = r4[int(win4_of[i])]
    row_src = np.concatenate([np.asarray(r, dtype=np.int64) for r in rows]).astype(np.int32) \
        if rows else np.zeros(0, np.int32)
    return Split(labels, row_src, counts, cu, tok_row)


# ---------------------------------------------------------------------------
# Step 3: pack (gather + average pooling)
# ---------------------------------------------------------------------------


def _split_lf(s, mask, k_keep, H: int, W: int, lf: int) -> Split:
    B, N = s.shape
    assert H % lf == 0 and W % lf == 0
    nlf = (H // lf) * (W // lf)
    p = np.arange(N) // W
    q = np.arange(N) % W
    win_of = (p // lf) * (W // lf) + (q // lf)
    labels = np.empty((B, N), dtype=np.uint8)
    counts = np.zeros((B, 3), dtype=np.int32)
    cu = np.zeros(B + 1, dtype=np.int32)
    tok_row = np.empty((B, N), dtype=np.int32)
    rows = []
    for b in range(B):
        keep = mask[b].astype(bool).copy()
        keep[ranking(s[b])[:int(k_keep[b])]] = True
        labels[b] = np.where(keep, KEEP, LF)
        kept = np.nonzero(keep)[0]
        counts[b] = (len(kept), nlf, 0)
        cu[b + 1] = cu[b] + len(kept) + nlf
        base = int(cu[b])
        tok_row[b, kept] = base + np.arange(len(kept))
        tok_row[b, ~keep] = base + len(kept) + win_of[~keep]
        rows += [kept, np.arange(nlf)]
    row_src = np.concatenate([np.asarray(r, dtype=np.int64) for r in rows]).astype(np.int32)
    return Split(labels, row_src, counts, cu, tok_row)


def window_members(w: int, size: int, W: int) -> list[int]:
    """Token ids of aligned size x size window ``w`` in raster order. Paper: Sec. 2.3 (the pooled low-frequency
    regions)."""
    wp, wq = divmod(w, W // size)
    return [(size * wp + i) * W + size * wq + j for i in range(size) for j in range(size)]


def pack(x_bits: np.ndarray, sp: Split, lf: int = 0) -> np.ndarray:
    """Packed image rows, uint16 [rows, d] (bf16). With lf > 0 (a split made
    with the same lf) the rows after the kept tokens are the lf x lf window
    means over all members.

    Paper: Sec. 2.3 (selected and low-frequency tokens concatenated along the token axis)."""
    B, H, W, d = x_bits.shape
    x = bf16_to_f32(x_bits).reshape(B, H * W, d)
    out = np.empty((int(sp.cu_img[-1]), d), dtype=np.uint16)
    for b in range(B):
        nk, n2, n4 = (int(c) for c in sp.counts[b])
        base = int(sp.cu_img[b])
        for r in range(nk + n2 + n4):
            src = int(sp.row_src[base + r])
            if r < nk:
                out[base + r] = x_bits.reshape(B, H * W, d)[b, src]
                continue
            if lf:
                members = window_members(src, lf, W)
            else:
                size, cls = (2, POOL2) if r < nk + n2 else (4, POOL4)
                members = [t for t in window_members(src, size, W) if sp.labels[b, t] == cls]
            acc = x[b, members[0]].copy()
            for t in members[1:]:
                acc = acc + x[b, t]
            mean = acc / np.float32(len(members))
            out[base + r] = f32_to_bf16(mean)
    return out


# ---------------------------------------------------------------------------
# Step 4: MMDiT block (fp64)
# ---------------------------------------------------------------------------


def layer_norm(u: np.ndarray, eps: float = 1e-6) -> np.ndarray:
    """LayerNorm over the last axis, no affine, biased variance. Paper: Sec. 2.1 (the DiT block of the editing
    generalist)."""
    mu = u.mean(axis=-1, keepdims=True)
    var = ((u - mu) ** 2).mean(axis=-1, keepdims=True)
    return (u - mu) / np.sqrt(var + eps)


def gelu_tanh(z: np.ndarray) -> np.ndarray:
    """GELU, tanh approximation. Paper: Sec. 2.1 (the DiT block's MLP)."""
    return 0.5 * z * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (z + 0.044715 * z ** 3)))


def softmax_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, key_n=None) -> np.ndarray:
    """Non-causal softmax attention of one head, scale 1/sqrt(head_dim).

    key_n (optional, one positive weight per key) is proportional attention:
    ln(key_n[j]) is added to every logit of key j, so a key standing for n
    tokens receives the attention mass of n identical copies of itself.

    Paper: Sec. 2.1 (the DiT's joint attention); Sec. 2.3 for the compressed keys."""
    sc = (q @ k.T) / math.sqrt(q.shape[-1])
    if key_n is not None:
        # a weight of 0 (a low-frequency row all of whose members are kept)
        # removes the key: ln 0 = -inf
        with np.errstate(divide="ignore"):
            sc = sc + np.log(np.asarray(key_n, dtype=np.float64))[None, :]
    sc = sc - sc.max(axis=-1, keepdims=True)
    p = np.exp(sc)
    p = p / p.sum(axis=-1, keepdims=True)
    return p @ v


def _w(bits) -> np.ndarray:
    """Weights as fp64: bf16 bit patterns are widened, float arrays pass through."""
    if bits.dtype == np.uint16:
        return bf16_to_f32(bits).astype(np.float64)
    return bits


def weights_f64(w):
    """A copy of block weights widened to fp64 once (same values as _w gives
    per call), for callers that run the block many times.

    Helper; no paper passage."""
    import copy
    out = copy.copy(w)
    for sname in ("txt", "img"):
        sw = copy.copy(getattr(w, sname))
        for f in ("w_qkv", "b_qkv", "w_o", "b_o", "w_1", "b_1", "w_2", "b_2"):
            v = getattr(sw, f, None)
            if v is not None:
                setattr(sw, f, _w(v))
        setattr(out, sname, sw)
    return out


def _as_f64(u) -> np.ndarray:
    return bf16_to_f32(u).astype(np.float64) if u.dtype == np.uint16 else np.asarray(u, np.float64)


def block(u_txt, u_img, cu_img, T: int, weights, heads: int, mlp: bool, n_img=None):
    """One MMDiT block on the joint sequence of each image.

    u_txt: [B*T, d] text rows (image b owns rows b*T .. b*T+T-1);
    u_img: [rows, d] packed image rows (image b owns cu_img[b] .. cu_img[b+1]-1).
    Either may be bf16 bits (uint16) or floats. Returns fp64 (txt, img).
    ``weights`` has ``.txt`` and ``.img`` with PyTorch-layout [out, in] arrays.
    n_img (optional): proportional attention, the number of grid tokens each
    packed image row stands for (text keys count 1), see softmax_attention.

    Paper: Sec. 2.1 (the DiT block) on the sequence Sec. 2.3 compresses.
    """
    ut = _as_f64(u_txt)
    ui = _as_f64(u_img)
    d = ut.shape[1] if ut.size else ui.shape[1]
    hd = d // heads
    B = len(cu_img) - 1
    streams = ((ut, weights.txt), (ui, weights.img))
    qkv = [layer_norm(u) @ _w(w.w_qkv).T + _w(w.b_qkv) for u, w in streams]
    att = [np.zeros_like(ut), np.zeros_like(ui)]
    for b in range(B):
        t0, t1 = b * T, (b + 1) * T
        i0, i1 = int(cu_img[b]), int(cu_img[b + 1])
        joint = np.concatenate([qkv[0][t0:t1], qkv[1][i0:i1]], axis=0)
        kn = None if n_img is None else np.concatenate([np.ones(T), np.asarray(n_img[i0:i1], np.float64)])
        o = np.empty((joint.shape[0], d))
        for h in range(heads):
            c = slice(h * hd, (h + 1) * hd)
            o[:, c] = softmax_attention(joint[:, c], joint[:, d:][:, c], joint[:, 2 * d:][:, c], kn)
        att[0][t0:t1] = o[:T]
        att[1][i0:i1] = o[T:]
    out = []
    for (u, w), a in zip(streams, att):
        u = u + a @ _w(w.w_o).T + _w(w.b_o)
        if mlp:
            u = u + gelu_tanh(layer_norm(u) @ _w(w.w_1).T + _w(w.b_1)) @ _w(w.w_2).T + _w(w.b_2)
        out.append(u)
    return out[0], out[1]


def block_rows(u_txt, u_img, cu_img, T: int, weights, heads: int, mlp: bool, b: int,
               txt_rows, img_rows, n_img=None):
    """The block's outputs for selected rows of image ``b`` only.

    Same arithmetic as ``block``; keys and values of the whole joint sequence
    of image b are projected, queries, attention and MLP only for the given
    rows (absolute row ids in u_txt / u_img). Returns fp64 (txt_out, img_out).

    Paper: Sec. 2.1, as block.
    """
    ut = _as_f64(u_txt)
    ui = _as_f64(u_img)
    d = ut.shape[1]
    hd = d // heads
    t0, t1 = b * T, (b + 1) * T
    i0, i1 = int(cu_img[b]), int(cu_img[b + 1])
    wt, wi = weights.txt, weights.img
    ln_t = layer_norm(ut[t0:t1])
    ln_i = layer_norm(ui[i0:i1])
    kv = np.concatenate([ln_t @ _w(wt.w_qkv[d:]).T + _w(wt.b_qkv[d:]),
                         ln_i @ _w(wi.w_qkv[d:]).T + _w(wi.b_qkv[d:])], axis=0)
    kn = None if n_img is None else np.concatenate([np.ones(t1 - t0), np.asarray(n_img[i0:i1], np.float64)])
    res = []
    for rows, u_all, w in ((np.asarray(txt_rows, int), ut, wt), (np.asarray(img_rows, int), ui, wi)):
        if rows.size == 0:
            res.append(np.zeros((0, d)))
            continue
        u = u_all[rows]
        q = layer_norm(u) @ _w(w.w_qkv[:d]).T + _w(w.b_qkv[:d])
        o = np.empty((len(rows), d))
        for h in range(heads):
            c = slice(h * hd, (h + 1) * hd)
            o[:, c] = softmax_attention(q[:, c], kv[:, :d][:, c], kv[:, d:][:, c], kn)
        u = u + o @ _w(w.w_o).T + _w(w.b_o)
        if mlp:
            u = u + gelu_tanh(layer_norm(u) @ _w(w.w_1).T + _w(w.b_1)) @ _w(w.w_2).T + _w(w.b_2)
        res.append(u)
    return res[0], res[1]


def block_dense(x_bits, text_bits, weights, heads: int, mlp: bool):
    """The uncompressed block: every grid token in raster order, no pooling. Paper: Sec. 2.1 (the uncompressed
    DiT the speed-ups of Sec. 3.3 are measured against)."""
    B, H, W, d = x_bits.shape
    cu = np.arange(B + 1, dtype=np.int64) * (H * W)
    return block(text_bits.reshape(B * text_bits.shape[1], d), x_bits.reshape(B * H * W, d),
                 cu, text_bits.shape[1], weights, heads, mlp)


# ---------------------------------------------------------------------------
# Step 5: unpack, and the denoising-loop update
# ---------------------------------------------------------------------------


def row_sizes(sp: Split) -> np.ndarray:
    """Number of grid tokens each packed image row stands for: 1 for a kept
    token, the number of its class members for a pooled window (fp32).

    Paper: Sec. 2.3 is silent on how pooled tokens attend; this supports the proportional reading."""
    n = np.zeros(int(sp.cu_img[-1]), dtype=np.float32)
    for b in range(sp.labels.shape[0]):
        np.add.at(n, sp.tok_row[b], np.float32(1.0))
    return n


def unpack(out_img: np.ndarray, sp: Split) -> np.ndarray:
    """y[b, i] = out_img[tok_row[b, i]]  ->  [B, N, d]. Paper: Sec. 2.3 (the compressed tokens restored to the
    full grid)."""
    return out_img[sp.tok_row]


def unpack_delta(out_img: np.ndarray, packed_bits: np.ndarray, x_bits: np.ndarray, sp: Split) -> np.ndarray:
    """Delta unpool (the additive reading of restoring pooled tokens to the
    grid): a kept token takes its own output row; a pooled member i of window
    row r keeps its own value and receives the window's update,
    y_i = x_i + (out_r - packed_r), two fp32 operations in that order, with
    x_i and packed_r the bf16 values widened to fp32. Returns fp32
    [B, H, W, d]."""
    B, H, W, d = x_bits.shape
    x = bf16_to_f32(x_bits).reshape(B, H * W, d)
    p = bf16_to_f32(packed_bits)
    out = np.asarray(out_img, dtype=np.float32)
    y = np.empty((B, H * W, d), dtype=np.float32)
    for b in range(B):
        for i in range(H * W):
            r = int(sp.tok_row[b, i])
            if sp.labels[b, i] == KEEP:
                y[b, i] = out[r]
            else:
                y[b, i] = x[b, i] + (out[r] - p[r])
    return y.reshape(B, H, W, d)


def update(x_bits: np.ndarray, y: np.ndarray, alpha: float) -> np.ndarray:
    """x <- bf16(x - alpha * y), fp32 multiply then subtract (no FMA). No paper formula: a plain update step of
    the denoising loop (Sec. 2.4 distils an 8-step sampler)."""
    x = bf16_to_f32(x_bits)
    t = np.float32(alpha) * np.asarray(y, dtype=np.float32)
    return f32_to_bf16(x - t)


# ---------------------------------------------------------------------------
# FP8 (e4m3) GEMM operands (Sec. 3.3 reports FP8 on top of HiLo-Token; the
# scheme below is this implementation's: per-row scaling of every GEMM
# operand, fp32 accumulation)
# ---------------------------------------------------------------------------

E4M3_MAX = 448.0


def e4m3_encode(t: np.ndarray) -> np.ndarray:
    """fp32 values -> e4m3 codes (uint8): 1 sign bit, 4 exponent bits (bias
    7), 3 mantissa bits; round to nearest, ties to even; values beyond the
    largest finite magnitude 448 saturate to +-448 (NaN is not expected).

    Worked on the fp32 bit pattern. A magnitude at or above 2^-6 (the
    smallest normal e4m3) keeps 3 of its 23 mantissa bits: add 2^19 - 1 plus
    the lowest kept bit (round half to even) and clear the 20 dropped bits; a
    carry into the exponent is the next binade's value, as it should be.
    Below 2^-6 the values are multiples of the subnormal quantum 2^-9,
    rounded half to even by rint.

    Paper: Sec. 3.3 reports FP8 on top of HiLo-Token; the format is IEEE-style e4m3."""
    t = np.asarray(t, dtype=np.float32)
    sign = ((t.view(np.uint32) >> 24) & 0x80).astype(np.uint8)
    a = np.abs(t)
    bits = a.view(np.uint32)  # sign cleared: adding < 2^20 cannot overflow
    rb = (bits + np.uint32(0x7FFFF) + ((bits >> 20) & np.uint32(1))) & np.uint32(0xFFF00000)
    vn = rb.view(np.float32)
    vs = (np.rint(a * np.float32(2.0 ** 9)) * np.float32(2.0 ** -9)).astype(np.float32)
    normal = a >= np.float32(2.0 ** -6)
    v = np.minimum(np.where(normal, vn, vs), np.float32(E4M3_MAX))
    # fields of the rounded magnitude
    vb = v.view(np.uint32)
    vnorm = v >= np.float32(2.0 ** -6)
    exp_field = np.where(vnorm, ((vb >> 23) & 0xFF).astype(np.int32) - 120, 0)
    mant = np.where(vnorm, (vb >> 20) & 7, (v * np.float32(2.0 ** 9)).astype(np.int32)).astype(np.int32)
    return sign | ((exp_field << 3) | mant).astype(np.uint8)


def e4m3_decode(c: np.ndarray) -> np.ndarray:
    """e4m3 codes -> values (fp64; 0x7f / 0xff are NaN). Paper: Sec. 3.3, as e4m3_encode."""
    c = np.asarray(c, dtype=np.uint8).astype(np.int64)
    s = np.where(c & 0x80, -1.0, 1.0)
    ef = (c >> 3) & 0xF
    mf = c & 0x7
    v = np.where(ef == 0, mf * 2.0 ** -9, (1 + mf / 8.0) * np.ldexp(1.0, ef - 7))
    v = np.where((c & 0x7F) == 0x7F, np.nan, v)
    return s * v


def quantize_rows(x) -> tuple[np.ndarray, np.ndarray]:
    """Per-row e4m3 quantisation of an fp32 matrix [R, C]: amax = max |x| of
    the row, inv = 448 / amax and scale = amax / 448 (each one correctly
    rounded fp32 division; 1 for an all-zero row), code = e4m3(x * inv) with
    the product rounded to fp32 first. Returns (codes uint8 [R, C], scale
    fp32 [R]); code value times scale approximates x.

    Paper: Sec. 3.3 (FP8); the scaling scheme is this implementation's."""
    x = np.asarray(x, dtype=np.float32)
    amax = np.abs(x).max(axis=1) if x.shape[1] else np.zeros(x.shape[0], np.float32)
    pos = amax > 0
    inv = np.where(pos, np.float32(E4M3_MAX) / np.where(pos, amax, 1).astype(np.float32), 1).astype(np.float32)
    scale = np.where(pos, amax.astype(np.float32) / np.float32(E4M3_MAX), 1).astype(np.float32)
    codes = e4m3_encode((x * inv[:, None]).astype(np.float32))
    return codes, scale


def dequant(codes, scale) -> np.ndarray:
    """Paper: Sec. 3.3 (FP8): codes times their row scales."""
    return e4m3_decode(codes) * np.asarray(scale, np.float64)[:, None]


def gemm_e4m3(a64, wq, bias=None) -> np.ndarray:
    """One FP8 GEMM as the kernels take it: the activations a [R, K] rounded
    to fp32 and quantised per row, the weights wq = (codes [N, K], scale [N])
    quantised per output channel; out = (codes_A codes_W^T) * scale_A[r] *
    scale_W[o] (+ bias), in fp64.

    Paper: Sec. 3.3 (FP8)."""
    ca, sa = quantize_rows(np.asarray(a64, dtype=np.float32))
    cw, sw = wq
    acc = e4m3_decode(ca) @ e4m3_decode(cw).T
    out = acc * sa.astype(np.float64)[:, None] * np.asarray(sw, np.float64)[None, :]
    return out if bias is None else out + _w(bias)


def f32_to_f16_sat(a) -> np.ndarray:
    """fp32 -> fp16 (round to nearest even, saturating at +-65504), as fp64. Numeric helper (the MLP's fp16
    operands); no paper passage."""
    a = np.clip(np.asarray(a, dtype=np.float64), -65504.0, 65504.0)
    return a.astype(np.float32).astype(np.float16).astype(np.float64)


def block_fp8(u_txt, u_img, cu_img, T: int, weights_q, heads: int, mlp: bool, n_img=None):
    """The MMDiT block of ``block`` with e4m3 GEMM operands, in the order the
    kernels take: LayerNorm -> fp32 -> per-row e4m3; QKV = (codes_A codes_W^T)
    * scale_A[r] * scale_W[o] + b, rounded to bf16; attention (fp64) rounded
    to bf16 -> per-row e4m3 -> out-projection; LayerNorm-2 -> per-row e4m3 ->
    MLP1 -> GELU rounded to fp16 -> per-row e4m3 -> MLP2. The residual stream
    stays fp64 here (fp32 in the kernels). ``weights_q`` per stream holds
    (codes, scale) for w_qkv, w_o, w_1, w_2 (see quantize_weights) and the
    bf16 biases. n_img (optional): proportional attention, as in ``block``.
    Returns fp64 (txt, img).

    Paper: Sec. 3.3 (FP8 on top of HiLo-Token) applied to the Sec. 2.1 block."""
    ut = _as_f64(u_txt)
    ui = _as_f64(u_img)
    d = ut.shape[1] if ut.size else ui.shape[1]
    hd = d // heads
    B = len(cu_img) - 1

    q_gemm = gemm_e4m3
    streams = ((ut, weights_q.txt), (ui, weights_q.img))
    qkv = [bf16_to_f32(f32_to_bf16(q_gemm(layer_norm(u), w.w_qkv, w.b_qkv))).astype(np.float64) if u.size else
           np.zeros((0, 3 * d)) for u, w in streams]
    att = [np.zeros_like(ut), np.zeros_like(ui)]
    for b in range(B):
        t0, t1 = b * T, (b + 1) * T
        i0, i1 = int(cu_img[b]), int(cu_img[b + 1])
        joint = np.concatenate([qkv[0][t0:t1], qkv[1][i0:i1]], axis=0)
        kn = None if n_img is None else np.concatenate([np.ones(T), np.asarray(n_img[i0:i1], np.float64)])
        o = np.empty((joint.shape[0], d))
        for h in range(heads):
            c = slice(h * hd, (h + 1) * hd)
            o[:, c] = softmax_attention(joint[:, c], joint[:, d:][:, c], joint[:, 2 * d:][:, c], kn)
        att[0][t0:t1] = o[:T]
        att[1][i0:i1] = o[T:]
    out = []
    for (u, w), a in zip(streams, att):
        if u.size == 0:
            out.append(u)
            continue
        a16 = bf16_to_f32(f32_to_bf16(a)).astype(np.float64)
        u = u + q_gemm(a16, w.w_o, w.b_o)
        if mlp:
            hid = f32_to_f16_sat(gelu_tanh(q_gemm(layer_norm(u), w.w_1, w.b_1)))
            u = u + q_gemm(hid, w.w_2, w.b_2)
        out.append(u)
    return out[0], out[1]


def block_rows_fp8(u_txt, u_img, cu_img, T: int, weights_q, heads: int, mlp: bool, b: int, txt_rows,
                   img_rows, n_img=None):
    """block_fp8's outputs for selected rows of image ``b`` only: keys and
    values of the whole joint sequence of image b (each row's quantisation
    depends on that row alone), queries, attention, out-projection and MLP
    for the given rows (absolute row ids in u_txt / u_img). n_img as in
    block_fp8. fp64 (txt, img).

    Paper: Sec. 3.3, as block_fp8."""
    ut = _as_f64(u_txt)
    ui = _as_f64(u_img)
    d = ut.shape[1] if ut.size else ui.shape[1]
    hd = d // heads
    t0, t1 = b * T, (b + 1) * T
    i0, i1 = int(cu_img[b]), int(cu_img[b + 1])
    wt, wi = weights_q.txt, weights_q.img

    def rows_of(wq, lo, hi):
        return (wq[0][lo:hi], wq[1][lo:hi])

    def qkv_part(u, w, lo, hi):
        # columns [lo, hi) of the QKV output, rounded to bf16 as the kernels store it
        r = gemm_e4m3(layer_norm(u), rows_of(w.w_qkv, lo, hi), np.asarray(w.b_qkv)[lo:hi])
        return bf16_to_f32(f32_to_bf16(r)).astype(np.float64)

    kv = np.concatenate([qkv_part(ut[t0:t1], wt, d, 3 * d) if t1 > t0 else np.zeros((0, 2 * d)),
                         qkv_part(ui[i0:i1], wi, d, 3 * d) if i1 > i0 else np.zeros((0, 2 * d))], axis=0)
    kn = None if n_img is None else np.concatenate([np.ones(t1 - t0), np.asarray(n_img[i0:i1], np.float64)])
    res = []
    for rows, u_all, w in ((np.asarray(txt_rows, int), ut, wt), (np.asarray(img_rows, int), ui, wi)):
        if rows.size == 0:
            res.append(np.zeros((0, d)))
            continue
        u = u_all[rows]
        q = qkv_part(u, w, 0, d)
        o = np.empty((len(rows), d))
        for h in range(heads):
            c = slice(h * hd, (h + 1) * hd)
            o[:, c] = softmax_attention(q[:, c], kv[:, :d][:, c], kv[:, d:][:, c], kn)
        a16 = bf16_to_f32(f32_to_bf16(o)).astype(np.float64)
        u = u + gemm_e4m3(a16, w.w_o, w.b_o)
        if mlp:
            hid = f32_to_f16_sat(gelu_tanh(gemm_e4m3(layer_norm(u), w.w_1, w.b_1)))
            u = u + gemm_e4m3(hid, w.w_2, w.b_2)
        res.append(u)
    return res[0], res[1]


@dataclasses.dataclass
class StreamWeightsQ:
    w_qkv: tuple
    b_qkv: np.ndarray
    w_o: tuple
    b_o: np.ndarray
    w_1: tuple = None
    b_1: np.ndarray = None
    w_2: tuple = None
    b_2: np.ndarray = None


@dataclasses.dataclass
class BlockWeightsQ:
    txt: StreamWeightsQ
    img: StreamWeightsQ


def quantize_weights(w) -> BlockWeightsQ:
    """Per-output-channel e4m3 weights (each row of W[out, in] quantised as
    in quantize_rows, from the bf16 values); biases stay bf16.

    Paper: Sec. 3.3 (FP8)."""
    def one(s):
        q = lambda m: quantize_rows(bf16_to_f32(m)) if m is not None else None
        return StreamWeightsQ(q(s.w_qkv), s.b_qkv, q(s.w_o), s.b_o, q(s.w_1), s.b_1, q(s.w_2), s.b_2)
    return BlockWeightsQ(one(w.txt), one(w.img))


# ---------------------------------------------------------------------------
# The paper's selector: Sobel frequency map, threshold, 16x regionalisation,
# dilated mask (Sec. 2.3 "HiLo-Token Selection")
# ---------------------------------------------------------------------------


def sobel_magnitude(img: np.ndarray) -> np.ndarray:
    """Per-pixel Sobel gradient magnitude of img [B, Hp, Wp, C] fp32 (Sec. 2.3:
    the spatial-frequency map), fp32 in the fixed order of the module header,
    replicate borders. Returns g [B, Hp, Wp] fp32."""
    img = np.ascontiguousarray(img, dtype=np.float32)
    p = np.pad(img, ((0, 0), (1, 1), (1, 1), (0, 0)), mode="edge")
    two = np.float32(2.0)
    # p[:, y + 1, x + 1] is pixel (y, x)
    up, mid, dn = p[:, :-2], p[:, 1:-1], p[:, 2:]
    right = (up[:, :, 2:] + two * mid[:, :, 2:]) + dn[:, :, 2:]
    left = (up[:, :, :-2] + two * mid[:, :, :-2]) + dn[:, :, :-2]
    gx = right - left
    lt, ct, rt = p[:, :, :-2], p[:, :, 1:-1], p[:, :, 2:]
    bottom = (lt[:, 2:] + two * ct[:, 2:]) + rt[:, 2:]
    top = (lt[:, :-2] + two * ct[:, :-2]) + rt[:, :-2]
    gy = bottom - top
    acc = np.zeros(img.shape[:3], dtype=np.float32)
    for c in range(img.shape[3]):
        acc = acc + (gx[..., c] * gx[..., c] + gy[..., c] * gy[..., c])
    return np.sqrt(acc)


def dilate_mask(mask: np.ndarray, H: int, W: int, radius: int) -> np.ndarray:
    """Mask [B, N] dilated on the H x W token grid by a square of radius R
    tokens (Sec. 2.3: the user mask is dilated to keep nearby context)."""
    m = np.asarray(mask, dtype=np.uint8).reshape(-1, H, W) != 0
    out = np.zeros_like(m)
    for dy in range(-radius, radius + 1):
        for dx in range(-radius, radius + 1):
            sh = np.zeros_like(m)
            ys, yd = (slice(0, H - dy), slice(dy, H)) if dy >= 0 else (slice(-dy, H), slice(0, H + dy))
            xs, xd = (slice(0, W - dx), slice(dx, W)) if dx >= 0 else (slice(-dx, W), slice(0, W + dx))
            sh[:, yd, xd] = m[:, ys, xs]
            out |= sh
    return out.reshape(mask.shape).astype(np.uint8)


def sobel_select(img: np.ndarray, mask: np.ndarray, H: int, W: int, patch: int, radius: int,
                 threshold: float) -> np.ndarray:
    """Keep map [B, N] u8 of the paper's selector (Sec. 2.3), in its order:
    normalised Sobel frequency map -> tokens whose magnitude exceeds the
    threshold, regionalised to the token grid by pooling each P x P patch
    (the token is selected when its largest normalised value exceeds the
    threshold) -> union with the user mask dilated by `radius` tokens."""
    g = sobel_magnitude(img)
    B = g.shape[0]
    tokmax = g.reshape(B, H, patch, W, patch).max(axis=(2, 4)).reshape(B, H * W)
    gmax = g.reshape(B, -1).max(axis=1).astype(np.float32)
    with np.errstate(invalid="ignore", divide="ignore"):
        f = tokmax / gmax[:, None]  # fp32 division; 0/0 = nan selects nothing
    hf = f > np.float32(threshold)
    return (hf | (dilate_mask(mask, H, W, radius) != 0)).astype(np.uint8)


def hot_path(x_bits, text_bits, mask, k_keep, k_mid, levels, weights_list, heads, mlp, regions=False,
             prop=False, lf=0):
    """score -> split -> pack -> blocks -> unpack for one batch; regions=True
    takes the window-granular split and the delta unpool, prop=True
    proportional attention (each packed row weighted by its row size).

    Returns (split, packed, (txt_out, img_out), y) with the block outputs in fp64.

    Paper: Sec. 2.3 (selection, the DiT on the compressed sequence, restoration).
    """
    B, H, W, d = x_bits.shape
    T = text_bits.shape[1]
    sp = split(score(x_bits), mask, k_keep, k_mid, H, W, levels, granular=regions, lf=lf)
    packed = pack(x_bits, sp, lf)
    ut, ui = text_bits.reshape(B * T, d), packed
    n_img = row_sizes(sp) if prop else None
    for wts in weights_list:
        ut, ui = block(ut, ui, sp.cu_img, T, wts, heads, mlp, n_img)
    y = unpack_delta(ui, packed, x_bits, sp) if (regions or lf) else unpack(ui, sp)
    return sp, packed, (ut, ui), y
