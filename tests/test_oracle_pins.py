"""Pins of the CPU oracle against facts that do not come from the oracle itself.

Closed forms, hand-worked examples (tests/golden), special cases that reduce to
a library routine, brute force on tiny inputs and invariants of the method
(Sec. 2.3 of the paper: kept tokens stay at full resolution, low-frequency
tokens are pooled, the sequence is concatenated along the token axis).
"""
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import hilo_oracle as O
from paper_2606_13898_gb300 import inputs as I

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def bits(a):
    return I.f32_to_bf16_bits(np.asarray(a, dtype=np.float32))


# ---------------------------------------------------------------- bf16 -----

def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(5)
    v = np.concatenate([rng.standard_normal(20000).astype(np.float32) * 10,
                        # exact ties between two bf16 neighbours (even and odd)
                        np.array([1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -1.0 - 2 ** -8, 0.0, -0.0,
                                  3.0e38, 1e-40], dtype=np.float32)])
    ref = torch.from_numpy(v).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(O.f32_to_bf16(v), ref)
    assert np.array_equal(O.bf16_to_f32(ref), torch.from_numpy(ref.view(np.int16)).view(torch.bfloat16).float().numpy())


# --------------------------------------------------------------- score -----

def test_score_constant_field_is_zero():
    x = np.full((1, 8, 8, 64), 1.75, dtype=np.float32)
    x[..., 5] = -3.0
    assert np.all(O.score(bits(x)) == 0.0)


def test_score_checkerboard_closed_form():
    # +-a alternating in both directions: every 2x2 window has mean 0, so each
    # channel contributes a^2 and the score is d * a^2 for every token.
    a, d = 0.75, 256
    p = np.arange(8)[:, None]
    q = np.arange(6)[None, :]
    sign = np.where((p + q) % 2 == 0, 1.0, -1.0)
    x = (a * sign)[None, :, :, None] * np.ones(d)[None, None, None, :]
    s = O.score(bits(x))
    assert np.all(s == np.float32(d * a * a))


def test_score_linear_ramp_closed_form():
    # x = alpha*p + beta*q (+ a per-channel constant): inside window (P,Q) the
    # mean is alpha*(2P+1/2) + beta*(2Q+1/2), so token (2P+i, 2Q+j) has the
    # residual alpha*(i-1/2) + beta*(j-1/2) in every channel.
    alpha, beta, d = 0.5, 0.25, 64
    H, W = 8, 8
    p = np.arange(H)[:, None, None]
    q = np.arange(W)[None, :, None]
    off = (np.arange(d) % 4)[None, None, :] * 0.25
    x = alpha * p + beta * q + off
    s = O.score(bits(x[None]))[0].reshape(H, W)
    for i in (0, 1):
        for j in (0, 1):
            e = alpha * (i - 0.5) + beta * (j - 0.5)
            assert np.all(s[i::2, j::2] == np.float32(d * e * e)), (i, j)


def test_score_single_token_delta_position():
    # zero field with one token (p0, q0) = (1, 2) set to c in every channel, on
    # a 4 x 6 grid: its window (rows 0-1, cols 2-3) has mean c/4, so the token
    # keeps 3c/4 and its three window mates -c/4; every other token is 0. The
    # positions pin the grid's orientation (a transposed read moves them).
    H, W, d, c = 4, 6, 16, 2.0
    x = np.zeros((1, H, W, d))
    x[0, 1, 2, :] = c
    s = O.score(bits(x))[0].reshape(H, W)
    want = np.zeros((H, W), dtype=np.float32)
    want[0:2, 2:4] = np.float32(d * (c / 4) ** 2)
    want[1, 2] = np.float32(d * (3 * c / 4) ** 2)
    assert np.array_equal(s, want)


def test_score_agrees_with_fp64_sum():
    wl = I.tiny_layer()
    b = I.make_batch(wl)
    s32 = O.score(b.x).astype(np.float64)
    s64 = O.score_f64(b.x)
    assert np.max(np.abs(s32 - s64) / np.maximum(s64, 1e-30)) < 1e-5


def test_score_fixed_order_scalar_walkthrough():
    # One token of a random field walked through the fixed order with scalar
    # fp32 arithmetic: pins the vectorised grouping and the halving tree.
    rng = np.random.default_rng(11)
    d = 3072
    xb = bits(rng.standard_normal((1, 2, 2, d)))
    x = O.bf16_to_f32(xb)[0]
    f = np.float32
    for t, (pi, qi) in enumerate(((0, 0), (0, 1), (1, 0), (1, 1))):
        part = [f(0.0)] * 128
        for c in range(d):
            m = ((x[0, 0, c] + x[0, 1, c]) + (x[1, 0, c] + x[1, 1, c])) * f(0.25)
            e = f(x[pi, qi, c] - m)
            g = c // 8
            part[g % 128] = f(part[g % 128] + f(e * e))
        for h in (64, 32, 16, 8, 4, 2, 1):
            for j in range(h):
                part[j] = f(part[j] + part[j + h])
        assert O.score(xb)[0, t] == part[0]


# --------------------------------------------------------------- split -----

def _golden_cases():
    with open(os.path.join(GOLDEN, "split_worked_examples.json")) as fh:
        return json.load(fh)["cases"]


@pytest.mark.parametrize("case", _golden_cases(), ids=lambda c: c["name"])
def test_split_hand_worked(case):
    s = np.array([case["score"]], dtype=np.float32)
    m = np.array([case["mask"]], dtype=np.uint8)
    sp = O.split(s, m, [case["k_keep"]], [case["k_mid"]], case["H"], case["W"], case["levels"])
    assert sp.labels[0].tolist() == case["labels"]
    assert sp.row_src.tolist() == case["row_src"]
    assert sp.counts[0].tolist() == case["counts"]
    assert sp.cu_img.tolist() == case["cu_img"]
    assert sp.tok_row[0].tolist() == case["tok_row"]


def _brute_split(s, m, k, kmid, H, W, levels):
    """Pure-Python split of one image from the rule, by full sort."""
    N = H * W
    order = sorted(range(N), key=lambda i: (-float(s[i]), i))
    keep = set(order[:k]) | {i for i in range(N) if m[i]}
    rest = [i for i in order if i not in keep]
    pool2 = set(rest[:kmid]) if levels == 2 else set(rest)
    pool4 = set(rest[kmid:]) if levels == 2 else set()
    w2 = sorted({(i // W // 2) * (W // 2) + (i % W) // 2 for i in pool2})
    w4 = sorted({(i // W // 4) * (W // 4) + (i % W) // 4 for i in pool4})
    return sorted(keep), w2, w4, pool2, pool4


@pytest.mark.parametrize("levels", [1, 2])
@pytest.mark.parametrize("seed", range(6))
def test_split_brute_force(seed, levels):
    rng = np.random.default_rng(seed)
    H, W = (8, 8) if seed % 2 else (4, 12)
    N = H * W
    B = 3
    # coarse scores so that ties are common
    s = (rng.integers(0, 6, size=(B, N)) * 0.5).astype(np.float32)
    m = (rng.random((B, N)) < 0.15).astype(np.uint8)
    kk = rng.integers(0, N + 1, size=B)
    km = rng.integers(0, N + 1, size=B)
    sp = O.split(s, m, kk, km, H, W, levels)
    for b in range(B):
        keep, w2, w4, pool2, pool4 = _brute_split(s[b], m[b], int(kk[b]), int(km[b]), H, W, levels)
        base = int(sp.cu_img[b])
        assert sp.counts[b].tolist() == [len(keep), len(w2), len(w4)]
        rows = sp.row_src[base:int(sp.cu_img[b + 1])].tolist()
        assert rows == keep + w2 + w4
        assert {i for i in range(N) if sp.labels[b, i] == O.POOL2} == pool2
        assert {i for i in range(N) if sp.labels[b, i] == O.POOL4} == pool4
        # every token reads back the row that holds it
        for i in range(N):
            r = int(sp.tok_row[b, i]) - base
            if i in keep:
                assert rows[r] == i and r < len(keep)
            elif i in pool2:
                assert len(keep) <= r < len(keep) + len(w2)
                assert rows[r] == (i // W // 2) * (W // 2) + (i % W) // 2
            else:
                assert r >= len(keep) + len(w2)
                assert rows[r] == (i // W // 4) * (W // 4) + (i % W) // 4


def test_split_ties_take_lowest_indices():
    N = 64
    s = np.ones((1, N), dtype=np.float32)
    sp = O.split(s, np.zeros((1, N), np.uint8), [10], [0], 8, 8, 1)
    assert np.nonzero(sp.labels[0] == O.KEEP)[0].tolist() == list(range(10))


def test_split_extremes():
    rng = np.random.default_rng(3)
    N = 64
    s = rng.random((1, N)).astype(np.float32)
    m = (rng.random((1, N)) < 0.2).astype(np.uint8)
    sp0 = O.split(s, m, [0], [0], 8, 8, 1)
    assert np.array_equal(sp0.labels[0] == O.KEEP, m[0] == 1)
    spN = O.split(s, m, [N], [0], 8, 8, 1)
    assert np.all(spN.labels == O.KEEP) and spN.counts[0].tolist() == [N, 0, 0]
    assert spN.row_src.tolist() == list(range(N))
    spall = O.split(s, np.ones_like(m), [0], [0], 8, 8, 2)
    assert np.all(spall.labels == O.KEEP)


def test_split_count_law():
    wl = I.tiny_layer()
    b = I.make_batch(wl)
    s = O.score(b.x)
    sp = O.split(s, b.mask, b.k_keep, b.k_mid, wl.H, wl.W, 1)
    top = set(O.ranking(s[0])[: int(b.k_keep[0])].tolist())
    assert int(sp.counts[0, 0]) == len(top | set(np.nonzero(b.mask[0])[0].tolist()))


def test_split_granular_hand_worked():
    """4 x 4 grid, one level, k_keep = 1, no mask. The largest score sits at
    token 5 (row 1, column 1), so its 2 x 2 window {0, 1, 4, 5} is kept whole
    and the three other windows are pooled with all four members each."""
    s = np.zeros((1, 16), dtype=np.float32)
    s[0, 5] = 3.0
    s[0, 10] = 2.0
    sp = O.split(s, np.zeros((1, 16), np.uint8), [1], [0], 4, 4, 1, granular=True)
    assert sp.labels[0].tolist() == [0, 0, 1, 1, 0, 0, 1, 1, 1, 1, 1, 1, 1, 1, 1, 1]
    assert sp.counts[0].tolist() == [4, 3, 0]
    assert sp.row_src.tolist() == [0, 1, 4, 5, 1, 2, 3]
    assert sp.tok_row[0].tolist() == [0, 1, 4, 4, 2, 3, 4, 4, 5, 5, 6, 6, 5, 5, 6, 6]
    # two levels on a 4 x 8 grid (4 x 4 blocks: columns 0-3 and 4-7; 2 x 2
    # window id = 4 * (row // 2) + col // 2): token 9 (row 1, column 1) ranks
    # first, token 22 (row 2, column 6, right block) second. k_keep = 1 keeps
    # window 0 = {0, 1, 8, 9} whole. With k_mid = 1 token 22 is above the
    # cut, so neither block is entirely below it: the left block's windows
    # 1, 4, 5 and the right block's 2, 3, 6, 7 are pooled 2 x 2.
    s = np.zeros((1, 32), dtype=np.float32)
    s[0, 9] = 3.0
    s[0, 22] = 2.0
    sp = O.split(s, np.zeros((1, 32), np.uint8), [1], [1], 4, 8, 2, granular=True)
    assert sp.counts[0].tolist() == [4, 7, 0]
    assert sp.row_src.tolist() == [0, 1, 8, 9, 1, 2, 3, 4, 5, 6, 7]
    # k_mid = 0: the whole right block is below the cut and is pooled 4 x 4
    # (4 x 4 window 1); the left block still holds the kept window
    sp = O.split(s, np.zeros((1, 32), np.uint8), [1], [0], 4, 8, 2, granular=True)
    assert sp.counts[0].tolist() == [4, 3, 1]
    assert sp.row_src.tolist() == [0, 1, 8, 9, 1, 4, 5, 1]


def _brute_split_granular(s, m, k, kmid, H, W, levels):
    """Pure-Python window-granular split of one image from the rule."""
    N = H * W
    order = sorted(range(N), key=lambda i: (-float(s[i]), i))
    sel = set(order[:k]) | {i for i in range(N) if m[i]}
    win2 = lambda i: (i // W // 2, (i % W) // 2)
    win4 = lambda i: (i // W // 4, (i % W) // 4)
    kept_w = {win2(i) for i in sel}
    keep = {i for i in range(N) if win2(i) in kept_w}
    rest = [i for i in order if i not in keep]
    if levels == 1:
        return keep, set(rest), set()
    below = set(rest[kmid:])
    pool4 = set()
    for bp in range(H // 4):
        for bq in range(W // 4):
            mem = [(4 * bp + i) * W + 4 * bq + j for i in range(4) for j in range(4)]
            if all(t in below for t in mem):
                pool4 |= set(mem)
    pool2 = set(rest) - pool4
    return keep, pool2, pool4


@pytest.mark.parametrize("levels", [1, 2])
@pytest.mark.parametrize("seed", range(6))
def test_split_granular_brute_force_and_invariants(seed, levels):
    rng = np.random.default_rng(100 + seed)
    H, W = (8, 8) if seed % 2 else (4, 12)
    N, B = H * W, 3
    s = (rng.integers(0, 6, size=(B, N)) * 0.5).astype(np.float32)
    m = (rng.random((B, N)) < 0.1).astype(np.uint8)
    kk = rng.integers(0, N // 3, size=B)
    km = rng.integers(0, N // 2, size=B)
    sp = O.split(s, m, kk, km, H, W, levels, granular=True)
    flat = O.split(s, m, kk, km, H, W, levels)
    for b in range(B):
        keep, pool2, pool4 = _brute_split_granular(s[b], m[b], int(kk[b]), int(km[b]), H, W, levels)
        lab = sp.labels[b]
        assert {i for i in range(N) if lab[i] == O.KEEP} == keep
        assert {i for i in range(N) if lab[i] == O.POOL2} == pool2
        assert {i for i in range(N) if lab[i] == O.POOL4} == pool4
        # every kept 2x2 window holds a token the flat split keeps, and the
        # flat kept set is covered
        fk = flat.labels[b] == O.KEEP
        assert np.all(lab[fk] == O.KEEP)
        g = lab.reshape(H // 2, 2, W // 2, 2).transpose(0, 2, 1, 3).reshape(-1, 4)
        f = fk.reshape(H // 2, 2, W // 2, 2).transpose(0, 2, 1, 3).reshape(-1, 4)
        for wl, wf in zip(g, f):
            assert len(set(wl.tolist())) == 1 or not np.any(wl == O.KEEP)   # kept windows are whole
            assert (wl[0] == O.KEEP) == bool(wf.any())
        nk, n2, n4 = (int(c) for c in sp.counts[b])
        assert nk == 4 * int(f.any(axis=1).sum())
        # pooled windows are full
        assert 4 * n2 == int(np.sum(lab == O.POOL2)) and 16 * n4 == int(np.sum(lab == O.POOL4))
        base = int(sp.cu_img[b])
        for i in range(N):
            r = int(sp.tok_row[b, i]) - base
            if lab[i] == O.KEEP:
                assert int(sp.row_src[base + r]) == i
    spN = O.split(s, m, [N] * B, [0] * B, H, W, levels, granular=True)
    assert np.all(spN.labels == O.KEEP)


def test_split_lf_hand_worked():
    """4 x 4 grid, lf = 2, k_keep = 1 (token 5 ranks first), mask token 15:
    kept [5, 15], then all four 2 x 2 windows of the grid; every other token
    reads its window's row."""
    s = np.zeros((1, 16), dtype=np.float32)
    s[0, 5] = 1.0
    m = np.zeros((1, 16), np.uint8)
    m[0, 15] = 1
    sp = O.split(s, m, [1], [0], 4, 4, 1, lf=2)
    assert sp.counts[0].tolist() == [2, 4, 0]
    assert sp.row_src.tolist() == [5, 15, 0, 1, 2, 3]
    assert sp.tok_row[0].tolist() == [2, 2, 3, 3, 2, 0, 3, 3, 4, 4, 5, 5, 4, 4, 5, 1]
    assert sp.labels[0].tolist() == [O.LF] * 5 + [O.KEEP] + [O.LF] * 9 + [O.KEEP]


@pytest.mark.parametrize("lf", [2, 4, 8])
def test_split_lf_count_law_and_rows(lf):
    rng = np.random.default_rng(50 + lf)
    H, W, B = 16, 24, 2
    N = H * W
    s = rng.random((B, N)).astype(np.float32)
    m = (rng.random((B, N)) < 0.1).astype(np.uint8)
    kk = [N // 5, 0]
    sp = O.split(s, m, kk, [0, 0], H, W, 1, lf=lf)
    nlf = (H // lf) * (W // lf)
    for b in range(B):
        top = set(O.ranking(s[b])[:kk[b]].tolist()) | set(np.nonzero(m[b])[0].tolist())
        base = int(sp.cu_img[b])
        assert sp.counts[b].tolist() == [len(top), nlf, 0]
        assert sp.row_src[base:base + len(top)].tolist() == sorted(top)
        assert sp.row_src[base + len(top):int(sp.cu_img[b + 1])].tolist() == list(range(nlf))
        for i in range(N):
            r = int(sp.tok_row[b, i]) - base
            if i in top:
                assert sp.labels[b, i] == O.KEEP and int(sp.row_src[base + r]) == i
            else:
                assert sp.labels[b, i] == O.LF
                assert r - len(top) == (i // W // lf) * (W // lf) + (i % W) // lf


@pytest.mark.parametrize("lf", [2, 4])
def test_pack_lf_is_the_downsampled_grid(lf):
    """LF rows are the grid average-pooled lf-fold per side (all members,
    kept ones included): the fp64 reshape-mean within one bf16 rounding and
    the fp32 summation; constant windows pool exactly and the delta unpool of
    an unchanged block returns every token."""
    rng = np.random.default_rng(60 + lf)
    H, W, d = 8, 16, 32
    x = rng.standard_normal((1, H, W, d)).astype(np.float32)
    xb = bits(x)
    xf = O.bf16_to_f32(xb)[0].astype(np.float64)
    s = O.score(xb)
    m = (rng.random((1, H * W)) < 0.2).astype(np.uint8)
    sp = O.split(s, m, [H * W // 4], [0], H, W, 1, lf=lf)
    packed = O.pack(xb, sp, lf)
    nk = int(sp.counts[0, 0])
    ref = xf.reshape(H // lf, lf, W // lf, lf, d).mean(axis=(1, 3)).reshape(-1, d)
    got = O.bf16_to_f32(packed[nk:]).astype(np.float64)
    assert np.all(np.abs(got - ref) <= np.abs(ref) * 2 ** -8 + 1e-6)
    # kept rows are the tokens themselves
    assert np.array_equal(packed[:nk], xb.reshape(-1, d)[sp.row_src[:nk]])
    # constant windows: exact pooling, and y = x through the delta unpool
    blk = rng.standard_normal((H // lf, W // lf, d)).astype(np.float32)
    xc = bits(np.repeat(np.repeat(blk, lf, axis=0), lf, axis=1)[None])
    pc = O.pack(xc, sp, lf)
    assert np.array_equal(pc[nk:], bits(blk).reshape(-1, d))
    y = O.unpack_delta(O.bf16_to_f32(pc), pc, xc, sp)
    assert np.array_equal(y, O.bf16_to_f32(xc))


# ---------------------------------------------------------- pack/unpack ----



def test_pack_sums_members_in_raster_order():
    # one 2x2 window, all four members pooled, channel values 2^26, 1, -2^26, 1
    # in raster order: in fp32, (2^26 + 1) rounds to 2^26, so the raster-order
    # sum is 1 and the mean 1/4 (column-major order would give 2 and 1/2)
    v = np.array([2.0 ** 26, 1.0, -(2.0 ** 26), 1.0])
    x = np.repeat(v.reshape(1, 2, 2, 1), 8, axis=3)
    sp = O.split(np.zeros((1, 4), np.float32), np.zeros((1, 4), np.uint8), [0], [0], 2, 2, 1)
    assert sp.counts[0].tolist() == [0, 1, 0]
    packed = O.bf16_to_f32(O.pack(bits(x), sp))
    assert np.all(packed == 0.25)


def test_pack_constant_windows_lossless():
    rng = np.random.default_rng(4)
    H, W, d = 8, 8, 32
    # each 4x4 block constant (distinct per block and channel)
    blk = rng.standard_normal((H // 4, W // 4, d)).astype(np.float32)
    x = np.repeat(np.repeat(blk, 4, axis=0), 4, axis=1)[None]
    xb = bits(x)
    s = rng.random((1, H * W)).astype(np.float32)
    for levels in (1, 2):
        sp = O.split(s, np.zeros((1, H * W), np.uint8), [10], [20], H, W, levels)
        packed = O.pack(xb, sp)
        y = O.unpack(O.bf16_to_f32(packed), sp)
        assert np.array_equal(y, O.bf16_to_f32(xb).reshape(1, H * W, d))


def test_unpack_pack_identity_on_kept_rows_and_brute_mean():
    wl = I.tiny_layer()
    b = I.make_batch(wl)
    s = O.score(b.x)
    sp = O.split(s, b.mask, b.k_keep, b.k_mid, wl.H, wl.W, 1)
    packed = O.pack(b.x, sp)
    xf = O.bf16_to_f32(b.x).reshape(1, wl.N, wl.d)
    y = O.unpack(O.bf16_to_f32(packed), sp)
    kept = sp.labels[0] == O.KEEP
    assert np.array_equal(y[0][kept], xf[0][kept])
    # pooled rows: the mean of the 2x2 window's pooled members (fp64 mean,
    # within one bf16 rounding)
    nk, n2, _ = sp.counts[0]
    W = wl.W
    for r in range(nk, nk + n2):
        w = int(sp.row_src[r])
        wp, wq = divmod(w, W // 2)
        mem = [(2 * wp + i) * W + 2 * wq + j for i in range(2) for j in range(2)]
        mem = [t for t in mem if sp.labels[0, t] == O.POOL2]
        assert 1 <= len(mem) <= 4
        ref = xf[0, mem].astype(np.float64).mean(axis=0)
        got = O.bf16_to_f32(packed[r]).astype(np.float64)
        assert np.all(np.abs(got - ref) <= np.abs(ref) * 2 ** -8 + 1e-30)


def _delta_case(granular=True, levels=2):
    rng = np.random.default_rng(21)
    H, W, d = 16, 16, 32
    x = rng.uniform(-4, 4, size=(1, H, W, d)).astype(np.float32)
    xb = bits(x)
    s = O.score(xb)
    # at most 8 of the 16 4 x 4 blocks hold a kept or above-cut token
    sp = O.split(s, np.zeros((1, H * W), np.uint8), [4], [4], H, W, levels, granular=granular)
    return xb, sp, O.pack(xb, sp)


@pytest.mark.parametrize("granular", [False, True])
def test_unpack_delta_identity_block_returns_x(granular):
    """A block that changes nothing (out = packed) leaves every pooled member
    at its own value, bit for bit; kept tokens read their own rows."""
    xb, sp, packed = _delta_case(granular)
    out = O.bf16_to_f32(packed)
    y = O.unpack_delta(out, packed, xb, sp)
    assert np.array_equal(y, O.bf16_to_f32(xb))


def test_unpack_delta_shift_is_exact():
    """A block that adds 0.5 everywhere: out - packed = 0.5 exactly and
    x + 0.5 is exact for |x| < 4, so every pooled member moves by exactly 0.5
    while kept tokens take their output rows."""
    xb, sp, packed = _delta_case()
    out = O.bf16_to_f32(packed) + np.float32(0.5)
    y = O.unpack_delta(out, packed, xb, sp).reshape(-1, xb.shape[-1])
    xf = O.bf16_to_f32(xb).reshape(-1, xb.shape[-1])
    lab = sp.labels[0]
    assert np.array_equal(y[lab != O.KEEP], xf[lab != O.KEEP] + np.float32(0.5))
    assert np.array_equal(y[lab == O.KEEP], xf[lab == O.KEEP] + np.float32(0.5))


def test_unpack_delta_window_mean_is_window_output():
    """Over a full window the members' mean equals the window's output up to
    the bf16 rounding of the pooled value: mean(y) - out = mean(x) - packed."""
    xb, sp, packed = _delta_case()
    rng = np.random.default_rng(5)
    out = rng.standard_normal((packed.shape[0], packed.shape[1])).astype(np.float32)
    y = O.unpack_delta(out, packed, xb, sp).reshape(-1, xb.shape[-1]).astype(np.float64)
    xf = O.bf16_to_f32(xb).reshape(-1, xb.shape[-1]).astype(np.float64)
    pf = O.bf16_to_f32(packed).astype(np.float64)
    nk, n2, n4 = (int(c) for c in sp.counts[0])
    assert n2 > 0 and n4 > 0
    for r in range(nk, nk + n2 + n4):
        mem = np.nonzero(sp.tok_row[0] == r)[0]
        assert len(mem) in (4, 16)
        lhs = y[mem].mean(axis=0) - out[r]
        rhs = xf[mem].mean(axis=0) - pf[r]
        assert np.all(np.abs(lhs - rhs) <= 4 * 2.0 ** -22 * (np.abs(out[r]) + 8))


# --------------------------------------------------------------- block -----


def test_layer_norm_and_gelu_closed_forms():
    ln = O.layer_norm(np.array([[1.0, -1.0, 1.0, -1.0], [3.0, 3.0, 3.0, 3.0]]))
    assert np.allclose(ln[0], np.array([1, -1, 1, -1]) / math.sqrt(1 + 1e-6), rtol=0, atol=1e-15)
    assert np.all(ln[1] == 0.0)
    z = np.linspace(-6, 6, 2001)
    from scipy.special import erf
    exact = 0.5 * z * (1 + erf(z / math.sqrt(2)))
    assert np.max(np.abs(O.gelu_tanh(z) - exact)) < 1e-3
    assert O.gelu_tanh(np.array([0.0]))[0] == 0.0


def test_attention_two_token_closed_form():
    # head_dim 1: logits 0 and ln 2 give weights 1/3 and 2/3
    q = np.array([[1.0]])
    k = np.array([[0.0], [math.log(2.0)]])
    v = np.array([[3.0], [6.0]])
    assert abs(O.softmax_attention(q, k, v)[0, 0] - 5.0) < 1e-12


def test_attention_scale_closed_form():
    # head_dim 4: the logit of key j is q.k_j / sqrt(4); with q.k = 2 ln 3
    # the weights are 1/4 and 3/4 (a scale of 1/d or 1 would give others)
    q = np.array([[1.0, 0.0, 0.0, 0.0]])
    k = np.array([[0.0, 0.0, 0.0, 0.0], [2.0 * math.log(3.0), 0.0, 0.0, 0.0]])
    v = np.array([[4.0, 0.0, 0.0, 0.0], [8.0, 0.0, 0.0, 0.0]])
    assert abs(O.softmax_attention(q, k, v)[0, 0] - 7.0) < 1e-12


def _rand_weights(rng, d, mlp):
    def one():
        s = I.StreamWeights(w_qkv=bits(rng.normal(0, 0.2, (3 * d, d))), b_qkv=bits(rng.normal(0, 0.2, 3 * d)),
                            w_o=bits(rng.normal(0, 0.2, (d, d))), b_o=bits(rng.normal(0, 0.2, d)))
        if mlp:
            s.w_1 = bits(rng.normal(0, 0.2, (4 * d, d)))
            s.b_1 = bits(rng.normal(0, 0.2, 4 * d))
            s.w_2 = bits(rng.normal(0, 0.2, (d, 4 * d)))
            s.b_2 = bits(rng.normal(0, 0.2, d))
        return s
    return I.BlockWeights(txt=one(), img=one())


def test_block_uniform_attention_closed_form():
    # Constant rows -> LayerNorm output 0 -> q, k, v equal their biases for
    # every token -> uniform attention returns b_v. With no MLP the block is
    # u + b_v W_o^T + b_o for each stream.
    rng = np.random.default_rng(2)
    d, heads, T = 16, 2, 3
    w = _rand_weights(rng, d, mlp=False)
    ut = np.ones((T, d)) * 0.5
    ui = np.ones((5, d)) * -2.0
    ot, oi = O.block(ut, ui, [0, 5], T, w, heads, mlp=False)
    f = lambda a: O.bf16_to_f32(a).astype(np.float64)
    bv_t = f(w.txt.b_qkv)[2 * d:]
    bv_i = f(w.img.b_qkv)[2 * d:]
    # every query sees 3 text keys (b_k of text) and 5 image keys (b_k of
    # image): two distinct logits per head, weighted by their multiplicity
    hd = d // heads
    o_ref = {}
    for name, bq in (("t", f(w.txt.b_qkv)[:d]), ("i", f(w.img.b_qkv)[:d])):
        o = np.empty(d)
        for h in range(heads):
            c = slice(h * hd, (h + 1) * hd)
            lt = bq[c] @ f(w.txt.b_qkv)[d:2 * d][c] / math.sqrt(hd)
            li = bq[c] @ f(w.img.b_qkv)[d:2 * d][c] / math.sqrt(hd)
            wt = 3 * math.exp(lt) / (3 * math.exp(lt) + 5 * math.exp(li))
            o[c] = wt * bv_t[c] + (1 - wt) * bv_i[c]
        o_ref[name] = o
    exp_t = ut + o_ref["t"] @ f(w.txt.w_o).T + f(w.txt.b_o)
    exp_i = ui + o_ref["i"] @ f(w.img.w_o).T + f(w.img.b_o)
    assert np.allclose(ot, exp_t, rtol=0, atol=1e-12)
    assert np.allclose(oi, exp_i, rtol=0, atol=1e-12)


def _brute_block(ut, ui, T, w, heads, mlp):
    """Scalar pure-Python block on one image (tiny shapes only)."""
    f = lambda a: O.bf16_to_f32(a).astype(np.float64).tolist()
    d = len(ut[0])
    hd = d // heads

    def ln(row):
        mu = sum(row) / d
        var = sum((x - mu) ** 2 for x in row) / d
        return [(x - mu) / math.sqrt(var + 1e-6) for x in row]

    def lin(row, W_, b_):
        return [sum(row[k] * W_[o][k] for k in range(len(row))) + b_[o] for o in range(len(W_))]

    def gelu(z):
        return 0.5 * z * (1 + math.tanh(math.sqrt(2 / math.pi) * (z + 0.044715 * z ** 3)))

    rows = [(list(r), w.txt) for r in ut] + [(list(r), w.img) for r in ui]
    qkv = [lin(ln(r), f(sw.w_qkv), f(sw.b_qkv)) for r, sw in rows]
    out = []
    for i, (r, sw) in enumerate(rows):
        o = [0.0] * d
        for h in range(heads):
            lg = [sum(qkv[i][h * hd + c] * qkv[j][d + h * hd + c] for c in range(hd)) / math.sqrt(hd)
                  for j in range(len(rows))]
            mx = max(lg)
            e = [math.exp(x - mx) for x in lg]
            z = sum(e)
            for c in range(hd):
                o[h * hd + c] = sum(e[j] / z * qkv[j][2 * d + h * hd + c] for j in range(len(rows)))
        u = [a + b for a, b in zip(r, lin(o, f(sw.w_o), f(sw.b_o)))]
        if mlp:
            hmid = [gelu(z) for z in lin(ln(u), f(sw.w_1), f(sw.b_1))]
            u = [a + b for a, b in zip(u, lin(hmid, f(sw.w_2), f(sw.b_2)))]
        out.append(u)
    return np.array(out[:T]), np.array(out[T:])


@pytest.mark.parametrize("grid,mlp", [((4, 4), True), ((8, 8), False)])
def test_block_brute_force_tiny(grid, mlp):
    rng = np.random.default_rng(7)
    H, W = grid
    d, heads, T = 16, 2, 3
    w = _rand_weights(rng, d, mlp)
    ut = bits(rng.standard_normal((T, d)))
    ui = bits(rng.standard_normal((H * W, d)))
    ot, oi = O.block(ut, ui, [0, H * W], T, w, heads, mlp)
    bt, bi = _brute_block(O.bf16_to_f32(ut).astype(np.float64), O.bf16_to_f32(ui).astype(np.float64),
                          T, w, heads, mlp)
    assert np.max(np.abs(ot - bt)) < 1e-9 and np.max(np.abs(oi - bi)) < 1e-9


def test_block_brute_force_d64_two_images():
    # d=64, 2 heads of 32, two images of different lengths in one packed batch
    rng = np.random.default_rng(8)
    d, heads, T = 64, 2, 2
    w = _rand_weights(rng, d, mlp=False)
    ut = bits(rng.standard_normal((2 * T, d)))
    ui = bits(rng.standard_normal((16 + 9, d)))
    cu = [0, 16, 25]
    ot, oi = O.block(ut, ui, cu, T, w, heads, mlp=False)
    for b in range(2):
        f = lambda a: O.bf16_to_f32(a).astype(np.float64)
        bt, bi = _brute_block(f(ut[b * T:(b + 1) * T]), f(ui[cu[b]:cu[b + 1]]), T, w, heads, False)
        assert np.max(np.abs(ot[b * T:(b + 1) * T] - bt)) < 1e-9
        assert np.max(np.abs(oi[cu[b]:cu[b + 1]] - bi)) < 1e-9


def test_block_rows_matches_block():
    rng = np.random.default_rng(9)
    d, heads, T = 32, 4, 5
    w = _rand_weights(rng, d, mlp=True)
    ut = bits(rng.standard_normal((2 * T, d)))
    ui = bits(rng.standard_normal((30, d)))
    cu = [0, 12, 30]
    ot, oi = O.block(ut, ui, cu, T, w, heads, True)
    rt, ri = O.block_rows(ut, ui, cu, T, w, heads, True, 1, [5, 8], [12, 20, 29])
    assert np.allclose(rt, ot[[5, 8]], rtol=0, atol=1e-12)
    assert np.allclose(ri, oi[[12, 20, 29]], rtol=0, atol=1e-12)


def test_block_permutation_equivariance():
    rng = np.random.default_rng(10)
    d, heads, T = 32, 2, 4
    w = _rand_weights(rng, d, mlp=True)
    ut = bits(rng.standard_normal((T, d)))
    ui = bits(rng.standard_normal((20, d)))
    perm = rng.permutation(20)
    _, oi = O.block(ut, ui, [0, 20], T, w, heads, True)
    _, op = O.block(ut, ui[perm], [0, 20], T, w, heads, True)
    assert np.allclose(op, oi[perm], rtol=0, atol=1e-10)


def test_proportional_attention_equals_duplicated_keys():
    """A key with weight n attends exactly like n identical copies of it."""
    rng = np.random.default_rng(30)
    q = rng.standard_normal((7, 16))
    k = rng.standard_normal((9, 16)) * 2
    v = rng.standard_normal((9, 16))
    n = rng.integers(1, 6, size=9)
    got = O.softmax_attention(q, k, v, n)
    ref = O.softmax_attention(q, np.repeat(k, n, axis=0), np.repeat(v, n, axis=0))
    assert np.allclose(got, ref, rtol=0, atol=1e-12)
    # two keys, equal logits: the weights split n0 : n1
    q2 = np.zeros((1, 4))
    k2 = rng.standard_normal((2, 4))
    v2 = np.array([[1.0, 0, 0, 0], [0, 1.0, 0, 0]])
    o = O.softmax_attention(q2, k2, v2, [3, 1])
    assert np.allclose(o[0, :2], [0.75, 0.25], rtol=0, atol=1e-15)


def test_block_proportional_ones_is_plain_block():
    rng = np.random.default_rng(31)
    d, heads, T = 32, 2, 4
    w = _rand_weights(rng, d, mlp=True)
    ut = bits(rng.standard_normal((2 * T, d)))
    ui = bits(rng.standard_normal((13, d)))
    cu = [0, 6, 13]
    a = O.block(ut, ui, cu, T, w, heads, True)
    b = O.block(ut, ui, cu, T, w, heads, True, n_img=np.ones(13, np.float32))
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


def test_block_proportional_equals_block_on_duplicated_rows():
    """The whole block with row weights n equals the plain block on the
    sequence where image row r appears n_r times (its first copy's output,
    and every text output, agree), for two images of one batch."""
    rng = np.random.default_rng(32)
    d, heads, T = 32, 2, 3
    w = _rand_weights(rng, d, mlp=True)
    ut = bits(rng.standard_normal((2 * T, d)))
    ui = bits(rng.standard_normal((9, d)))
    cu = [0, 5, 9]
    n = np.array([1, 3, 1, 2, 4, 2, 1, 1, 3], dtype=np.float32)
    pt, pi = O.block(ut, ui, cu, T, w, heads, True, n_img=n)
    rep = np.repeat(np.arange(9), n.astype(int))
    cu_dup = [0, int(n[:5].sum()), int(n.sum())]
    dt, di = O.block(ut, ui[rep], cu_dup, T, w, heads, True)
    first = np.searchsorted(rep, np.arange(9))
    assert np.allclose(pt, dt, rtol=0, atol=1e-10)
    assert np.allclose(pi, di[first], rtol=0, atol=1e-10)
    # the sampled-rows form agrees with the whole block
    rt, ri = O.block_rows(ut, ui, cu, T, w, heads, True, 1, [3, 5], [6, 8], n_img=n)
    assert np.allclose(rt, pt[[3, 5]], rtol=0, atol=1e-12) and np.allclose(ri, pi[[6, 8]], rtol=0, atol=1e-12)


@pytest.mark.parametrize("granular", [False, True])
def test_row_sizes_count_the_grid(granular):
    rng = np.random.default_rng(33)
    H, W, B = 8, 12, 2
    N = H * W
    s = rng.random((B, N)).astype(np.float32)
    m = (rng.random((B, N)) < 0.1).astype(np.uint8)
    sp = O.split(s, m, [10, 30], [20, 10], H, W, 2, granular=granular)
    n = O.row_sizes(sp)
    for b in range(B):
        r0, r1 = int(sp.cu_img[b]), int(sp.cu_img[b + 1])
        assert n[r0:r1].sum() == N
        nk, n2, n4 = (int(c) for c in sp.counts[b])
        assert np.all(n[r0:r0 + nk] == 1)
        for r in range(r0 + nk, r1):
            size, cls = (2, O.POOL2) if r < r0 + nk + n2 else (4, O.POOL4)
            mem = O.window_members(int(sp.row_src[r]), size, W)
            assert n[r] == sum(1 for t in mem if sp.labels[b, t] == cls)
            if granular:
                assert n[r] == size * size


# ------------------------------------------------------------------- FP8 --

def test_e4m3_codes_roundtrip_and_match_torch():
    """Every finite e4m3 code decodes and re-encodes to itself (both zeros
    keep their sign); in-range fp32 values round like torch's float8_e4m3fn
    cast (round to nearest, ties to even)."""
    codes = np.arange(256, dtype=np.uint8)
    vals = O.e4m3_decode(codes)
    fin = ~np.isnan(vals)
    assert fin.sum() == 254 and np.nanmax(vals) == 448.0 and np.nanmin(vals) == -448.0
    assert np.array_equal(O.e4m3_encode(vals[fin].astype(np.float32)), codes[fin])
    x = (np.random.default_rng(7).standard_normal(200000) * 40).astype(np.float32)
    x = np.concatenate([x[np.abs(x) <= 448], (np.random.default_rng(8).random(20000) * 0.03).astype(np.float32)])
    ref = torch.from_numpy(x).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    assert np.array_equal(O.e4m3_encode(x), ref)


def test_e4m3_ties_saturation_subnormals():
    t = np.array([1.0625, 1.1875, 1.0625 + 2 ** -20, 464.0, 1000.0, -1e30, 2 ** -10, 3 * 2 ** -10, 2 ** -6,
                  0.9375 + 2 ** -5], dtype=np.float32)
    got = O.e4m3_decode(O.e4m3_encode(t))
    # 1.0625 is halfway between 1 and 1.125: to the even mantissa (1);
    # 1.1875 halfway between 1.125 and 1.25: to 1.25; just above halfway
    # rounds up; beyond 448 saturates; 2^-10 is half the smallest
    # subnormal 2^-9 (ties to 0); 3 * 2^-10 rounds to 2 * 2^-9; 2^-6 is
    # the smallest normal; 0.96875 sits halfway between 0.9375 and 1.0
    assert got.tolist() == [1.0, 1.25, 1.125, 448.0, 448.0, -448.0, 0.0, 2 ** -8, 2 ** -6, 1.0]


def test_quantize_rows_error_bound():
    rng = np.random.default_rng(9)
    x = (rng.standard_normal((64, 300)) * np.exp(rng.uniform(-8, 8, (64, 1)))).astype(np.float32)
    x[3] = 0.0
    codes, scale = O.quantize_rows(x)
    deq = O.dequant(codes, scale)
    assert scale[3] == 1.0 and np.all(deq[3] == 0)
    amax = np.abs(x).max(axis=1)
    # the row maximum maps to the largest code
    assert np.all(np.abs(O.e4m3_decode(codes[np.arange(64), np.abs(x).argmax(axis=1)]))[amax > 0] == 448.0)
    # half a quantum of the binade (2^-4 relative), or half the subnormal
    # quantum 2^-10 of the scaled value, plus fp32 rounding of x * inv
    bound = np.maximum(2.0 ** -4 * np.abs(x), 2.0 ** -10 * scale[:, None]) * (1 + 2.0 ** -20)
    assert np.all(np.abs(deq - x) <= bound)


def test_gemm_e4m3_exact_on_representable_operands_and_scale_invariance():
    rng = np.random.default_rng(10)
    # rows whose maximum is 448 * 2^k and all entries e4m3 values times 2^k:
    # quantisation is exact, so the GEMM is the exact product
    grid = O.e4m3_decode(np.arange(0, 126, dtype=np.uint8))
    def rep(shape, k):
        m = rng.choice(grid, size=shape) * rng.choice([-1, 1], size=shape)
        m[:, 0] = 448.0
        return (m * 2.0 ** k).astype(np.float32)
    a = rep((5, 64), -7)
    w = rep((7, 64), -9)
    wq = O.quantize_rows(w)
    assert np.array_equal(O.dequant(*wq), w.astype(np.float64))
    assert np.array_equal(O.gemm_e4m3(a, wq), a.astype(np.float64) @ w.astype(np.float64).T)
    # a power-of-two factor on one weight row moves into its scale only
    w2 = w.copy()
    w2[2] *= 8
    out1, out2 = O.gemm_e4m3(a, wq), O.gemm_e4m3(a, O.quantize_rows(w2))
    assert np.array_equal(out2[:, 2], 8 * out1[:, 2]) and np.array_equal(np.delete(out2, 2, 1), np.delete(out1, 2, 1))


def test_block_fp8_error_follows_the_e4m3_model():
    """Against the exact block, the FP8 block's error is a few percent of the
    block's update (e4m3 keeps 3 mantissa bits: at most 2^-4 relative per
    operand, about 3.6% RMS, so about 5% per GEMM output): between 1% and
    10% of ||out - u||. A swapped or missing scale is off by orders of
    magnitude."""
    rng = np.random.default_rng(11)
    d, heads, T = 256, 2, 16
    std = 1 / np.sqrt(d)   # logits of order one: attention does not amplify q/k errors

    def one():
        s = I.StreamWeights(w_qkv=bits(rng.normal(0, std, (3 * d, d))), b_qkv=bits(rng.normal(0, std, 3 * d)),
                            w_o=bits(rng.normal(0, std, (d, d))), b_o=bits(rng.normal(0, std, d)))
        s.w_1, s.b_1 = bits(rng.normal(0, std, (4 * d, d))), bits(rng.normal(0, std, 4 * d))
        s.w_2, s.b_2 = bits(rng.normal(0, std / 2, (d, 4 * d))), bits(rng.normal(0, std, d))
        return s
    w = I.BlockWeights(txt=one(), img=one())
    ut = bits(rng.standard_normal((T, d)))
    ui = bits(rng.standard_normal((40, d)))
    et, ei = O.block(ut, ui, [0, 40], T, w, heads, True)
    qt, qi = O.block_fp8(ut, ui, [0, 40], T, O.quantize_weights(w), heads, True)
    for got, ref, u in ((qi, ei, ui), (qt, et, ut)):
        delta = ref - O.bf16_to_f32(u).astype(np.float64)
        r = np.linalg.norm(got - ref) / np.linalg.norm(delta)
        assert 0.01 < r < 0.1, r
    # a block with no image rows leaves the text stream's FP8 result alone
    qt0, _ = O.block_fp8(ut, ui[:0], [0, 0], T, O.quantize_weights(w), heads, True)
    assert qt0.shape == qt.shape


def test_block_rows_fp8_matches_block_fp8():
    rng = np.random.default_rng(12)
    d, heads, T = 128, 2, 6
    std = 1 / np.sqrt(d)

    def one():
        s = I.StreamWeights(w_qkv=bits(rng.normal(0, std, (3 * d, d))), b_qkv=bits(rng.normal(0, std, 3 * d)),
                            w_o=bits(rng.normal(0, std, (d, d))), b_o=bits(rng.normal(0, std, d)))
        s.w_1, s.b_1 = bits(rng.normal(0, std, (4 * d, d))), bits(rng.normal(0, std, 4 * d))
        s.w_2, s.b_2 = bits(rng.normal(0, std / 2, (d, 4 * d))), bits(rng.normal(0, std, d))
        return s
    wq = O.quantize_weights(I.BlockWeights(txt=one(), img=one()))
    ut = bits(rng.standard_normal((2 * T, d)))
    ui = bits(rng.standard_normal((23, d)))
    cu = [0, 9, 23]
    ft, fi = O.block_fp8(ut, ui, cu, T, wq, heads, True)
    rt, ri = O.block_rows_fp8(ut, ui, cu, T, wq, heads, True, 1, [6, 11], [9, 15, 22])
    assert np.allclose(rt, ft[[6, 11]], rtol=0, atol=1e-12)
    assert np.allclose(ri, fi[[9, 15, 22]], rtol=0, atol=1e-12)


def _fp8_weights(rng, d):
    std = 1 / np.sqrt(d)

    def one():
        s = I.StreamWeights(w_qkv=bits(rng.normal(0, std, (3 * d, d))), b_qkv=bits(rng.normal(0, std, 3 * d)),
                            w_o=bits(rng.normal(0, std, (d, d))), b_o=bits(rng.normal(0, std, d)))
        s.w_1, s.b_1 = bits(rng.normal(0, std, (4 * d, d))), bits(rng.normal(0, std, 4 * d))
        s.w_2, s.b_2 = bits(rng.normal(0, std / 2, (d, 4 * d))), bits(rng.normal(0, std, d))
        return s
    return O.quantize_weights(I.BlockWeights(txt=one(), img=one()))


def test_block_fp8_proportional_ones_is_plain_fp8_block():
    """Row weights of one add ln 1 = 0 to every logit: the FP8 block with
    proportional attention is then the plain FP8 block, bit for bit."""
    rng = np.random.default_rng(34)
    d, heads, T = 64, 2, 4
    wq = _fp8_weights(rng, d)
    ut = bits(rng.standard_normal((2 * T, d)))
    ui = bits(rng.standard_normal((13, d)))
    cu = [0, 6, 13]
    a = O.block_fp8(ut, ui, cu, T, wq, heads, True)
    b = O.block_fp8(ut, ui, cu, T, wq, heads, True, n_img=np.ones(13, np.float32))
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


def test_block_fp8_proportional_equals_fp8_block_on_duplicated_rows():
    """The FP8 block with row weights n equals the plain FP8 block on the
    sequence where image row r appears n_r times: every row's quantisation
    depends on that row alone, so the copies carry the same codes and the
    softmax over n copies of a key is the weighted one. Checked on the text
    rows and the first copy of each image row, and through block_rows_fp8."""
    rng = np.random.default_rng(35)
    d, heads, T = 64, 2, 3
    wq = _fp8_weights(rng, d)
    ut = bits(rng.standard_normal((2 * T, d)))
    ui = bits(rng.standard_normal((9, d)))
    cu = [0, 5, 9]
    n = np.array([1, 3, 1, 2, 4, 2, 1, 1, 3], dtype=np.float32)
    pt, pi = O.block_fp8(ut, ui, cu, T, wq, heads, True, n_img=n)
    rep = np.repeat(np.arange(9), n.astype(int))
    cu_dup = [0, int(n[:5].sum()), int(n.sum())]
    dt, di = O.block_fp8(ut, ui[rep], cu_dup, T, wq, heads, True)
    first = np.searchsorted(rep, np.arange(9))
    assert np.allclose(pt, dt, rtol=0, atol=1e-9)
    assert np.allclose(pi, di[first], rtol=0, atol=1e-9)
    # the weights matter: the plain FP8 block differs
    qt, qi = O.block_fp8(ut, ui, cu, T, wq, heads, True)
    assert np.abs(qi - pi).max() > 1e-3
    rt, ri = O.block_rows_fp8(ut, ui, cu, T, wq, heads, True, 1, [3, 5], [6, 8], n_img=n)
    assert np.allclose(rt, pt[[3, 5]], rtol=0, atol=1e-12) and np.allclose(ri, pi[[6, 8]], rtol=0, atol=1e-12)


def test_keep_ratio_one_is_dense_block():
    wl = I.tiny_layer(keep_ratio=1024, H=16, W=16, d=64, heads=2, T=8)
    b = I.make_batch(wl)
    w = I.make_weights(wl.d, wl.mlp, seed=1)
    sp, packed, (ot, oi), y = O.hot_path(b.x, b.text, b.mask, [wl.N], b.k_mid, 1, [w], wl.heads, wl.mlp)
    assert np.array_equal(packed, b.x.reshape(wl.N, wl.d))
    dt, di = O.block_dense(b.x, b.text, w, wl.heads, wl.mlp)
    assert np.array_equal(oi, di) and np.array_equal(ot, dt)
    assert np.array_equal(y[0], di)


def test_update_closed_form():
    x = bits(np.array([1.0, -2.0, 0.5]))
    y = np.array([1.0, 0.0, -4.0])
    got = O.bf16_to_f32(O.update(x, y, 0.035))
    want = np.array([1.0 - np.float32(0.035), -2.0, 0.5 + 4 * np.float32(0.035)], dtype=np.float32)
    assert np.array_equal(got, O.bf16_to_f32(I.f32_to_bf16_bits(want)))


def test_weights_f64_same_block():
    rng = np.random.default_rng(12)
    d, heads, T = 32, 2, 3
    w = _rand_weights(rng, d, mlp=True)
    ut = bits(rng.standard_normal((T, d)))
    ui = bits(rng.standard_normal((7, d)))
    a = O.block(ut, ui, [0, 7], T, w, heads, True)
    b = O.block(ut, ui, [0, 7], T, O.weights_f64(w), heads, True)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


# ------------------------------------------------ Sobel selector (Sec. 2.3) --

def _brute_sobel_select(img, mask, H, W, P, R, t):
    """Pixel-by-pixel loops, written independently of the oracle's slicing."""
    B, Hp, Wp, C = img.shape
    keep = np.zeros((B, H * W), dtype=np.uint8)
    for b in range(B):
        def px(y, x, c):
            return np.float32(img[b, min(max(y, 0), Hp - 1), min(max(x, 0), Wp - 1), c])
        g = np.zeros((Hp, Wp), dtype=np.float32)
        for y in range(Hp):
            for x in range(Wp):
                acc = np.float32(0.0)
                for c in range(C):
                    gx = ((px(y - 1, x + 1, c) + np.float32(2) * px(y, x + 1, c)) + px(y + 1, x + 1, c)) - \
                         ((px(y - 1, x - 1, c) + np.float32(2) * px(y, x - 1, c)) + px(y + 1, x - 1, c))
                    gy = ((px(y + 1, x - 1, c) + np.float32(2) * px(y + 1, x, c)) + px(y + 1, x + 1, c)) - \
                         ((px(y - 1, x - 1, c) + np.float32(2) * px(y - 1, x, c)) + px(y - 1, x + 1, c))
                    acc = np.float32(acc + np.float32(np.float32(gx * gx) + np.float32(gy * gy)))
                g[y, x] = np.sqrt(acc)
        gmax = g.max()
        for i in range(H):
            for j in range(W):
                hf = False
                if gmax > 0:
                    hf = np.float32(g[i * P:(i + 1) * P, j * P:(j + 1) * P].max() / gmax) > np.float32(t)
                dil = any(mask[b, ii * W + jj] for ii in range(max(0, i - R), min(H, i + R + 1))
                          for jj in range(max(0, j - R), min(W, j + R + 1)))
                keep[b, i * W + j] = 1 if (hf or dil) else 0
    return keep


@pytest.mark.parametrize("R,t", [(0, 0.1), (1, 0.3), (2, 0.05)])
def test_sobel_select_brute_force(R, t):
    rng = np.random.default_rng(40 + R)
    B, H, W, P, C = 2, 3, 4, 4, 3
    img = rng.random((B, H * P, W * P, C)).astype(np.float32)
    img[:, :, :5] *= 0.1   # a flat-ish region, so the threshold matters
    mask = (rng.random((B, H * W)) < 0.15).astype(np.uint8)
    assert np.array_equal(O.sobel_select(img, mask, H, W, P, R, t), _brute_sobel_select(img, mask, H, W, P, R, t))


def test_sobel_magnitude_matches_scipy_per_channel():
    nd = pytest.importorskip("scipy.ndimage")
    rng = np.random.default_rng(41)
    img = rng.standard_normal((2, 24, 40, 3)).astype(np.float32)
    ref = np.zeros(img.shape[:3])
    for b in range(2):
        acc = 0.0
        for c in range(3):
            a = img[b, :, :, c].astype(np.float64)
            acc = acc + nd.sobel(a, axis=1, mode="nearest") ** 2 + nd.sobel(a, axis=0, mode="nearest") ** 2
        ref[b] = np.sqrt(acc)
    assert np.abs(O.sobel_magnitude(img) - ref).max() <= 1e-6 * ref.max()


def test_sobel_select_constant_image_keeps_only_dilated_mask():
    H, W, P = 4, 5, 8
    img = np.full((1, H * P, W * P, 3), 0.7, dtype=np.float32)
    mask = np.zeros((1, H * W), dtype=np.uint8)
    mask[0, 2 * W + 2] = 1
    keep = O.sobel_select(img, mask, H, W, P, 1, 0.1).reshape(H, W)
    exp = np.zeros((H, W), dtype=np.uint8)
    exp[1:4, 1:4] = 1
    assert np.array_equal(keep, exp)


def test_sobel_select_step_edge_closed_form():
    """A vertical step between pixel columns e-1 and e gives |G| = 4 exactly in
    those two columns and 0 elsewhere (the 3-wide Sobel support), so exactly the
    token columns holding pixel column e-1 or e are selected, in every row."""
    H, W, P = 3, 6, 8
    for e in (8, 13, 40):
        img = np.zeros((1, H * P, W * P, 1), dtype=np.float32)
        img[:, :, e:] = 1.0
        g = O.sobel_magnitude(img)[0]
        assert np.all(g[:, e - 1:e + 1] == 4.0) and np.count_nonzero(g) == 2 * H * P
        keep = O.sobel_select(img, np.zeros((1, H * W), np.uint8), H, W, P, 0, 0.1).reshape(H, W)
        cols = {(e - 1) // P, e // P}
        exp = np.zeros((H, W), dtype=np.uint8)
        exp[:, sorted(cols)] = 1
        assert np.array_equal(keep, exp)


def test_sobel_select_ramp_and_strict_threshold():
    """A ramp P(y, x) = a x has |G| = 8a inside and 4a in the two replicated
    border columns: normalised 1 and 1/2. Every token is selected at t = 0.1 and
    at t = 0.5 (its largest value is 1), none at t = 1 (the test is strict)."""
    H, W, P, a = 2, 3, 4, 0.25
    x = np.arange(W * P, dtype=np.float32) * np.float32(a)
    img = np.broadcast_to(x[None, None, :, None], (1, H * P, W * P, 1)).copy()
    g = O.sobel_magnitude(img)[0]
    assert np.all(g[:, 1:-1] == np.float32(8 * a)) and np.all(g[:, [0, -1]] == np.float32(4 * a))
    z = np.zeros((1, H * W), np.uint8)
    assert O.sobel_select(img, z, H, W, P, 0, 0.1).all()
    assert O.sobel_select(img, z, H, W, P, 0, 0.5).all()
    assert not O.sobel_select(img, z, H, W, P, 0, 1.0).any()


def test_dilate_mask_brute_and_monotone_threshold():
    rng = np.random.default_rng(42)
    H, W = 7, 9
    m = (rng.random((2, H * W)) < 0.1).astype(np.uint8)
    for R in (0, 1, 3):
        d = O.dilate_mask(m, H, W, R).reshape(2, H, W)
        for b in range(2):
            mm = m[b].reshape(H, W)
            for i in range(H):
                for j in range(W):
                    assert d[b, i, j] == int(mm[max(0, i - R):i + R + 1, max(0, j - R):j + R + 1].any())
    assert np.array_equal(O.dilate_mask(m, H, W, 0), m)
    img = rng.random((2, H * 4, W * 4, 3)).astype(np.float32)
    k1 = O.sobel_select(img, m, H, W, 4, 1, 0.2)
    k2 = O.sobel_select(img, m, H, W, 4, 1, 0.4)
    assert np.all(k2 <= k1)
