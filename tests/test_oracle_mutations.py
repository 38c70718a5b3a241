"""The oracle's pins catch plausible mistakes.

Each case plants one mistake in the oracle (on the CPU, through monkeypatch:
the module's own helper is replaced by a wrong version) and runs the pins
that should notice it. At least one of them must fail, which shows that the
pins constrain that part of the oracle and do not just restate it:
- a wrong tie-break, a flipped ranking and a transposed grid in the selection;
- a wrong variance, a wrong GELU and a wrong softmax scale in the block;
- a dropped value operand, and the row-size bias put on queries instead of keys;
- square weights read transposed, the wrong pooling window, a different
  summation order of a window's members, a wrong e4m3 exponent bias and row
  sizes off by one;
- a delta unpool without the member's own value, e4m3 overflow to NaN, the
  Sobel energy for its magnitude and a mask dilated one token short;
- bf16 by truncation, the update's sign, e4m3 scales on the wrong axis, an
  FP8 GEMM without its weight scale, an inclusive selector threshold and an
  unpack that reads the next row.
"""
import math

import numpy as np
import pytest

from oracle import hilo_oracle as O
from tests import test_oracle_pins as P

_ranking, _layer_norm, _softmax, _bf16 = O.ranking, O.layer_norm, O.softmax_attention, O.bf16_to_f32
_w, _members, _decode, _row_sizes = O._w, O.window_members, O.e4m3_decode, O.row_sizes
_delta, _encode, _sobel, _dilate = O.unpack_delta, O.e4m3_encode, O.sobel_magnitude, O.dilate_mask
_update, _select = O.update, O.sobel_select


def ranking_ties_high_index(s):
    return np.lexsort((-np.arange(s.shape[0]), -s.astype(np.float64)))


def ranking_ascending(s):
    return np.lexsort((np.arange(s.shape[0]), s.astype(np.float64)))


def bf16_grid_transposed(bits):
    x = _bf16(bits)
    return np.ascontiguousarray(np.swapaxes(x, 1, 2)) if x.ndim == 4 else x


def layer_norm_unbiased(u, eps=1e-6):
    mu = u.mean(axis=-1, keepdims=True)
    var = ((u - mu) ** 2).sum(axis=-1, keepdims=True) / (u.shape[-1] - 1)
    return (u - mu) / np.sqrt(var + eps)


def gelu_sigmoid(z):
    # a different GELU approximation, z * sigmoid(1.702 z)
    return z / (1.0 + np.exp(-1.702 * z))


def softmax_scale_by_dim(q, k, v, key_n=None):
    return _softmax(q / math.sqrt(q.shape[-1]), k, v, key_n)


def softmax_values_are_keys(q, k, v, key_n=None):
    return _softmax(q, k, k, key_n)


def softmax_weights_on_queries(q, k, v, key_n=None):
    if key_n is None:
        return _softmax(q, k, v)
    sc = (q @ k.T) / math.sqrt(q.shape[-1])
    n = np.asarray(key_n, dtype=np.float64)
    if n.shape[0] == sc.shape[0]:
        sc = sc + np.log(n)[:, None]
    sc = sc - sc.max(axis=-1, keepdims=True)
    p = np.exp(sc)
    return (p / p.sum(axis=-1, keepdims=True)) @ v


def weights_square_transposed(bits):
    # W read as W^T where the shapes allow it unnoticed (the d x d matrices)
    w = _w(bits)
    return w.T if w.ndim == 2 and w.shape[0] == w.shape[1] else w


def members_column_major(w, size, W):
    # the window's members in column-major instead of raster order
    m = _members(w, size, W)
    return [m[j * size + i] for i in range(size) for j in range(size)]


def members_next_window(w, size, W):
    n = (W // size)
    return _members(w + 1 if (w + 1) % n else w - 1, size, W)


def decode_exponent_bias_off(c):
    return _decode(c) * 2.0


def row_sizes_plus_one(sp):
    return _row_sizes(sp) + np.float32(1.0)


def delta_without_own_value(out_img, packed_bits, x_bits, sp):
    # a pooled member gets the window's update but not its own value back
    return _delta(out_img, packed_bits, np.zeros_like(x_bits), sp)


def encode_no_saturation(t):
    # magnitudes beyond 448 become NaN codes instead of saturating
    c = _encode(t).copy()
    big = np.abs(np.asarray(t, dtype=np.float64)) > 448.0
    c[big] = (c[big] & 0x80) | 0x7F
    return c


def sobel_squared_magnitude(img):
    # the gradient energy instead of its magnitude (square root dropped)
    return _sobel(img) ** 2


def dilate_one_short(mask, H, W, radius):
    return _dilate(mask, H, W, max(0, radius - 1))


def bf16_truncating(a):
    # fp32 -> bf16 by dropping the low half instead of rounding to nearest even
    return (np.ascontiguousarray(a, dtype=np.float32).view(np.uint32) >> np.uint32(16)).astype(np.uint16)


def update_sign_flipped(x_bits, y, alpha):
    return _update(x_bits, y, -alpha)


def dequant_scale_on_columns(codes, scale):
    return O.e4m3_decode(codes) * np.asarray(scale, np.float64)[None, :]


def gemm_e4m3_without_weight_scale(a64, wq, bias=None):
    ca, sa = O.quantize_rows(np.asarray(a64, dtype=np.float32))
    cw, _ = wq
    out = (O.e4m3_decode(ca) @ O.e4m3_decode(cw).T) * sa.astype(np.float64)[:, None]
    return out if bias is None else out + O._w(bias)


def select_inclusive_threshold(img, mask, H, W, patch, radius, threshold):
    # ">=" instead of the strict ">"
    return _select(img, mask, H, W, patch, radius, float(np.nextafter(np.float32(threshold), np.float32(-1))))


def unpack_next_row(out_img, sp):
    return out_img[np.minimum(sp.tok_row + 1, out_img.shape[0] - 1)]


def _brute_force_split():
    for seed in range(6):
        for levels in (1, 2):
            P.test_split_brute_force(seed, levels)


def _block_brute_force():
    for grid, mlp in (((4, 4), True), ((8, 8), False)):
        P.test_block_brute_force_tiny(grid, mlp)


def _row_sizes_pins():
    for granular in (False, True):
        P.test_row_sizes_count_the_grid(granular)


def _delta_pins():
    for granular in (False, True):
        P.test_unpack_delta_identity_block_returns_x(granular)


def _hand_worked_splits():
    for case in P._golden_cases():
        P.test_split_hand_worked(case)


MUTATIONS = {
    "tie-break by the highest index": ("ranking", ranking_ties_high_index,
                                       [P.test_split_ties_take_lowest_indices, _brute_force_split]),
    "lowest scores kept": ("ranking", ranking_ascending, [_hand_worked_splits, _brute_force_split]),
    "grid read transposed": ("bf16_to_f32", bf16_grid_transposed,
                             [P.test_score_linear_ramp_closed_form, P.test_score_single_token_delta_position]),
    "unbiased variance in LayerNorm": ("layer_norm", layer_norm_unbiased,
                                       [P.test_layer_norm_and_gelu_closed_forms]),
    "sigmoid GELU": ("gelu_tanh", gelu_sigmoid, [P.test_layer_norm_and_gelu_closed_forms]),
    "logits scaled by 1/d": ("softmax_attention", softmax_scale_by_dim,
                             [P.test_attention_two_token_closed_form, P.test_attention_scale_closed_form]),
    "keys used as values": ("softmax_attention", softmax_values_are_keys,
                            [P.test_attention_two_token_closed_form, P.test_block_uniform_attention_closed_form]),
    "row sizes on the queries": ("softmax_attention", softmax_weights_on_queries,
                                 [P.test_proportional_attention_equals_duplicated_keys]),
    "square weights transposed": ("_w", weights_square_transposed,
                                  [P.test_block_uniform_attention_closed_form, _block_brute_force]),
    "pooled window of the neighbour": ("window_members", members_next_window,
                                       [P.test_pack_constant_windows_lossless,
                                        P.test_unpack_pack_identity_on_kept_rows_and_brute_mean]),
    "pooled members summed column-major": ("window_members", members_column_major,
                                           [P.test_unpack_pack_identity_on_kept_rows_and_brute_mean,
                                            P.test_pack_sums_members_in_raster_order]),
    "e4m3 exponent bias off by one": ("e4m3_decode", decode_exponent_bias_off,
                                      [P.test_e4m3_codes_roundtrip_and_match_torch]),
    "row sizes off by one": ("row_sizes", row_sizes_plus_one, [_row_sizes_pins]),
    "delta unpool drops the member's own value": ("unpack_delta", delta_without_own_value, [_delta_pins]),
    "e4m3 overflow to NaN instead of saturation": ("e4m3_encode", encode_no_saturation,
                                                   [P.test_e4m3_ties_saturation_subnormals]),
    "Sobel energy instead of magnitude": ("sobel_magnitude", sobel_squared_magnitude,
                                          [P.test_sobel_magnitude_matches_scipy_per_channel]),
    "mask dilated one token short": ("dilate_mask", dilate_one_short,
                                     [P.test_dilate_mask_brute_and_monotone_threshold]),
    "bf16 by truncation": ("f32_to_bf16", bf16_truncating,
                           [P.test_bf16_rounding_matches_torch, P.test_update_closed_form]),
    "update adds instead of subtracting": ("update", update_sign_flipped, [P.test_update_closed_form]),
    "e4m3 scales broadcast over columns": ("dequant", dequant_scale_on_columns,
                                          [P.test_quantize_rows_error_bound,
                                           P.test_gemm_e4m3_exact_on_representable_operands_and_scale_invariance]),
    "FP8 GEMM without the weight scale": ("gemm_e4m3", gemm_e4m3_without_weight_scale,
                                          [P.test_gemm_e4m3_exact_on_representable_operands_and_scale_invariance]),
    "selector threshold inclusive": ("sobel_select", select_inclusive_threshold,
                                     [P.test_sobel_select_ramp_and_strict_threshold]),
    "unpack reads the next row": ("unpack", unpack_next_row,
                                  [P.test_pack_constant_windows_lossless,
                                   P.test_unpack_pack_identity_on_kept_rows_and_brute_mean]),
}


def test_unmutated_pins_pass():
    for _, _, pins in MUTATIONS.values():
        for pin in pins:
            pin()


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, monkeypatch):
    attr, wrong, pins = MUTATIONS[name]
    monkeypatch.setattr(O, attr, wrong)
    caught = []
    for pin in pins:
        try:
            pin()
        except Exception:  # an assertion, or a shape or index error the mistake causes
            caught.append(pin.__name__)
    assert caught, f"no pin noticed: {name}"
