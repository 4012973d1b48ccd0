"""Mistakes planted in the oracle, on the CPU, must fail the pins.

Each case replaces one oracle function by a copy with one plausible mistake
(a truncating shift, the flip before the shift, a dropped term, no bias, no
saturation or a saturation before the bias, a left shift, a true convolution
instead of cross-correlation, a truncating average, a max-pool that pads with
zeros, a residual join with the ReLU first or with wraparound, a swapped
nibble, a wrong column constant, a wrong term sign, a quantizer that floors
log2|W| or rounds in the linear domain, a truncating Q16.16 conversion or one
with ties away from zero, an input gradient without the rot180 or with the
flip first, sampled-element and layout helpers with one slip each, an int32
bound that drops a term, a ResNet block joined after its ReLU, a 5-bit code
with the signs swapped or its shift off by one, 5-bit planes in reverse
order) and runs the
pins of tests/test_oracle_pins.py until one fails.  A
mistake that no pin catches fails this test.  The unmutated oracle passes every
pin (test_oracle_pins.py itself).
"""
import numpy as np
import pytest

import test_codes5_cpu as pins5
import test_oracle_pins as pins
from oracle import deepshift_oracle as O
from oracle import networks as ON

_ORIG = {name: getattr(O, name) for name in ("linear_shift_acc", "conv2d_shift_acc", "sat32", "avgpool_floor",
                                              "pack_planes6", "column_constants", "term", "shift",
                                              "quantize_weights", "quantize_activations",
                                              "conv2d_shift_backward_x_acc", "linear_shift_backward_x_acc",
                                              "maxpool2d", "conv2d_shift_at", "linear_shift_at",
                                              "int32_accumulation_is_exact", "expand_codes", "weights_bf16_bits",
                                              "unpack_planes6", "backward_codes", "backward_phase_codes",
                                              "code5", "pack_codes5")}

# the pins to run, cheapest first (parametrized pins with their first case)
_PINS = [
    pins.test_term_golden_cases,
    pins.test_linear_golden_cases,
    pins.test_conv_golden_cases,
    pins.test_avgpool_floor_golden_and_library,
    pins.test_pack_golden_tiny_blob,
    pins.test_column_constants_closed_forms,
    pins.test_linear_saturation_boundaries,
    pins.test_linear_trivial_weights,
    pins.test_linear_negation_invariance,
    pins.test_linear_exact_float64_when_x_multiple_of_2_15,
    pins.test_linear_ternary_p0_is_int_matmul,
    pins.test_term_exhaustive_codes_vs_rational_floor_and_bit_strings,
    pins.test_linear_brute_force_tiny,
    pins.test_conv_identity_and_sampled_elements,
    pins.test_conv_negation_invariance,
    lambda: pins.test_conv_exact_float64_when_x_multiple_of_2_15((2, 3, 7, 6, 4, 3, 3, 1, 1, 1, 1)),
    lambda: pins.test_conv_equals_im2col_plus_linear((2, 3, 6, 5, 4, 3, 3, 1, 1, 1, 1)),
    pins.test_quantize_weights_powers_of_two_are_fixed_points,
    pins.test_quantize_weights_against_exact_rationals,
    pins.test_quantize_activations_ties_saturation_and_specials,
    pins.test_quantize_activations_against_exact_rationals_and_torch_round,
    pins.test_linear_backward_x_equals_float64_matmul_on_exact_inputs,
    lambda: pins.test_conv_backward_x_equals_float64_autograd_on_exact_inputs(pins.BWD_GEOMS[0]),
    lambda: pins.test_conv_backward_x_equals_float64_autograd_on_exact_inputs(pins.BWD_GEOMS[1]),
    pins.test_linear_backward_x_is_forward_with_transposed_codes,
    lambda: pins.test_conv_backward_x_brute_force_gather_with_floor(pins.BWD_GEOMS[0]),
    pins.test_maxpool_golden_and_library,
    pins.test_add_relu_golden,
    pins.test_accumulation_bound_is_sound_at_the_int32_edge,
    pins.test_expand_layout_closed_form,
    pins.test_bf16_weight_bits_decode_to_s_times_power_of_two,
    pins.test_pack_round_trip_and_sizes,
    lambda: pins.test_conv_backward_x_stride1_is_forward_conv_with_rot180_codes(pins.BWD_GEOMS[0]),
    lambda: pins.test_conv_backward_x_phase_decomposition(pins.BWD_GEOMS[1]),
    lambda: pins.test_resnet_chain_matches_float64_library_case("resnet18", "basic", [2, 2, 2, 2]),
    pins5.test_every_state_has_a_distinct_code_and_reads_back,
    pins5.test_hand_written_blob,
    pins5.test_round_trip_of_random_codes,
]


def _linear_acc(rule, drop_last=False, use_bias=True):
    """LinearShift accumulator with the per-term rule rule(x_col, s_col, p_col) -> [M, N] terms."""
    def acc_fn(x, s, p, b=None):
        x = np.asarray(x, dtype=np.int64)
        s = np.asarray(s, dtype=np.int64)
        p = np.asarray(p, dtype=np.int64)
        M, K = x.shape
        acc = np.zeros((M, s.shape[0]), dtype=np.int64)
        if b is not None and use_bias:
            acc += np.asarray(b, dtype=np.int64)[None, :]
        for k in range(K - 1 if drop_last and K > 1 else K):
            acc += rule(x[:, k][:, None], s[:, k][None, :], p[:, k][None, :])
        return acc
    return acc_fn


def _floor_rule(x, s, p):
    return s * np.floor_divide(x, np.left_shift(np.int64(1), -p))


def _trunc_rule(x, s, p):  # division rounding toward zero
    d = np.left_shift(np.int64(1), -p)
    return s * (np.sign(x) * (np.abs(x) // d))


def _flip_first_rule(x, s, p):  # (s * x) >> -p
    return np.floor_divide(s * x, np.left_shift(np.int64(1), -p))


def _left_shift_rule(x, s, p):  # x << -p
    return s * (x * np.left_shift(np.int64(1), -p))


def _true_convolution(x, s, p, b=None, stride=(1, 1), pad=(0, 0)):
    s = np.asarray(s)[:, :, ::-1, ::-1]
    p = np.asarray(p)[:, :, ::-1, ::-1]
    return _ORIG["conv2d_shift_acc"](x, s, p, b, stride, pad)


def _conv_without_bias(x, s, p, b=None, stride=(1, 1), pad=(0, 0)):
    return _ORIG["conv2d_shift_acc"](x, s, p, None, stride, pad)


def _trunc_average(x, k, stride):
    x = np.asarray(x, dtype=np.int64)
    N, C, H, W = x.shape
    OH, OW = (H - k) // stride + 1, (W - k) // stride + 1
    out = np.zeros((N, C, OH, OW), dtype=np.int64)
    for oh in range(OH):
        for ow in range(OW):
            sm = x[:, :, oh * stride:oh * stride + k, ow * stride:ow * stride + k].sum(axis=(2, 3))
            out[:, :, oh, ow] = np.sign(sm) * (np.abs(sm) // (k * k))
    return out.astype(np.int32)


def _swapped_nibbles(s, p):
    blob = _ORIG["pack_planes6"](s, p).copy()
    L = O.blob_layout(*np.shape(s))
    nib = blob[L["nib"]:L["bits"]]
    blob[L["nib"]:L["bits"]] = ((nib & 0x0F) << 4) | (nib >> 4)  # the two nibbles of each byte swapped
    return blob


def _wrong_column_a(s, p):
    A, nnz = _ORIG["column_constants"](s, p)
    s2 = np.asarray(s, dtype=np.int64).reshape(np.shape(s)[0], -1)
    p2 = np.asarray(p, dtype=np.int64).reshape(np.shape(p)[0], -1)
    A = (np.abs(s2) * np.left_shift(np.int64(1), 14 + p2)).sum(axis=1)  # 2^(14 + p) instead of 2^(15 + p)
    return A.astype(np.int64), nnz


def _floor_log2_quantizer(W, p_min=O.P_MIN):  # floor(log2|W|) instead of round
    s, p = _ORIG["quantize_weights"](W, p_min)
    w = np.abs(np.asarray(W, dtype=np.float32).astype(np.float64))
    ok = np.isfinite(w) & (w > 0)
    _, e = np.frexp(np.where(ok, w, 1.0))
    p2 = np.where(ok, np.clip(e.astype(np.int64) - 1, p_min, 0), p)
    return s, p2.astype(np.int8)


def _truncating_q16(x):  # x * 2^16 truncated toward zero instead of rounded half to even
    y = np.asarray(x, dtype=np.float32).astype(np.float64) * 65536.0
    y = np.where(np.isnan(y), 0.0, np.trunc(y))
    return np.clip(y, O.INT32_MIN, O.INT32_MAX).astype(np.int64).astype(np.int32)


def _backward_without_rot180(dy, s, p, in_hw, stride=(1, 1), pad=(0, 0)):
    s = np.asarray(s)[:, :, ::-1, ::-1]
    p = np.asarray(p)[:, :, ::-1, ::-1]
    return _ORIG["conv2d_shift_backward_x_acc"](dy, s, p, in_hw, stride, pad)


def _linear_backward_flip_first(dy, s, p):  # (s * dy) >> -p
    dy = np.asarray(dy, dtype=np.int64)
    s = np.asarray(s, dtype=np.int64)
    p = np.asarray(p, dtype=np.int64)
    acc = np.zeros((dy.shape[0], s.shape[1]), dtype=np.int64)
    for n in range(s.shape[0]):
        acc += np.floor_divide(s[n][None, :] * dy[:, n][:, None], np.left_shift(np.int64(1), -p[n])[None, :])
    return acc


def _maxpool_zero_padding(x, k, stride, pad):  # padded taps read as 0 instead of being ignored
    x = np.pad(np.asarray(x, dtype=np.int64), ((0, 0), (0, 0), (pad, pad), (pad, pad)))
    return _ORIG["maxpool2d"](x, k, stride, 0)


def _relu_before_join(a, b):  # ReLU(a) + b, nothing after the join
    return O.sat32(np.maximum(np.asarray(a, np.int64), 0) + np.asarray(b, np.int64)).astype(np.int32)


def _wrapping_join(a, b):  # int32 wraparound instead of saturation
    v = (np.asarray(a, np.int64) + np.asarray(b, np.int64) + (1 << 31)) % (1 << 32) - (1 << 31)
    return np.maximum(v, 0).astype(np.int32)


def _saturate_before_bias(x, s, p, b=None, relu=False):  # sat32(sat32(sum) + b) instead of one saturation
    y = np.asarray(O.sat32(O.linear_shift_acc(x, s, p, None)), np.int64)
    if b is not None:
        y = O.sat32(y + np.asarray(b, np.int64)[None, :])
    y = np.maximum(y, 0) if relu else y
    return np.asarray(y).astype(np.int32)


def _quantizer_rounds_linearly(W, p_min=O.P_MIN):  # nearest power of two by |W - 2^n|, not round(log2|W|)
    s, p = _ORIG["quantize_weights"](W, p_min)
    w = np.abs(np.asarray(W, dtype=np.float32).astype(np.float64))
    ok = np.isfinite(w) & (w > 0)
    m, e = np.frexp(np.where(ok, w, 1.0))  # w between 2^(e-1) and 2^e; their midpoint is at m = 3/4
    p2 = np.where(ok, np.clip(e.astype(np.int64) - 1 + (m >= 0.75), p_min, 0), p)
    return s, p2.astype(np.int8)


def _q16_ties_away(x):  # ties rounded away from zero instead of to even
    y = np.asarray(x, dtype=np.float32).astype(np.float64) * 65536.0
    y = np.where(np.isnan(y), 0.0, np.sign(y) * np.floor(np.abs(y) + 0.5))
    return np.clip(y, O.INT32_MIN, O.INT32_MAX).astype(np.int64).astype(np.int32)


def _expand_halves_swapped(s, p):  # signs in words 0..31, shifts in 32..63
    e = _ORIG["expand_codes"](s, p)
    return np.ascontiguousarray(np.concatenate([e[..., 32:], e[..., :32]], axis=-1))


def _bf16_exponent_off_by_one(s, p):  # exponent 128 + p
    bits = _ORIG["weights_bf16_bits"](s, p).astype(np.int64)
    return np.where(bits != 0, bits + (1 << 7), 0).astype(np.uint16)


def _unpack_without_sign_plane(blob, n_out, k_red):
    s, p = _ORIG["unpack_planes6"](blob, n_out, k_red)
    return np.abs(s).astype(np.int8), p


def _backward_codes_without_rot180(s, p):  # channels swapped, taps not rotated
    sb, pb = _ORIG["backward_codes"](s, p)
    return np.ascontiguousarray(sb[:, :, ::-1, ::-1]), np.ascontiguousarray(pb[:, :, ::-1, ::-1])


def _phase_codes_without_rot180(s, p, stride):
    out = _ORIG["backward_phase_codes"](s, p, stride)
    return {key: None if v is None else tuple(np.ascontiguousarray(a[:, :, ::-1, ::-1]) for a in v)
            for key, v in out.items()}


def _join_after_relu(x, prm, stride, pad, relu, residual=None):  # ReLU on the branch, then a plain join
    s, p, b = prm
    y = O.conv2d_shift(x, s, p, b, (stride, stride), (pad, pad), relu=relu or residual is not None)
    if residual is not None:
        return O.sat32(y.astype(np.int64) + np.asarray(residual, np.int64)).astype(np.int32)
    return y


def _code5_signs_swapped(s, p):  # +1 weights numbered from 16, -1 weights from 1
    c = _ORIG["code5"](s, p)
    return c if c == 0 else (c + 15 if c <= 15 else c - 15)


def _pack5_planes_reversed(s, p):  # bit b of a code stored in plane 4 - b
    blob = _ORIG["pack_codes5"](s, p).copy()
    n_out, k_red = np.shape(s)
    L = O.codes5_layout(n_out, k_red)
    end = L["planes"] + n_out * L["n_chunks"] * 20
    rec = blob[L["planes"]:end].view(np.uint32).reshape(-1, 5)
    blob[L["planes"]:end] = np.ascontiguousarray(rec[:, ::-1]).view(np.uint8).reshape(-1)
    return blob


MUTANTS = {  # each case patches exactly one oracle function ("networks." names one in oracle/networks.py)
    "max-pool pads with zeros": {"maxpool2d": _maxpool_zero_padding},
    "ReLU before the residual join": {"add_relu": _relu_before_join},
    "residual join wraps": {"add_relu": _wrapping_join},
    "saturation before the bias": {"linear_shift": _saturate_before_bias},
    "sampled conv element shifted by the pad": {
        "conv2d_shift_at": lambda x, s, p, b, stride, pad, n, k, oh, ow:
            _ORIG["conv2d_shift_at"](x, s, p, b, stride, (-pad[0], -pad[1]), n, k, oh, ow)},
    "sampled FC element without bias": {
        "linear_shift_at": lambda x, s, p, b, m, n: _ORIG["linear_shift_at"](x, s, p, None, m, n)},
    "int32 bound without nnz": {
        "int32_accumulation_is_exact": lambda amax, A, nnz, babs:
            _ORIG["int32_accumulation_is_exact"](amax, A, 0, babs)},
    "int32 bound without the bias": {
        "int32_accumulation_is_exact": lambda amax, A, nnz, babs:
            _ORIG["int32_accumulation_is_exact"](amax, A, nnz, 0)},
    "quantizer rounds in the linear domain": {"quantize_weights": _quantizer_rounds_linearly},
    "Q16.16 ties away from zero": {"quantize_activations": _q16_ties_away},
    "expanded layout halves swapped": {"expand_codes": _expand_halves_swapped},
    "bf16 exponent off by one": {"weights_bf16_bits": _bf16_exponent_off_by_one},
    "unpack ignores the sign plane": {"unpack_planes6": _unpack_without_sign_plane},
    "input-gradient codes without rot180": {"backward_codes": _backward_codes_without_rot180},
    "phase codes without rot180": {"backward_phase_codes": _phase_codes_without_rot180},
    "ResNet joins after the ReLU": {"networks._conv": _join_after_relu},
    "quantizer floors log2": {"quantize_weights": _floor_log2_quantizer},
    "Q16.16 truncates": {"quantize_activations": _truncating_q16},
    "input gradient without rot180": {"conv2d_shift_backward_x_acc": _backward_without_rot180},
    "input gradient flips first (FC)": {"linear_shift_backward_x_acc": _linear_backward_flip_first},
    "truncating shift (term)": {"shift": lambda x, p: int(np.sign(x)) * (abs(x) >> (-p))},
    "truncating shift (LinearShift)": {"linear_shift_acc": _linear_acc(_trunc_rule)},
    "flip before shift (term)": {"term": lambda x, s, p: (s * x) // (1 << (-p))},
    "flip before shift (LinearShift)": {"linear_shift_acc": _linear_acc(_flip_first_rule)},
    "left shift (term)": {"shift": lambda x, p: x << (-p)},
    "left shift (LinearShift)": {"linear_shift_acc": _linear_acc(_left_shift_rule)},
    "wrong term sign (term)": {"term": lambda x, s, p: -s * (x // (1 << (-p)))},
    "wrong term sign (LinearShift)": {"linear_shift_acc": _linear_acc(lambda x, s, p: -_floor_rule(x, s, p))},
    "dropped term (LinearShift)": {"linear_shift_acc": _linear_acc(_floor_rule, drop_last=True)},
    "no bias (LinearShift)": {"linear_shift_acc": _linear_acc(_floor_rule, use_bias=False)},
    "no bias (ConvShift)": {"conv2d_shift_acc": _conv_without_bias},
    "true convolution (ConvShift)": {"conv2d_shift_acc": _true_convolution},
    "no saturation": {"sat32": lambda v: np.asarray(v)},
    "truncating average": {"avgpool_floor": _trunc_average},
    "swapped nibbles (packing)": {"pack_planes6": _swapped_nibbles},
    "wrong column constant": {"column_constants": _wrong_column_a},
    "5-bit codes with the signs swapped": {"code5": _code5_signs_swapped},
    "5-bit code off by one in the shift": {"code5": lambda s, p: _ORIG["code5"](s, p) + (1 if s != 0 else 0)},
    "5-bit planes in reverse order": {"pack_codes5": _pack5_planes_reversed},
}


@pytest.mark.parametrize("name", list(MUTANTS))
def test_planted_mistake_is_caught(name, monkeypatch):
    for fn_name, fn in MUTANTS[name].items():
        if fn_name.startswith("networks."):
            monkeypatch.setattr(ON, fn_name.split(".", 1)[1], fn)
        else:
            monkeypatch.setattr(O, fn_name, fn)
    caught = []
    for pin in _PINS:
        try:
            pin()
        except (AssertionError, ValueError, IndexError) as e:
            caught.append((getattr(pin, "__name__", "pin"), type(e).__name__))
            break
    assert caught, f"no pin caught the planted mistake: {name}"


def test_control_correct_rewrite_passes_every_pin(monkeypatch):
    """The harness itself: a correct restatement put in through the same plumbing fails no pin."""
    monkeypatch.setattr(O, "linear_shift_acc", _linear_acc(_floor_rule))
    monkeypatch.setattr(O, "conv2d_shift_acc", lambda x, s, p, b=None, stride=(1, 1), pad=(0, 0):
                        _ORIG["conv2d_shift_acc"](x, s, p, b, stride, pad))
    for pin in _PINS:
        pin()
