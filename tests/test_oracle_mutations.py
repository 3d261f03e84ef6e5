"""The oracle's pins catch plausible mistakes.

Each test plants one mistake in the oracle on the CPU: a dropped term, a wrong sign or
boundary, a transposed operand, an off-by-one level count, a wrong constant. It monkeypatches
the oracle function, then runs the pins written for that part of the paper and requires every
one of them to fail. A pin that still passed with the mistake in place would say nothing about
that part. The pins are the functions of the `test_oracle_*.py` files, called directly. Their
modules are imported as modules, so pytest does not collect them here a second time.
"""
import numpy as np
import pytest

import test_oracle_agp as ta
import test_oracle_forward as tf
import test_oracle_gamma as tg
import test_oracle_philox as tp
import test_oracle_quantizer as tq
import test_oracle_worked as tw
from oracle import method as om
from oracle import philox

f32 = np.float32
TWO32 = 1 << 32


def _fails(pin, *args):
    with pytest.raises(AssertionError):
        pin(*args)


# ---------------------------------------------------------------- forward (Sec. 5.1, App. C)
def test_sign_of_zero_as_plus_one_is_caught(monkeypatch):
    """Sec. 5.1's sign gives -1 at 0. Taking x >= 0 as +1 is the usual slip."""
    monkeypatch.setattr(om, "sign", lambda x: np.where(np.asarray(x) >= 0, 1, -1).astype(np.int8))
    _fails(tf.test_sign_definition)
    _fails(tf.test_forward_brute_force)
    _fails(tg.test_colsum_sign_plain_loops)


def test_forward_without_gamma_is_caught(monkeypatch):
    orig = om.forward
    monkeypatch.setattr(om, "forward", lambda x_u, w, gamma: orig(x_u, w, None))
    _fails(tf.test_forward_brute_force)


def test_bias_before_the_scale_is_caught(monkeypatch):
    """Reading R10 adds the bias after Gamma scales the product. Gamma (acc + bias) is the other order."""
    def forward_bias(x_u, w, gamma, bias):
        acc, _ = om.forward(x_u, w, None)
        if bias is None:
            return om.forward(x_u, w, gamma)
        y = (np.asarray(gamma, f32)[None, :] * (acc.astype(f32) + np.asarray(bias, f32)[None, :])).astype(f32)
        return acc, y
    monkeypatch.setattr(om, "forward_bias", forward_bias)
    _fails(tg.test_forward_bias_plain_loops)
    _fails(tf.test_forward_bias_adds_after_the_scale)


def test_scale_gradient_without_the_product_is_caught(monkeypatch):
    orig = om.scale_bias_grad
    monkeypatch.setattr(om, "scale_bias_grad", lambda gy, acc: orig(gy, np.ones_like(acc)))
    _fails(tf.test_scale_bias_grad_matches_autograd)


def test_ste_open_boundary_is_caught(monkeypatch):
    """Reading R10 passes the gradient at |x| = t. A strict < drops it."""
    monkeypatch.setattr(om, "ste_clip", lambda x, dx, t=1.0: np.where(np.abs(np.asarray(x)) < t, dx, 0).astype(
        np.asarray(dx).dtype))
    _fails(tf.test_ste_clip_matches_hardtanh_gradient)


def test_colsum_over_the_wrong_axis_is_caught(monkeypatch):
    monkeypatch.setattr(om, "colsum_sign", lambda a: om.sign(a).astype(np.int64).sum(axis=1))
    _fails(tg.test_colsum_sign_plain_loops)


def test_unfolder_padding_with_plus_one_is_caught(monkeypatch):
    """Reading R1 pads X with zeros, so padded taps have sign -1. Padding with +1 flips them."""
    orig = om.unfold

    def unfold(x, kh, kw, stride, pad):
        xp = np.pad(np.asarray(x, f32), ((0, 0), (0, 0), (pad, pad), (pad, pad)), constant_values=1.0)
        return orig(xp, kh, kw, stride, 0)
    monkeypatch.setattr(om, "unfold", unfold)
    _fails(tf.test_unfold_fold_match_torch, 2, 3, 7, 6, 3, 1, 1)
    _fails(tf.test_conv_forward_pads_as_minus_one)


def test_folder_with_transposed_taps_is_caught(monkeypatch):
    orig = om.fold_int

    def fold_int(acc_u, N, C, H, W, kh, kw, stride, pad):
        a = np.asarray(acc_u).reshape(-1, C, kh, kw).transpose(0, 1, 3, 2).reshape(-1, C * kh * kw)
        return orig(a, N, C, H, W, kh, kw, stride, pad)
    monkeypatch.setattr(om, "fold_int", fold_int)
    _fails(tf.test_unfold_fold_match_torch, 2, 3, 7, 6, 3, 1, 1)
    _fails(tq.test_conv_grad_input_matches_transposed_conv)


def test_folder_ignoring_the_stride_is_caught(monkeypatch):
    def fold_int(acc_u, N, C, H, W, kh, kw, stride, pad):
        Ho, Wo = om.conv_out_hw(H, W, kh, kw, stride, pad)
        a = np.asarray(acc_u, dtype=np.int64).reshape(N, Ho, Wo, C, kh, kw)
        out = np.zeros((N, C, H + 2 * pad, W + 2 * pad), dtype=np.int64)
        for i in range(kh):
            for j in range(kw):
                out[:, :, i:i + Ho, j:j + Wo] += a[:, :, :, :, i, j].transpose(0, 3, 1, 2)  # stride dropped
        return out[:, :, pad:pad + H, pad:pad + W]
    monkeypatch.setattr(om, "fold_int", fold_int)
    _fails(tf.test_unfold_fold_match_torch, 1, 2, 9, 9, 7, 2, 3)
    _fails(tq.test_conv_grad_input_matches_transposed_conv)


def test_implicit_product_padding_with_plus_one_is_caught(monkeypatch):
    orig = om.implicit_conv_acc

    def implicit_conv_acc(x, w, pad):
        xp = np.pad(np.asarray(x, f32), ((0, 0), (0, 0), (pad, pad), (pad, pad)), constant_values=1.0)
        return orig(xp, w, 0)
    monkeypatch.setattr(om, "implicit_conv_acc", implicit_conv_acc)
    _fails(tf.test_implicit_conv_matches_direct_convolution, 2, 3, 4, 5, 3, 3, 1)


def test_channel_major_weight_taps_are_caught(monkeypatch):
    """The implicit product contracts k' = t C + c. A channel-major order is the transposed layout."""
    monkeypatch.setattr(om, "tap_major_signs",
                        lambda w: om.sign(np.asarray(w, f32).reshape(np.asarray(w).shape[0], -1)))
    _fails(tf.test_implicit_conv_matches_direct_convolution, 2, 3, 4, 5, 3, 3, 1)


# ---------------------------------------------------------------- AGP (Sec. 5.2, App. B)
def test_water_filling_without_the_cap_is_caught(monkeypatch):
    """Sec. 5.2 caps p_i at 1 and hands the excess to the other groups. Clipping alone drops budget."""
    orig = om.agp_probabilities

    def agp_probabilities(r, bits, mode=om.SYSTEMATIC):
        if bits == 1 or mode == om.TOPK:
            return orig(r, bits, mode)
        rt = om.fixed_point_ranges(r)
        n, s = len(rt), sum(rt)
        order = sorted(range(n), key=lambda i: (-rt[i], i))
        return [min(TWO32, (n * v * TWO32) // (bits * s)) if s else 0 for v in rt], order
    monkeypatch.setattr(om, "agp_probabilities", agp_probabilities)
    _fails(tw.test_water_filling_with_one_binding_cap)
    _fails(ta.test_water_filling_matches_bisection, 64, 2)


def test_systematic_mask_boundary_is_caught(monkeypatch):
    """A group is kept when [C_i, C_i + P_i) holds a multiple of 2^32. Testing >= keeps every group."""
    orig = om.agp_masks

    def agp_masks(P, seed, stream, mode=om.SYSTEMATIC):
        if mode != om.SYSTEMATIC:
            return orig(P, seed, stream, mode)
        c = int(philox.uniform_u32(seed, stream, np.uint64(0)))
        kept = np.zeros(len(P), dtype=bool)
        for i, p in enumerate(P):
            kept[i] = ((c + p) >> 32) >= (c >> 32)
            c += p
        return kept
    monkeypatch.setattr(om, "agp_masks", agp_masks)
    _fails(tw.test_no_cap_probabilities_and_systematic_masks_by_hand)
    _fails(ta.test_mask_inclusion_frequencies, om.SYSTEMATIC)


def test_topk_keeping_the_smallest_is_caught(monkeypatch):
    orig = om.agp_probabilities

    def agp_probabilities(r, bits, mode=om.SYSTEMATIC):
        P, order = orig(r, bits, mode)
        if mode != om.TOPK or bits == 1:
            return P, order
        k = max(1, len(P) // bits)
        Q = [0] * len(P)
        for i in order[-k:]:
            Q[i] = TWO32
        return Q, order
    monkeypatch.setattr(om, "agp_probabilities", agp_probabilities)
    _fails(ta.test_topk_keeps_largest)


def test_gamma_left_out_of_the_quantized_gradient_is_caught(monkeypatch):
    """Reading R2 quantizes G = gY (.) Gamma. Quantizing gY itself drops the pre-scale."""
    monkeypatch.setattr(om, "grad_to_quantize", lambda gy, gamma: np.asarray(gy, f32).copy())
    _fails(tg.test_grad_to_quantize_is_per_channel)


# ---------------------------------------------------------------- stochastic rounding (Sec. 3.2)
def test_round_to_nearest_is_caught(monkeypatch):
    """Sec. 3.2 rounds stochastically. Nearest rounding is biased."""
    def sr_codes(x, z, r, bits, seed, stream, flat_index):
        B = f32((1 << bits) - 1)
        with np.errstate(divide="ignore", invalid="ignore"):
            t = ((np.asarray(x, f32) - f32(z)).astype(f32) * (B / np.asarray(r, f32)).astype(f32)).astype(f32)
        q = np.clip(np.floor(t + f32(0.5)), f32(0), B)
        return np.where(np.isfinite(q), q, 0).astype(np.int64)
    monkeypatch.setattr(om, "sr_codes", sr_codes)
    _fails(tq.test_sr_unbiased_and_variance)
    _fails(tw.test_stochastic_rounding_thresholds_by_hand)


def test_levels_off_by_one_are_caught(monkeypatch):
    """B = 2^b - 1 levels above zero. Scaling by 2^b instead shifts every code."""
    orig = om.sr_codes

    def sr_codes(x, z, r, bits, seed, stream, flat_index):
        B = (1 << bits) - 1
        return orig(x, z, (np.asarray(r, f32) * f32(B / (B + 1))).astype(f32), bits, seed, stream, flat_index)
    monkeypatch.setattr(om, "sr_codes", sr_codes)
    _fails(tq.test_sr_unbiased_and_variance)
    _fails(tw.test_stochastic_rounding_thresholds_by_hand)


def test_philox_key_bump_is_caught(monkeypatch):
    """A wrong Weyl constant still gives uniform-looking words, but not Philox4x32-10's. Only the
    comparison with Triton's independent generator can see it: the other pins draw their
    expected words from the same generator."""
    pytest.importorskip("triton")
    monkeypatch.setattr(philox, "_W1", 0xBB67AE87)
    _fails(tp.test_philox_matches_triton_interpreter)


# ---------------------------------------------------------------- SCQ rescale and products (Sec. 5.2-5.3)
def test_rescale_without_the_keep_probability_is_caught(monkeypatch):
    """M = diag(m / p) divides kept groups by p. Dropping it biases the pruned estimate."""
    orig = om.group_scale
    monkeypatch.setattr(om, "group_scale",
                        lambda r, z, p_hat, bits: orig(r, z, np.ones(len(np.atleast_1d(p_hat))), bits))
    _fails(tw.test_rescale_of_a_kept_group_by_hand)
    _fails(tq.test_agp_quantizer_unbiased, 0)


def test_scale_over_two_to_the_b_is_caught(monkeypatch):
    orig = om.group_scale

    def group_scale(r, z, p_hat, bits):
        s, zz = orig(r, z, p_hat, bits)
        B = (1 << bits) - 1
        return (s.astype(np.float64) * B / (B + 1)).astype(f32), zz
    monkeypatch.setattr(om, "group_scale", group_scale)
    _fails(tw.test_rescale_of_a_kept_group_by_hand)


def test_dequantization_without_the_zero_point_term_is_caught(monkeypatch):
    """Eq. 21 with SCQ: out = S' acc + Z' colsum. Dropping the colsum term loses the zero point."""
    orig = om.dequant
    monkeypatch.setattr(om, "dequant", lambda scale, acc, zero, colsum: orig(scale, acc, np.zeros_like(
        np.asarray(zero, f32)), colsum))
    _fails(tq.test_scq_factoring_and_bit_planes)


def test_bit_planes_in_reverse_order_are_caught(monkeypatch):
    orig = om.bit_planes
    monkeypatch.setattr(om, "bit_planes", lambda codes, bits: orig(codes, bits)[::-1])
    _fails(tq.test_scq_factoring_and_bit_planes)
