"""Pins of the oracle's Gamma path, column sums and forward bias against things other than
their own formulas (Sec. 5.1 y = acc (.) Gamma; Eq. 21 with Sec. 5.3's scales; reading R2).

The backward quantizes G = gY (.) Gamma (reading R2).  Because AGP + SR is unbiased (Sec. 5.2),
the mean over many seeds of the oracle's grad_input and grad_weight must converge to the
exact chain-rule gradients of y = Gamma (.) (sign(X) sign(W)^T) with the identity STE, which
torch autograd computes here in float64.  A Gamma on the wrong axis, a missing Gamma or a
Gamma applied twice moves that limit, and the same statistical check rejects each of them.
"""
import numpy as np
import pytest
import torch

from oracle import method as om

f32 = np.float32


def _stats(samples):
    s = np.stack(samples).astype(np.float64)
    return s.mean(axis=0), s.std(axis=0) / np.sqrt(s.shape[0])


def _within(mean, se, ref, slack):
    """Every element of the sample mean within 6 standard errors (+ fp32 slack) of ref."""
    return bool(np.all(np.abs(mean - ref) <= 6.0 * se + slack))


def _linear_autograd(x, w, gamma, gy):
    sx = torch.tensor(om.sign(x), dtype=torch.float64, requires_grad=True)
    sw = torch.tensor(om.sign(w), dtype=torch.float64, requires_grad=True)
    y = (sx @ sw.T) * torch.tensor(gamma, dtype=torch.float64)
    y.backward(torch.tensor(gy, dtype=torch.float64))
    return sx.grad.numpy(), sw.grad.numpy()


def test_linear_gamma_path_mean_matches_autograd():
    rng = np.random.default_rng(31)
    M, K, D, trials = 8, 6, 5, 2500
    x = rng.standard_normal((M, K)).astype(f32)
    w = rng.standard_normal((D, K)).astype(f32)
    gamma = np.array([0.1, 3.0, 0.5, 8.0, 1.5], dtype=f32)
    gy = (rng.standard_normal((M, D)) * 10.0 ** rng.uniform(-1, 1, (M, 1))).astype(f32)
    dxs, dws = [], []
    for seed in range(trials):
        r = om.layer_step_linear(x, w, gamma, gy, 2, om.SYSTEMATIC, seed, 2, om.SYSTEMATIC, 77777 + seed)
        dxs.append(r["dx"])
        dws.append(r["dw"])
    mx, sx_ = _stats(dxs)
    mw, sw_ = _stats(dws)
    ref_dx, ref_dw = _linear_autograd(x, w, gamma, gy)
    slack_x = 1e-5 * np.abs(ref_dx).max()
    slack_w = 1e-5 * np.abs(ref_dw).max()
    assert _within(mx, sx_, ref_dx, slack_x)
    assert _within(mw, sw_, ref_dw, slack_w)
    # the check has power: each plausible mistake in the Gamma pre-scale is rejected
    for bad in (np.ones(D, f32), gamma[::-1].copy(), (gamma * gamma).astype(f32)):
        bdx, bdw = _linear_autograd(x, w, bad, gy)
        assert not _within(mx, sx_, bdx, slack_x)
        assert not _within(mw, sw_, bdw, slack_w)


def _conv_autograd(x, w, gamma, gy, stride, pad):
    """Chain rule of y = Gamma (.) conv(sign(X) padded with sign -1 (reading R1), sign(W))."""
    N, C, H, W = x.shape
    D = w.shape[0]
    sx = torch.tensor(om.sign(x), dtype=torch.float64, requires_grad=True)
    sw = torch.tensor(om.sign(w), dtype=torch.float64, requires_grad=True)
    sxp = torch.nn.functional.pad(sx, (pad, pad, pad, pad), value=-1.0)
    y = torch.nn.functional.conv2d(sxp, sw, stride=stride) * torch.tensor(gamma, dtype=torch.float64)[None, :, None, None]
    Ho, Wo = y.shape[2], y.shape[3]
    g = torch.tensor(gy, dtype=torch.float64).reshape(N, Ho, Wo, D).permute(0, 3, 1, 2)
    y.backward(g)
    return sx.grad.numpy(), sw.grad.numpy()


def test_conv_gamma_path_mean_matches_autograd():
    rng = np.random.default_rng(32)
    N, C, H, W, D, k, s, p, trials = 4, 2, 4, 4, 3, 3, 1, 1, 1500
    x = rng.standard_normal((N, C, H, W)).astype(f32)
    w = rng.standard_normal((D, C, k, k)).astype(f32)
    gamma = np.array([0.2, 4.0, 1.0], dtype=f32)
    Ho, Wo = om.conv_out_hw(H, W, k, k, s, p)
    gy = (rng.standard_normal((N * Ho * Wo, D)) *
          np.repeat(10.0 ** rng.uniform(-1, 1, (N, 1)), Ho * Wo, axis=0)).astype(f32)
    dxs, dws = [], []
    for seed in range(trials):
        r = om.layer_step_conv(x, w, gamma, gy, s, p, 2, om.SYSTEMATIC, seed, 2, om.SYSTEMATIC, 55555 + seed)
        dxs.append(r["dx"])
        dws.append(r["dw"])
    mx, sx_ = _stats(dxs)
    mw, sw_ = _stats(dws)
    ref_dx, ref_dw = _conv_autograd(x, w, gamma, gy, s, p)
    slack_x = 1e-5 * np.abs(ref_dx).max()
    slack_w = 1e-5 * np.abs(ref_dw).max()
    assert _within(mx, sx_, ref_dx, slack_x)
    assert _within(mw, sw_, ref_dw, slack_w)
    for bad in (np.ones(D, f32), gamma[::-1].copy()):
        bdx, bdw = _conv_autograd(x, w, bad, gy, s, p)
        assert not _within(mx, sx_, bdx, slack_x)
        assert not _within(mw, sw_, bdw, slack_w)


def test_grad_to_quantize_is_per_channel():
    """G[m, j] = fp32(gY[m, j] * Gamma[j]), checked element by element with Python floats
    (an fp32 product of two fp32 values is exact in float64, then rounded once)."""
    rng = np.random.default_rng(33)
    gy = rng.standard_normal((6, 4)).astype(f32)
    gamma = rng.uniform(0.1, 5, 4).astype(f32)
    g = om.grad_to_quantize(gy, gamma)
    for m in range(6):
        for j in range(4):
            assert g[m, j] == f32(float(gy[m, j]) * float(gamma[j]))
    assert np.array_equal(om.grad_to_quantize(gy, None), gy)


def test_colsum_sign_plain_loops():
    """colsum[k] = sum over rows of sign(a[r, k]) (Sec. 5.1 sign: +1 iff a > 0), by loops."""
    rng = np.random.default_rng(34)
    a = rng.standard_normal((23, 9)).astype(f32)
    a[0, 0], a[1, 1], a[2, 2], a[3, 3], a[4, 4] = 0.0, -0.0, np.nan, np.inf, -np.inf
    a[:, 5] = 1.0   # all +1
    a[:, 6] = -1.0  # all -1
    cs = om.colsum_sign(a)
    for k in range(a.shape[1]):
        tot = 0
        for r in range(a.shape[0]):
            tot += 1 if a[r, k] > 0 else -1
        assert cs[k] == tot
    assert cs[5] == 23 and cs[6] == -23


def test_forward_bias_plain_loops():
    """y[m, j] = fp32(fp32(Gamma_j acc[m, j]) + bias_j) (reading R10), by loops with Python
    floats: the product of an fp32 value and an integer below 2^24 is exact in float64 and the
    sum of two fp32 values rounded once from float64 is the fp32 sum.  The other order
    (Gamma (acc + bias)) gives different values on these inputs, so it would fail."""
    rng = np.random.default_rng(35)
    M, K, D = 6, 50, 5
    x = rng.standard_normal((M, K)).astype(f32)
    w = rng.standard_normal((D, K)).astype(f32)
    gamma = rng.uniform(0.3, 3, D).astype(f32)
    bias = (rng.standard_normal(D) * 3).astype(f32)
    acc, y = om.forward_bias(x, w, gamma, bias)
    other = 0
    for m in range(M):
        for j in range(D):
            s = sum((1 if x[m, k] > 0 else -1) * (1 if w[j, k] > 0 else -1) for k in range(K))
            assert acc[m, j] == s
            ref = f32(float(f32(float(gamma[j]) * s)) + float(bias[j]))
            assert y[m, j] == ref
            other += int(f32(float(gamma[j]) * (s + float(bias[j]))) != ref)
    assert other > 0


@pytest.mark.parametrize("stride,pad,k", [(1, 1, 3), (2, 0, 1)])
def test_conv_gamma_none_equals_unit_gamma(stride, pad, k):
    """Gamma = None and Gamma = 1 give the same step (the pre-scale by 1 is exact)."""
    rng = np.random.default_rng(36 + k)
    N, C, H, W, D = 2, 2, 4, 4, 3
    x = rng.standard_normal((N, C, H, W)).astype(f32)
    w = rng.standard_normal((D, C, k, k)).astype(f32)
    Ho, Wo = om.conv_out_hw(H, W, k, k, stride, pad)
    gy = rng.standard_normal((N * Ho * Wo, D)).astype(f32)
    a = om.layer_step_conv(x, w, None, gy, stride, pad, 2, om.SYSTEMATIC, 3, 2, om.SYSTEMATIC, 4)
    b = om.layer_step_conv(x, w, np.ones(D, f32), gy, stride, pad, 2, om.SYSTEMATIC, 3, 2, om.SYSTEMATIC, 4)
    assert np.array_equal(a["dx"], b["dx"]) and np.array_equal(a["dw"], b["dw"])
