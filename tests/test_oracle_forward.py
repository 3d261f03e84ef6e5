"""Pins of the oracle's forward pass: sign, binary product, Unfolder / Folder (Sec. 5.1, App. C)."""
import itertools

import numpy as np
import pytest
import torch

from oracle import method as om


def test_sign_definition():
    """Sec. 5.1: sign(x) = -1 if x <= 0 else +1 (so 0, -0 and NaN give -1)."""
    x = np.array([0.0, -0.0, np.nan, 1e-45, -1e-45, 3.0, -2.0, np.inf, -np.inf], dtype=np.float32)
    assert om.sign(x).tolist() == [-1, -1, -1, 1, -1, 1, -1, 1, -1]


def _xnor_popcount_dot(a_bits, b_bits, K):
    """App. C: SUM(X1 (.) X2) = (bitcount(XNOR(x1, x2)) << 1) - K for K-element words."""
    mask = (1 << K) - 1
    return (bin(~(a_bits ^ b_bits) & mask).count("1") << 1) - K


@pytest.mark.parametrize("K", [1, 2, 5, 8])
def test_binary_product_exhaustive_xnor(K):
    """Every pair of +-1 vectors of length K: oracle product == XNOR-popcount form."""
    vecs = list(itertools.product([0, 1], repeat=K))
    a = np.array([[1.0 if b else -1.0 for b in v] for v in vecs], dtype=np.float32)
    acc, _ = om.forward(a, a, np.ones(len(vecs), dtype=np.float32))
    bits = [sum(b << i for i, b in enumerate(v)) for v in vecs]
    for i, bi in enumerate(bits):
        for j, bj in enumerate(bits):
            assert acc[i, j] == _xnor_popcount_dot(bi, bj, K)


def test_forward_brute_force():
    rng = np.random.default_rng(3)
    M, K, D = 5, 37, 7
    x = rng.standard_normal((M, K)).astype(np.float32)
    x[0, :3] = 0.0
    w = rng.standard_normal((D, K)).astype(np.float32)
    gamma = rng.uniform(0.1, 2, D).astype(np.float32)
    acc, y = om.forward(x, w, gamma)
    for m in range(M):
        for j in range(D):
            s = 0
            for k in range(K):
                sx = 1 if x[m, k] > 0 else -1
                sw = 1 if w[j, k] > 0 else -1
                s += sx * sw
            assert acc[m, j] == s
            assert y[m, j] == np.float32(gamma[j]) * np.float32(s)
    assert y.dtype == np.float32


@pytest.mark.parametrize("N,C,H,W,k,s,p", [(2, 3, 7, 6, 3, 1, 1), (1, 2, 9, 9, 7, 2, 3), (2, 4, 6, 6, 1, 2, 0),
                                           (3, 1, 5, 4, 3, 2, 1), (1, 5, 4, 4, 3, 1, 0)])
def test_unfold_fold_match_torch(N, C, H, W, k, s, p):
    """Unfolder == torch unfold (rows NHW, columns C*k*k); Folder == torch fold."""
    rng = np.random.default_rng(N * 100 + C)
    x = rng.standard_normal((N, C, H, W)).astype(np.float32)
    xu = om.unfold(x, k, k, s, p)
    ref = torch.nn.functional.unfold(torch.from_numpy(x), k, padding=p, stride=s)  # [N, C*k*k, L]
    ref = ref.transpose(1, 2).reshape(-1, C * k * k).numpy()
    assert np.array_equal(xu, ref)
    Ho, Wo = om.conv_out_hw(H, W, k, k, s, p)
    acc = rng.integers(-1000, 1000, size=(N * Ho * Wo, C * k * k))
    folded = om.fold_int(acc, N, C, H, W, k, k, s, p)
    t = torch.from_numpy(acc.astype(np.float64)).reshape(N, Ho * Wo, C * k * k).transpose(1, 2)
    reff = torch.nn.functional.fold(t, (H, W), k, padding=p, stride=s).numpy()
    assert np.array_equal(folded, reff.astype(np.int64))


def test_conv_forward_pads_as_minus_one():
    """Conv forward through the Unfolder equals a convolution of sign(zero-padded X) (reading R1)."""
    rng = np.random.default_rng(11)
    N, C, H, W, D, k, s, p = 2, 3, 6, 5, 4, 3, 2, 1
    x = rng.standard_normal((N, C, H, W)).astype(np.float32)
    w = rng.standard_normal((D, C, k, k)).astype(np.float32)
    acc, _ = om.forward(om.unfold(x, k, k, s, p), w.reshape(D, -1), np.ones(D, np.float32))
    xp = np.pad(x, ((0, 0), (0, 0), (p, p), (p, p)))
    sx = torch.from_numpy(np.where(xp > 0, 1.0, -1.0))
    sw = torch.from_numpy(np.where(w > 0, 1.0, -1.0))
    ref = torch.nn.functional.conv2d(sx, sw, stride=s).numpy()  # [N, D, Ho, Wo]
    assert np.array_equal(acc.reshape(N, -1, D), ref.reshape(N, D, -1).transpose(0, 2, 1).astype(np.int64))


def _direct_conv_signs(x, w, pad):
    """Brute-force stride-1 convolution of sign(zero-padded x) with sign(w), plain loops."""
    N, C, H, W = x.shape
    D, _, kh, kw = w.shape
    Ho, Wo = H + 2 * pad - kh + 1, W + 2 * pad - kw + 1
    out = np.zeros((N * Ho * Wo, D), dtype=np.int64)
    for n in range(N):
        for oh in range(Ho):
            for ow in range(Wo):
                for d in range(D):
                    s = 0
                    for c in range(C):
                        for i in range(kh):
                            for j in range(kw):
                                h, ww = oh + i - pad, ow + j - pad
                                v = x[n, c, h, ww] if 0 <= h < H and 0 <= ww < W else 0.0
                                s += (1 if v > 0 else -1) * (1 if w[d, c, i, j] > 0 else -1)
                    out[(n * Ho + oh) * Wo + ow, d] = s
    return out


@pytest.mark.parametrize("N,C,H,W,D,k,p", [(2, 3, 4, 5, 3, 3, 1), (1, 4, 3, 3, 2, 1, 0), (2, 2, 5, 4, 2, 5, 2),
                                           (1, 3, 4, 4, 2, 3, 0)])
def test_implicit_conv_matches_direct_convolution(N, C, H, W, D, k, p):
    """The tap-by-tap implicit product equals a brute-force convolution of the signs and the
    Unfolder product; regathering the pixel-major rows by tap against the tap-major weight
    signs gives the same integers (pins both layouts: a transposed one fails)."""
    rng = np.random.default_rng(N * 31 + C * 7 + k)
    x = rng.standard_normal((N, C, H, W)).astype(np.float32)
    x[0, 0, 0, :2] = 0.0
    w = rng.standard_normal((D, C, k, k)).astype(np.float32)
    ref = _direct_conv_signs(x, w, p)
    assert np.array_equal(om.implicit_conv_acc(x, w, p), ref)
    acc_u, _ = om.forward(om.unfold(x, k, k, 1, p), w.reshape(D, -1), None)
    assert np.array_equal(acc_u, ref)
    Ho, Wo = H + 2 * p - k + 1, W + 2 * p - k + 1
    px = om.pixel_signs(x).astype(np.int64).reshape(N, H, W, C)
    a = np.full((N, Ho, Wo, k * k, C), -1, dtype=np.int64)  # row m, k' = t C + c
    for i in range(k):
        for j in range(k):
            for oh in range(Ho):
                for ow in range(Wo):
                    h, ww = oh + i - p, ow + j - p
                    if 0 <= h < H and 0 <= ww < W:
                        a[:, oh, ow, i * k + j, :] = px[:, h, ww, :]
    acc_t = om.int_matmul(a.reshape(N * Ho * Wo, k * k * C), om.tap_major_signs(w))
    assert np.array_equal(acc_t, ref)


def test_scale_bias_grad_matches_autograd():
    """dGamma and dbias of y = (sign(X) sign(W)^T) (.) Gamma + bias (Sec. 5.1 with a bias):
    the oracle's closed sums against torch autograd of the plain float64 formula."""
    rng = np.random.default_rng(21)
    M, K, D = 37, 45, 19
    x = rng.standard_normal((M, K))
    w = rng.standard_normal((D, K))
    gy = rng.standard_normal((M, D))
    sx = torch.tensor(om.sign(x), dtype=torch.float64)
    sw = torch.tensor(om.sign(w), dtype=torch.float64)
    gamma = torch.tensor(rng.uniform(0.5, 2.0, D), dtype=torch.float64, requires_grad=True)
    bias = torch.tensor(rng.standard_normal(D), dtype=torch.float64, requires_grad=True)
    y = (sx @ sw.T) * gamma + bias
    (y * torch.tensor(gy)).sum().backward()
    acc, _ = om.forward(x, w, np.ones(D, np.float32))
    dgamma, dbias = om.scale_bias_grad(gy, acc)
    assert np.allclose(dgamma, gamma.grad.numpy(), rtol=1e-12, atol=1e-12)
    assert np.allclose(dbias, bias.grad.numpy(), rtol=1e-12, atol=1e-12)


def test_forward_bias_adds_after_the_scale():
    rng = np.random.default_rng(22)
    x, w = rng.standard_normal((5, 40)), rng.standard_normal((7, 40))
    gamma = rng.uniform(0.5, 2.0, 7).astype(np.float32)
    bias = rng.standard_normal(7).astype(np.float32)
    acc, y0 = om.forward(x, w, gamma)
    acc1, y1 = om.forward_bias(x, w, gamma, bias)
    assert np.array_equal(acc, acc1)
    assert np.array_equal(y1, (y0 + bias[None, :]).astype(np.float32))
    assert np.array_equal(om.forward_bias(x, w, gamma, None)[1], y0)


def test_ste_clip_matches_hardtanh_gradient():
    """Clipped STE: the gradient of hardtanh(x) = clip(x, -1, 1) is 1 strictly inside (-1, 1)
    and 0 outside; the boundary |x| = 1 and NaN are the reading's own choices (pass, zero)."""
    rng = np.random.default_rng(23)
    x = rng.uniform(-3, 3, 1000)
    x = x[np.abs(np.abs(x) - 1) > 1e-9]
    g = rng.standard_normal(x.shape)
    xt = torch.tensor(x, requires_grad=True)
    torch.nn.functional.hardtanh(xt).backward(torch.tensor(g))
    assert np.array_equal(om.ste_clip(x, g, 1.0), xt.grad.numpy())
    assert np.array_equal(om.ste_clip(np.array([1.0, -1.0, np.nan, 0.5]), np.ones(4), 1.0), [1.0, 1.0, 0.0, 1.0])
    assert np.array_equal(om.ste_clip(np.array([0.3, 0.6]), np.array([2.0, 3.0]), 0.5), [2.0, 0.0])
