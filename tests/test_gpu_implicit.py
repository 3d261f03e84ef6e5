"""GPU parity of the implicit-GEMM convolution forward (the Unfolder of App. C left implicit).

The pixel-major and tap-major sign packings must equal the oracle's layouts bit for bit, and
the product must equal the oracle's forward on the unfolded matrix exactly (acc int32 and
y = Gamma acc + bias in fp32): it is the same integer sum in another order.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

from oracle import method as om  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2408_14267_gb300 import build
    build.build()


def unpack(words_i32, n):
    w = words_i32.cpu().numpy().view(np.uint32)
    bits = ((w[:, :, None] >> np.arange(32, dtype=np.uint32)) & 1).reshape(w.shape[0], -1)
    return bits[:, :n].astype(np.int8) * 2 - 1, bits[:, n:]


def inputs(N, C, H, W, D, k, seed):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((N, C, H, W)).astype(np.float32)
    x[0, :3, 0, 0] = 0.0  # zero is sign -1
    w = rng.standard_normal((D, C, k, k)).astype(np.float32)
    return x, w


@pytest.mark.parametrize("N,C,H,W", [(3, 128, 5, 7), (2, 256, 8, 8), (1, 384, 3, 11), (4, 128, 1, 1)])
def test_pack_pixels_matches_layout(N, C, H, W):
    from paper_2408_14267_gb300 import fqt1
    x, _ = inputs(N, C, H, W, 1, 1, N + C + H)
    xt = torch.from_numpy(x).cuda()
    out = torch.full((N * H * W, fqt1.packed_words(C)), -1, dtype=torch.int32, device="cuda")
    fqt1.pack_pixels(xt, N, C, H, W, out)
    torch.cuda.synchronize()
    bits, pad = unpack(out, C)
    assert np.array_equal(bits, om.pixel_signs(x)) and not pad.any()


@pytest.mark.parametrize("D,C,k", [(3, 32, 3), (17, 96, 1), (5, 256, 5), (2, 64, 7), (8, 1056, 3)])
def test_pack_weight_taps_matches_layout(D, C, k):
    from paper_2408_14267_gb300 import fqt1
    _, w = inputs(1, C, 1, 1, D, k, D + C + k)
    wt = torch.from_numpy(w).cuda()
    K = C * k * k
    out = torch.full((D, fqt1.packed_words(K)), -1, dtype=torch.int32, device="cuda")
    fqt1.pack_weight_taps(wt, D, C, k, k, out)
    torch.cuda.synchronize()
    bits, pad = unpack(out, K)
    assert np.array_equal(bits, om.tap_major_signs(w)) and not pad.any()


@pytest.mark.parametrize("N,C,H,W,D,k,bias,keep_acc", [
    (5, 128, 8, 8, 48, 3, True, True),      # 2 images per tile, ragged last tile (1 image)
    (2, 256, 16, 16, 136, 3, False, True),  # tiles of 8 image rows; two column tiles, the last ragged
    (9, 128, 4, 4, 24, 1, True, False),     # 1x1, 8 images per tile
    (1, 128, 32, 32, 16, 5, False, True),   # 5x5 over 32-pixel rows, last stage 1 of 4 sub-tiles
    (3, 128, 16, 8, 20, 7, True, True),     # 7x7 (pad 3 is wider than the 16-row tile halves)
    (64, 128, 2, 2, 8, 3, False, True),     # 32 images per tile; most taps read the padding
    (3, 512, 4, 4, 16, 3, True, True),      # four sub-tiles per box (C = 512)
    (2, 384, 8, 8, 16, 3, False, True),     # C / 128 = 3: one sub-tile per box
])
def test_conv_fwd_implicit_exact(N, C, H, W, D, k, bias, keep_acc):
    from paper_2408_14267_gb300 import fqt1
    x, w = inputs(N, C, H, W, D, k, N * 7 + C + D + k)
    rng = np.random.default_rng(D)
    gamma = rng.uniform(0.5, 2.0, D).astype(np.float32)
    b = rng.standard_normal(D).astype(np.float32) if bias else None
    pad = (k - 1) // 2
    assert fqt1.conv_implicit_supported(N, C, H, W, k, k, 1, pad)
    dev = "cuda"
    xp = torch.empty(N * H * W, fqt1.packed_words(C), dtype=torch.int32, device=dev)
    wt = torch.empty(D, fqt1.packed_words(C * k * k), dtype=torch.int32, device=dev)
    fqt1.pack_pixels(torch.from_numpy(x).to(dev), N, C, H, W, xp)
    fqt1.pack_weight_taps(torch.from_numpy(w).to(dev), D, C, k, k, wt)
    M = N * H * W
    acc = torch.full((M, D), 7, dtype=torch.int32, device=dev) if keep_acc else None
    y = torch.full((M, D), 7.0, dtype=torch.float32, device=dev)
    fqt1.conv_fwd_implicit(xp, wt, N, C, H, W, k, k, 1, pad, D, torch.from_numpy(gamma).to(dev),
                           None if b is None else torch.from_numpy(b).to(dev), acc, y)
    torch.cuda.synchronize()
    acc_ref, y_ref = om.forward_bias(om.unfold(x, k, k, 1, pad), w.reshape(D, -1), gamma, b)
    assert np.array_equal(acc_ref, om.implicit_conv_acc(x, w, pad))
    if keep_acc:
        assert np.array_equal(acc.cpu().numpy(), acc_ref), "acc"
    assert np.array_equal(y.cpu().numpy(), y_ref), "y"


def test_unsupported_shape_is_rejected():
    from paper_2408_14267_gb300 import fqt1
    t = torch.empty(64, dtype=torch.int32, device="cuda")
    g = torch.ones(16, device="cuda")
    with pytest.raises(fqt1.Fqt1Error, match="UNSUPPORTED"):
        fqt1.conv_fwd_implicit(t, t, 2, 128, 12, 12, 3, 3, 1, 1, 16, g, None, None, t.float())
