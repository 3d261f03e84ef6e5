"""GPU parity of the binop layers (Linear, Conv2d) against the oracle.

Forward: y = fp32(Gamma * acc) + bias bit for bit (Sec. 5.1, reading R10).  Backward with
the seeds of the oracle step: the input and weight gradients of Eq. 21 with SCQ within
1e-5 of the magnitudes of their two dequantization terms (as the layer-step parity tests),
the Gamma and bias gradients within 1e-5 of sum |terms|, and the clipped STE exactly.
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


def close_terms(gpu, ref, a_mag, c_mag, what):
    tol = 1e-5 * (a_mag + c_mag) + 1e-30
    err = np.abs(gpu.astype(np.float64) - ref.astype(np.float64))
    assert not (err > tol).any(), f"{what}: {(err > tol).sum()} elements out of tolerance, max err {err.max()}"


def dequant_magnitudes(acc, qb, colsum, rows_per_group, n_rows, row_len):
    """|S' acc| and |Z' colsum| per output element of a kept group (0 for pruned groups)."""
    a = np.zeros((n_rows, row_len))
    c = np.zeros((n_rows, row_len))
    for s_, g in enumerate(qb["kept"]):
        rows = slice(g * rows_per_group, (g + 1) * rows_per_group)
        a[rows] = np.abs(np.float64(qb["scale"][s_]) * acc[s_ * rows_per_group:(s_ + 1) * rows_per_group])
        c[rows] = np.abs(np.float64(qb["zero"][s_]) * colsum)[None, :]
    return a, c


def check_scale_bias(layer, gy2, acc):
    dg, db = om.scale_bias_grad(gy2, acc)
    tg = (np.abs(gy2.astype(np.float64)) * np.abs(acc)).sum(axis=0)
    tb = np.abs(gy2.astype(np.float64)).sum(axis=0)
    assert np.all(np.abs(layer.gamma.grad.cpu().numpy() - dg) <= 1e-5 * tg + 1e-30), "dGamma"
    if layer.bias is not None:
        assert np.all(np.abs(layer.bias.grad.cpu().numpy() - db) <= 1e-5 * tb + 1e-30), "dbias"


@pytest.mark.parametrize("M,K,D,bits,mode,clip,bias", [
    (40, 200, 96, 4, om.SYSTEMATIC, None, True),
    (33, 70, 30, 2, om.BERNOULLI, 1.0, False),
    (64, 512, 128, 8, om.SYSTEMATIC, 0.5, True),
])
def test_linear(M, K, D, bits, mode, clip, bias):
    from paper_2408_14267_gb300 import binop
    rng = np.random.default_rng(M + K + D)
    x = rng.standard_normal((M, K)).astype(np.float32)
    w = rng.standard_normal((D, K)).astype(np.float32)
    gamma = rng.uniform(0.5, 2.0, D).astype(np.float32)
    b = rng.standard_normal(D).astype(np.float32) if bias else None
    s = 10.0 ** rng.uniform(-2, 2, (M, 1))
    gy = (rng.laplace(0, 1e-3, (M, D)) * s).astype(np.float32)
    layer = binop.Linear(K, D, bias=bias, qcfg=binop.QuantConfig(bits, mode, ste_clip=clip))
    with torch.no_grad():
        layer.weight.copy_(torch.from_numpy(w))
        layer.gamma.copy_(torch.from_numpy(gamma))
        if bias:
            layer.bias.copy_(torch.from_numpy(b))
    xt = torch.from_numpy(x).cuda().requires_grad_(True)
    y = layer(xt)
    acc, y_ref = om.forward_bias(x, w, gamma, b)
    assert np.array_equal(y.detach().cpu().numpy(), y_ref), "forward"
    layer.next_seeds = (5, 6)
    y.backward(torch.from_numpy(gy).cuda())
    ref = om.layer_step_linear(x, w, gamma, gy, bits, mode, 5, bits, mode, 6, 1)
    assert not layer.nonfinite_gradient()
    a, c = dequant_magnitudes(ref["acc_dx"], ref["psq"], om.colsum_sign(w), 1, M, K)
    dx_ref = ref["dx"] if clip is None else om.ste_clip(x, ref["dx"], clip)
    close_terms(xt.grad.cpu().numpy(), dx_ref, a, c, "dx")
    a, c = dequant_magnitudes(ref["acc_dw"], ref["pcq"], om.colsum_sign(x), 1, D, K)
    dw_ref = ref["dw"] if clip is None else om.ste_clip(w, ref["dw"], clip)
    close_terms(layer.weight.grad.cpu().numpy(), dw_ref, a, c, "dW")
    check_scale_bias(layer, gy, acc)


@pytest.mark.parametrize("N,C,H,W,D,k,stride,pad,bits,clip,bias", [
    (5, 30, 8, 8, 24, 3, 1, 1, 4, None, True),    # Folder in the grad_input epilogue
    (3, 12, 10, 10, 32, 3, 1, 1, 2, 1.0, False),  # 100 pixels per sample: two-call grad_input + Folder
    (2, 8, 16, 16, 16, 3, 2, 1, 8, None, True),   # stride 2 (fused Folder), 8-bit codes
])
def test_conv2d(N, C, H, W, D, k, stride, pad, bits, clip, bias):
    from paper_2408_14267_gb300 import binop
    rng = np.random.default_rng(N * C + D)
    x = rng.standard_normal((N, C, H, W)).astype(np.float32)
    w = (rng.standard_normal((D, C, k, k)) * 0.1).astype(np.float32)
    gamma = rng.uniform(0.5, 2.0, D).astype(np.float32)
    b = rng.standard_normal(D).astype(np.float32) if bias else None
    Ho, Wo = om.conv_out_hw(H, W, k, k, stride, pad)
    s = np.exp(1.5 * rng.standard_normal((N, 1, 1)))
    gy = (rng.standard_normal((N, Ho * Wo, D)) * 1e-3 * s).reshape(N * Ho * Wo, D).astype(np.float32)
    layer = binop.Conv2d(C, D, k, stride=stride, padding=pad, bias=bias,
                         qcfg=binop.QuantConfig(bits, om.SYSTEMATIC, ste_clip=clip))
    with torch.no_grad():
        layer.weight.copy_(torch.from_numpy(w))
        layer.gamma.copy_(torch.from_numpy(gamma))
        if bias:
            layer.bias.copy_(torch.from_numpy(b))
    xt = torch.from_numpy(x).cuda().requires_grad_(True)
    y = layer(xt)
    assert tuple(y.shape) == (N, D, Ho, Wo)
    x_u = om.unfold(x, k, k, stride, pad)
    acc, y_ref = om.forward_bias(x_u, w.reshape(D, -1), gamma, b)
    y_rows = y.detach().permute(0, 2, 3, 1).reshape(N * Ho * Wo, D).cpu().numpy()
    assert np.array_equal(y_rows, y_ref), "forward"
    layer.next_seeds = (7, 8)
    gy_nchw = torch.from_numpy(gy.reshape(N, Ho, Wo, D)).cuda().permute(0, 3, 1, 2)
    y.backward(gy_nchw)
    ref = om.layer_step_conv(x, w, gamma, gy, stride, pad, bits, om.SYSTEMATIC, 7, bits, om.SYSTEMATIC, 8)
    assert not layer.nonfinite_gradient()
    psq = ref["psq"]
    a_mag = np.zeros(ref["dx"].shape)
    c_mag = np.zeros(ref["dx"].shape)
    for s_, g in enumerate(psq["kept"]):
        a_mag[g] = np.abs(np.float64(psq["scale"][s_]) * ref["acc_fold"][g])
        c_mag[g] = np.abs(np.float64(psq["zero"][s_]) * ref["cs_fold"])
    dx_ref = ref["dx"] if clip is None else om.ste_clip(x, ref["dx"], clip)
    close_terms(xt.grad.cpu().numpy(), dx_ref, a_mag, c_mag, "dx")
    w_u = w.reshape(D, -1)
    a, c = dequant_magnitudes(ref["acc_dw"], ref["pcq"], om.colsum_sign(x_u), 1, D, w_u.shape[1])
    dw_ref = ref["dw"].reshape(D, -1) if clip is None else om.ste_clip(w_u, ref["dw"].reshape(D, -1), clip)
    close_terms(layer.weight.grad.cpu().numpy().reshape(D, -1), dw_ref, a, c, "dW")
    check_scale_bias(layer, gy, acc)


def test_layers_compose_with_torch():
    """binop layers inside an ordinary torch model: gradients reach every parameter and are
    finite, and the per-backward seeds change the stochastic gradient between steps."""
    from paper_2408_14267_gb300 import binop
    torch.manual_seed(0)
    net = torch.nn.Sequential(
        binop.Conv2d(16, 32, 3, padding=1), torch.nn.BatchNorm2d(32).cuda(), torch.nn.Hardtanh(),
        binop.Conv2d(32, 32, 3, padding=1, bias=True), torch.nn.BatchNorm2d(32).cuda(), torch.nn.Hardtanh(),
        torch.nn.Flatten(), binop.Linear(32 * 8 * 8, 10, bias=True))
    x = torch.randn(16, 16, 8, 8, device="cuda")
    target = torch.randint(0, 10, (16,), device="cuda")
    grads = []
    for _ in range(2):
        net.zero_grad()
        torch.nn.functional.cross_entropy(net(x), target).backward()
        for p in net.parameters():
            assert p.grad is not None and torch.isfinite(p.grad).all()
        grads.append(net[0].weight.grad.clone())
    assert not torch.equal(grads[0], grads[1])


def test_conv2d_channels_last_input_matches_nchw():
    """A channels-last input takes the plane-bit Unfolder path (no copy of x) and gives the
    same output and gradients as the same input in NCHW layout."""
    from paper_2408_14267_gb300 import binop
    torch.manual_seed(3)
    layer = binop.Conv2d(64, 32, 3, padding=1, bias=True)
    x = torch.randn(4, 64, 16, 16, device="cuda")
    gy = torch.randn(4, 32, 16, 16, device="cuda") * 1e-3
    _check_layouts(layer, x, gy)
    small = binop.Conv2d(32, 16, 3, padding=1, qcfg=binop.QuantConfig(4, ste_clip=1.0))  # 8 x 8: fused Folder
    _check_layouts(small, torch.randn(6, 32, 8, 8, device="cuda"), torch.randn(6, 16, 8, 8, device="cuda") * 1e-3)


def _check_layouts(layer, x, gy):
    res = []
    for fmt in (torch.contiguous_format, torch.channels_last):
        xi = x.clone().contiguous(memory_format=fmt).requires_grad_(True)
        layer.zero_grad()
        layer.next_seeds = (11, 12)
        y = layer(xi)
        y.backward(gy)
        if fmt is torch.channels_last:  # the gradient comes back in the input's layout
            assert xi.grad.is_contiguous(memory_format=torch.channels_last)
        res.append((y.detach().clone(), xi.grad.clone(), layer.weight.grad.clone(), layer.gamma.grad.clone(),
                    layer.bias.grad.clone() if layer.bias is not None else layer.gamma.grad.clone()))
    for a, b in zip(*res):
        assert torch.equal(a, b)
