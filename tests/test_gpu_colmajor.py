"""grad_input through column-major int32 accumulators and the column-major Folder.

fqt1_bwd_input_gemm_colmajor must give the oracle's integer accumulators bit for bit
(stored column-major), and fqt1_col2im_colmajor the same dx as the row-major two-call
Folder, bit for bit, and the oracle's folded gradient within 1e-5 of the magnitude of the
dequantization terms; pruned samples are zero.  Shapes: every window, stride and padding
the layer shapes use (3 x 3 stride 1 and 2, 1 x 1 stride 1 and 2, the 7 x 7 stride-2 stem),
maps whose H W does not divide 128, ragged channel counts and the runtime-window kernel
(5 x 5 stride 3, 2 x 4 windows).
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

from oracle import method as om  # noqa: E402

from test_gpu_parity import assert_dequant_close, conv_case, run_oracle  # noqa: E402

SYS, BER, TOP = om.SYSTEMATIC, om.BERNOULLI, om.TOPK


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2408_14267_gb300 import build
    build.build()


def _rect_case(N, C, H, W, D, kh, kw, s, p, bits, mode, seed):
    """A convolution with a kh x kw window (conv_case draws square windows)."""
    from paper_2408_14267_gb300 import workloads as wl
    d = wl.conv_layer(f"conv N{N} C{C} {H}x{W} D{D} k{kh}x{kw}s{s}p{p} b{bits}", N, C, H, W, D, kh, s, p, bits,
                      seed + 5, seed + 77, sample_sigma=1.5)
    rng = np.random.default_rng(seed)
    d["w"] = rng.standard_normal((D, C, kh, kw)).astype(np.float32)
    Ho, Wo = (H + 2 * p - kh) // s + 1, (W + 2 * p - kw) // s + 1
    n_rows = N * Ho * Wo
    scale = 10.0 ** rng.uniform(-2, 2, size=(N, 1, 1))
    d["gy"] = (rng.standard_t(3, (N, Ho * Wo, D)) * 1e-3 * scale).reshape(n_rows, D).astype(np.float32)
    d["rows_per_group"] = Ho * Wo
    d["mode_s"] = d["mode_c"] = mode
    return d


COLMAJOR_CASES = [
    ("56x56-3x3-s1-64ch", lambda: conv_case(3, 64, 56, 56, 64, 3, 1, 1, 4, SYS, seed=31)),
    ("28x28-3x3-s1-b8", lambda: conv_case(4, 20, 28, 28, 36, 3, 1, 1, 8, SYS, seed=32)),
    ("56x56-3x3-s2", lambda: conv_case(3, 16, 56, 56, 32, 3, 2, 1, 4, BER, seed=33)),
    ("7x7-3x3-s1-512ch", lambda: conv_case(8, 512, 7, 7, 24, 3, 1, 1, 4, SYS, seed=34)),
    ("14x14-1x1-s2", lambda: conv_case(6, 40, 14, 14, 48, 1, 2, 0, 2, SYS, seed=35)),
    ("9x9-1x1-s1-ragged", lambda: conv_case(5, 33, 9, 9, 20, 1, 1, 0, 4, TOP, seed=36)),
    ("stem-7x7-s2-64x64", lambda: conv_case(4, 3, 64, 64, 32, 7, 2, 3, 4, SYS, seed=37)),
    ("stem-7x7-s2-odd-map", lambda: conv_case(3, 3, 37, 29, 16, 7, 2, 3, 2, BER, seed=38)),
    ("5x5-s3-p2-runtime-window", lambda: conv_case(3, 6, 17, 13, 8, 5, 3, 2, 4, SYS, seed=39)),
    ("2x4-window-s1-p0", lambda: _rect_case(3, 7, 11, 10, 12, 2, 4, 1, 0, 4, SYS, seed=40)),
    ("single-sample-b1", lambda: conv_case(1, 9, 12, 12, 10, 3, 1, 1, 1, SYS, seed=41)),
    # 255 x 200 > 32767: the accumulators stay int32 (chosen by LayerStep, checked below)
    ("b8-wide-D-int32", lambda: conv_case(3, 10, 12, 12, 200, 3, 1, 1, 8, SYS, seed=42)),
]


@pytest.mark.parametrize("name,make", COLMAJOR_CASES, ids=[c[0] for c in COLMAJOR_CASES])
def test_colmajor_grad_input_matches_oracle_and_row_major_folder(name, make):
    from paper_2408_14267_gb300.layer import LayerStep
    w = make()
    ref = run_oracle(w)
    cm = LayerStep(w, keep_acc=False, fold=False, colmajor=True)
    rm = LayerStep(w, keep_acc=True, fold=False, colmajor=False)
    assert cm.colmajor and not rm.colmajor
    # int16 exactly where every sum fits: (2^b - 1) D <= 32767
    assert cm.acc_bits_cm == (16 if ((1 << w["bits_s"]) - 1) * cm.D <= 32767 else 32)
    cm.dx.fill_(7.0)  # pruned samples must be overwritten with zeros
    cm.step()
    rm.step()
    torch.cuda.synchronize()
    psq = ref["psq"]
    rows = len(psq["kept"]) * cm.rpg
    assert cm.psq.count() == len(psq["kept"])
    acc = cm.acc_dx_cm.cpu().numpy()[:, :rows].T.astype(np.int64)
    assert np.array_equal(acc, ref["acc_dx"]), f"column-major int{cm.acc_bits_cm} accumulators"
    assert torch.equal(cm.dx, rm.dx), "column-major Folder against the row-major Folder"
    a_mag = np.zeros(ref["dx"].shape)
    c_mag = np.zeros(ref["dx"].shape)
    for s_, g in enumerate(psq["kept"]):
        a_mag[g] = np.abs(np.float64(psq["scale"][s_]) * ref["acc_fold"][g])
        c_mag[g] = np.abs(np.float64(psq["zero"][s_]) * ref["cs_fold"])
    dx = cm.dx.cpu().numpy()
    assert_dequant_close(dx, ref["dx"], a_mag, c_mag, "grad_input (column-major Folder)")
    for g in np.setdiff1d(np.arange(w["x"].shape[0]), psq["kept"]):
        assert np.all(dx[g] == 0)
    # a second step on the same buffers reproduces the first
    dx0 = cm.dx.clone()
    cm.step()
    torch.cuda.synchronize()
    assert torch.equal(cm.dx, dx0)


def test_colmajor_is_the_default_without_fused_folder():
    """keep_acc=False (the benchmark's configuration) takes the column-major path exactly where
    the fused Folder does not apply."""
    from paper_2408_14267_gb300.layer import LayerStep
    from paper_2408_14267_gb300 import workloads as wl
    assert LayerStep(COLMAJOR_CASES[0][1](), keep_acc=False).colmajor
    st = LayerStep(wl.resnet18_cifar_conv(), keep_acc=False)
    assert st.fold and not st.colmajor
    assert not LayerStep(COLMAJOR_CASES[0][1](), keep_acc=True).colmajor


@pytest.mark.parametrize("name,make", [COLMAJOR_CASES[i] for i in (0, 2, 6, 8)],
                         ids=[COLMAJOR_CASES[i][0] for i in (0, 2, 6, 8)])
def test_colmajor_e4m3_weights_equal_packed(name, make):
    """fqt1_bwd_input_gemm_colmajor_e4m3w (sign(W)^T bytes by TMA) gives the packed-sign
    product's accumulators and dx bit for bit."""
    from paper_2408_14267_gb300.layer import LayerStep
    w = make()
    a = LayerStep(w, keep_acc=False, fold=False, colmajor=True, e4m3_weights="colmajor")
    b = LayerStep(w, keep_acc=False, fold=False, colmajor=True, e4m3_weights=False)
    assert a.wt8 is not None and b.wt8 is None
    a.step()
    b.step()
    torch.cuda.synchronize()
    rows = a.psq.count() * a.rpg
    assert rows == b.psq.count() * b.rpg
    assert torch.equal(a.acc_dx_cm[:, :rows], b.acc_dx_cm[:, :rows])
    assert torch.equal(a.dx, b.dx)


@pytest.mark.parametrize("name,make", [COLMAJOR_CASES[i] for i in (0, 3, 6, 8, 10)],
                         ids=[COLMAJOR_CASES[i][0] for i in (0, 3, 6, 8, 10)])
def test_colmajor_int16_equals_int32(name, make):
    """int16 column-major accumulators (chosen where (2^b - 1) D fits) give the int32 path's
    accumulators and dx bit for bit."""
    from paper_2408_14267_gb300.layer import LayerStep
    w = make()
    a = LayerStep(w, keep_acc=False, fold=False, colmajor=True, acc16=True)
    b = LayerStep(w, keep_acc=False, fold=False, colmajor=True, acc16=False)
    assert a.acc_bits_cm == 16 and b.acc_bits_cm == 32
    a.step()
    b.step()
    torch.cuda.synchronize()
    rows = a.psq.count() * a.rpg
    assert torch.equal(a.acc_dx_cm[:, :rows].to(torch.int32), b.acc_dx_cm[:, :rows])
    assert torch.equal(a.dx, b.dx)


def test_colmajor_int16_bound():
    """int16 is taken exactly when every accumulator fits: (2^b - 1) D <= 32767."""
    from paper_2408_14267_gb300 import fqt1
    assert fqt1.colmajor_acc_bits(4, 2184) == 16 and fqt1.colmajor_acc_bits(4, 2185) == 32
    assert fqt1.colmajor_acc_bits(8, 128) == 16 and fqt1.colmajor_acc_bits(8, 129) == 32
    assert fqt1.colmajor_acc_bits(1, 32767) == 16 and fqt1.colmajor_acc_bits(1, 32768) == 32


@pytest.mark.parametrize("name,make", [COLMAJOR_CASES[i] for i in (0, 2, 4, 6, 8, 9)],
                         ids=[COLMAJOR_CASES[i][0] for i in (0, 2, 4, 6, 8, 9)])
def test_colmajor_channels_last_output(name, make):
    """fqt1_col2im_colmajor_nhwc writes the NCHW Folder's values in N, H, W, C order (pruned
    samples included), from int16 and from int32 accumulators."""
    from paper_2408_14267_gb300 import fqt1
    from paper_2408_14267_gb300.layer import LayerStep
    w = make()
    for acc16 in (True, False):
        st = LayerStep(w, keep_acc=False, fold=False, colmajor=True, acc16=acc16)
        st.step()
        N, C, H, W, kh, kw = st.conv
        dx = torch.full((N, H, W, C), 3.0, device="cuda")
        fqt1.col2im_colmajor(st.acc_dx_cm, st.psq, st.cs_w, N, C, H, W, kh, kw, st.stride, st.pad, dx, nhwc=True)
        torch.cuda.synchronize()
        assert torch.equal(dx.permute(0, 3, 1, 2), st.dx)
