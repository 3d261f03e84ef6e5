"""GPU parity: the CUDA path through the C-ABI against the CPU oracle.

Integer and byte results (packed signs, column sums, ranges, keep
probabilities, kept lists, codes, int32 accumulators) must match bit for bit;
fp32 results within |gpu - ref| <= 1e-5 (|a| + |c|) + 1e-30 where a = S' acc
and c = Z' colsum are the two terms of the dequantization (1e-5 relative to
the magnitude of the terms, so cancellation between them cannot hide an error).
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

from oracle import method as om  # noqa: E402
from paper_2408_14267_gb300 import workloads as wl  # noqa: E402

SYS, BER, TOP = om.SYSTEMATIC, om.BERNOULLI, om.TOPK


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2408_14267_gb300 import build
    build.build()


def unpack_bits(words_i32, n):
    w = words_i32.cpu().numpy().view(np.uint32)
    bits = ((w[:, :, None] >> np.arange(32, dtype=np.uint32)) & 1).reshape(w.shape[0], -1)
    return bits[:, :n].astype(np.int8) * 2 - 1, bits[:, n:]


def unpack_e4m3(t, n):
    """e4m3 sign bytes [rows][ld] -> (+-1 int8 [rows][n], the bytes n .. next multiple of 16)."""
    b = t.cpu().numpy()
    v = b[:, :n]
    assert np.isin(v, (0x38, 0xB8)).all(), "bytes other than +-1 in e4m3 signs"
    return np.where(v == 0x38, 1, -1).astype(np.int8), b[:, n:(n + 15) // 16 * 16]


def linear_case(M, K, D, rpg, bits, mode, seed=0, gamma=True, bits_c=None, mode_c=None):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((M, K)).astype(np.float32)
    x[0, : min(3, K)] = 0.0
    w = rng.standard_normal((D, K)).astype(np.float32)
    s = 10.0 ** rng.uniform(-2, 2, size=(M // rpg, 1, 1))
    gy = (rng.laplace(0, 1e-3, (M // rpg, rpg, D)) * s).reshape(M, D).astype(np.float32)
    g = rng.uniform(0.5, 2.0, D).astype(np.float32) if gamma else None
    return dict(name=f"linear M{M} K{K} D{D} rpg{rpg} b{bits} m{mode}", kind="linear", x=x, w=w, gamma=g, gy=gy,
                rows_per_group=rpg, bits_s=bits, mode_s=mode, seed_s=seed + 11, bits_c=bits_c or bits,
                mode_c=mode if mode_c is None else mode_c, seed_c=seed + 12)


def conv_case(N, C, H, W, D, k, s, p, bits, mode, seed=0):
    d = wl.conv_layer(f"conv N{N} C{C} {H}x{W} D{D} k{k}s{s}p{p} b{bits}", N, C, H, W, D, k, s, p, bits, seed + 5,
                      seed + 77, sample_sigma=1.5)
    d["mode_s"] = d["mode_c"] = mode
    return d


def run_oracle(w):
    if w["kind"] == "conv":
        return om.layer_step_conv(w["x"], w["w"], w["gamma"], w["gy"], w["stride"], w["pad"], w["bits_s"],
                                  w["mode_s"], w["seed_s"], w["bits_c"], w["mode_c"], w["seed_c"])
    return om.layer_step_linear(w["x"], w["w"], w["gamma"], w["gy"], w["bits_s"], w["mode_s"], w["seed_s"],
                                w["bits_c"], w["mode_c"], w["seed_c"], w["rows_per_group"])


def assert_dequant_close(gpu, ref, a_mag, c_mag, what):
    tol = 1e-5 * (a_mag + c_mag) + 1e-30
    err = np.abs(gpu.astype(np.float64) - ref.astype(np.float64))
    bad = err > tol
    assert not bad.any(), f"{what}: {bad.sum()} elements out of tolerance, max err {err.max()}"


def check_branch(gq, rq, code_len, rpg, what):
    n = gq.n
    assert np.array_equal(gq.group_min.cpu().numpy(), rq["z"]), what + " Z"
    assert np.array_equal(gq.group_range.cpu().numpy(), rq["r"]), what + " R"
    assert np.array_equal(gq.p_hat.cpu().numpy(), rq["p_hat"]), what + " p_hat"
    cnt = gq.count()
    kept = rq["kept"]
    assert cnt == len(kept), what + " kept count"
    assert gq.kept_idx.cpu().numpy()[:cnt].tolist() == kept.tolist(), what + " kept ids"
    assert np.all(gq.kept_idx.cpu().numpy()[cnt:gq.capacity] == -1)
    slots = np.full(n, -1)
    slots[kept] = np.arange(len(kept))
    assert np.array_equal(gq.slot_of_group.cpu().numpy(), slots), what + " slots"
    assert np.array_equal(gq.scale.cpu().numpy()[:cnt], rq["scale"]), what + " scale"
    assert np.array_equal(gq.zero.cpu().numpy()[:cnt], rq["zero"]), what + " zero"
    codes = gq.codes.cpu().numpy()[: cnt * rpg, :code_len].astype(np.int64)
    assert np.array_equal(codes, rq["codes"]), what + " codes"


def check_step(w, st, ref):
    M, K, D, rpg = st.M, st.K, st.D, st.rpg
    x_u = ref["x_u"] if w["kind"] == "conv" else w["x"]
    w_u = w["w"].reshape(D, -1)
    if st.implicit:  # implicit-GEMM forward: pixel-major sign(X), tap-major sign(W)
        sp, pad_bits = unpack_bits(st.x_pix, w["x"].shape[1])
        assert np.array_equal(sp, om.pixel_signs(w["x"])) and not pad_bits.any(), "sign(X) pixel bits"
        swt, pad_bits = unpack_bits(st.w_taps, K)
        assert np.array_equal(swt, om.tap_major_signs(w["w"])) and not pad_bits.any(), "sign(W) tap-major bits"
    elif st.e4m3_x:  # e4m3 bytes of sign(X_u): 0x38 (+1), 0xB8 (-1), zeros to the next 16 bytes
        xr, pad_r = unpack_e4m3(st.x8_row, K)
        assert np.array_equal(xr, om.sign(x_u)) and not pad_r.any(), "sign(X) e4m3 rows"
        sw, _ = unpack_bits(st.sw_row, K)
        assert np.array_equal(sw, om.sign(w_u)), "sign(W) row bits"
    else:
        sx, pad_bits = unpack_bits(st.sx_row, K)
        assert np.array_equal(sx, om.sign(x_u)) and not pad_bits.any(), "sign(X) row bits"
        sw, _ = unpack_bits(st.sw_row, K)
        assert np.array_equal(sw, om.sign(w_u)), "sign(W) row bits"
    if st.e4m3_x:
        xc, pad_c = unpack_e4m3(st.x8_col, M)
        assert np.array_equal(xc, om.sign(x_u).T) and not pad_c.any(), "sign(X) e4m3 columns"
    else:
        sxc, pad_bits = unpack_bits(st.sx_col, M)
        assert np.array_equal(sxc, om.sign(x_u).T) and not pad_bits.any(), "sign(X) col bits"
    swc, _ = unpack_bits(st.sw_col, D)
    assert np.array_equal(swc, om.sign(w_u).T), "sign(W) col bits"
    assert np.array_equal(st.cs_x.cpu().numpy(), om.colsum_sign(x_u)), "colsum X"
    assert np.array_equal(st.cs_w.cpu().numpy(), om.colsum_sign(w_u)), "colsum W"
    assert np.array_equal(st.acc_y.cpu().numpy(), ref["acc_y"]), "forward acc"
    assert np.array_equal(st.y.cpu().numpy(), ref["y"]), "forward y"
    assert int(st.dev_status[0].item()) == 0
    check_branch(st.psq, ref["psq"], D, rpg, "PSQ")
    check_branch(st.pcq, ref["pcq"], M, 1, "PCQ")
    cnt_s = st.psq.count()
    assert np.array_equal(st.acc_dx.cpu().numpy()[: cnt_s * rpg], ref["acc_dx"]), "grad_input acc"
    cnt_c = st.pcq.count()
    assert np.array_equal(st.acc_dw.cpu().numpy()[:cnt_c], ref["acc_dw"]), "grad_weight acc"
    psq, pcq = ref["psq"], ref["pcq"]
    # magnitudes of the two dequantization terms
    if w["kind"] == "conv":
        N = w["x"].shape[0]
        a_mag = np.zeros(ref["dx"].shape)
        c_mag = np.zeros(ref["dx"].shape)
        for s_, g in enumerate(psq["kept"]):
            a_mag[g] = np.abs(np.float64(psq["scale"][s_]) * ref["acc_fold"][g])
            c_mag[g] = np.abs(np.float64(psq["zero"][s_]) * ref["cs_fold"])
        assert ref["dx"].shape == (N,) + tuple(w["x"].shape[1:])
    else:
        a_mag = np.zeros((M, K))
        c_mag = np.zeros((M, K))
        cs = om.colsum_sign(w_u)
        for s_, g in enumerate(psq["kept"]):
            rows = slice(g * rpg, (g + 1) * rpg)
            a_mag[rows] = np.abs(np.float64(psq["scale"][s_]) * ref["acc_dx"][s_ * rpg:(s_ + 1) * rpg])
            c_mag[rows] = np.abs(np.float64(psq["zero"][s_]) * cs)[None, :]
    assert_dequant_close(st.dx.cpu().numpy(), ref["dx"], a_mag, c_mag, "grad_input")
    aw = np.zeros((D, K))
    cw = np.zeros((D, K))
    csx = om.colsum_sign(x_u)
    for s_, j in enumerate(pcq["kept"]):
        aw[j] = np.abs(np.float64(pcq["scale"][s_]) * ref["acc_dw"][s_])
        cw[j] = np.abs(np.float64(pcq["zero"][s_]) * csx)
    assert_dequant_close(st.dw.cpu().numpy().reshape(D, K), ref["dw"].reshape(D, K), aw, cw, "grad_weight")


CASES = [
    ("linear-64x512x512-b2", lambda: wl.linear_small()),
    ("conv-resnet18-cifar-8192x2304x256-b4", lambda: wl.resnet18_cifar_conv()),
    ("linear-ragged-b4", lambda: linear_case(40, 33, 10, 4, 4, SYS)),
    ("linear-b8-bernoulli", lambda: linear_case(96, 200, 100, 1, 8, BER, seed=3)),
    ("linear-oddD-b1", lambda: linear_case(50, 70, 30, 5, 1, SYS, seed=4)),
    ("linear-n-lt-b", lambda: linear_case(3, 64, 16, 1, 8, SYS, seed=5)),
    ("linear-single-group-topk", lambda: linear_case(64, 96, 48, 64, 2, TOP, seed=6, gamma=False)),
    ("linear-mixed-bits", lambda: linear_case(128, 300, 64, 2, 4, SYS, seed=7, bits_c=2, mode_c=BER)),
    ("conv-ragged-s2-topk", lambda: conv_case(3, 5, 7, 6, 12, 3, 2, 1, 2, TOP)),
    ("conv-7x7-s2-b4", lambda: conv_case(2, 3, 20, 20, 16, 7, 2, 3, 4, SYS, seed=1)),
    ("conv-1x1-s2-b8", lambda: conv_case(4, 8, 9, 9, 24, 1, 2, 0, 8, SYS, seed=2)),
    # region of a 256-column tile too large for the bit-level Unfolder: the generic gather path
    ("conv-1x1-256ch-56x56-gather", lambda: conv_case(2, 256, 56, 56, 16, 1, 1, 0, 4, SYS, seed=3)),
    ("conv-3x3-s1-multi-image-tiles", lambda: conv_case(9, 20, 5, 7, 40, 3, 1, 1, 2, BER, seed=4)),
    ("conv-5x5-s3-p2", lambda: conv_case(3, 6, 17, 13, 8, 5, 3, 2, 4, SYS, seed=5)),
    # "same" convolutions whose tiles hold whole images (contiguous-region Unfolder):
    # ragged last image tile and last column tile, 16x16 planes (256-pixel tiles), 1x1,
    # 7x7 with pad 3, and rows wider than 32 pixels (per-sub-tile column masks)
    ("conv-same-8x8-ragged", lambda: conv_case(5, 30, 8, 8, 24, 3, 1, 1, 4, SYS, seed=6)),
    ("conv-same-16x16-5x5", lambda: conv_case(3, 12, 16, 16, 20, 5, 1, 2, 2, BER, seed=7)),
    ("conv-same-4x8-1x1", lambda: conv_case(7, 300, 4, 8, 16, 1, 1, 0, 8, SYS, seed=8)),
    ("conv-same-8x16-7x7", lambda: conv_case(3, 4, 8, 16, 8, 7, 1, 3, 4, SYS, seed=9)),
    ("conv-same-4x64", lambda: conv_case(2, 6, 4, 64, 8, 3, 1, 1, 2, SYS, seed=10)),
    # implicit-GEMM forward (C a multiple of 128): a ragged last tile of whole images, tiles of
    # image rows, 1x1 with 8 images per tile, and 5x5 taps over 32-pixel rows with a partial
    # last contraction stage (K = 3200)
    ("conv-implicit-8x8-ragged", lambda: conv_case(5, 128, 8, 8, 48, 3, 1, 1, 4, SYS, seed=12)),
    ("conv-implicit-16x16-rows", lambda: conv_case(2, 128, 16, 16, 40, 3, 1, 1, 2, BER, seed=13)),
    ("conv-implicit-4x4-1x1", lambda: conv_case(9, 256, 4, 4, 24, 1, 1, 0, 8, SYS, seed=14)),
    ("conv-implicit-32x32-5x5", lambda: conv_case(1, 128, 32, 32, 16, 5, 1, 2, 4, SYS, seed=15)),
]


@pytest.mark.parametrize("name,make", CASES, ids=[c[0] for c in CASES])
def test_layer_step_parity(name, make):
    from paper_2408_14267_gb300.layer import LayerStep
    w = make()
    ref = run_oracle(w)
    st = LayerStep(w, implicit="implicit" in name)
    if "implicit" in name:
        assert st.implicit
    st.dev_status.zero_()
    st.step()
    torch.cuda.synchronize()
    check_step(w, st, ref)
    # a second step on the same buffers reproduces the first (no state leaks between calls)
    y0, dx0, dw0 = st.y.clone(), st.dx.clone(), st.dw.clone()
    st.step()
    torch.cuda.synchronize()
    assert torch.equal(st.y, y0) and torch.equal(st.dx, dx0) and torch.equal(st.dw, dw0)


LINEAR_CASES = [c for c in CASES if c[0].startswith("linear")]


@pytest.mark.parametrize("name,make", [CASES[1], CASES[-4]], ids=[CASES[1][0], CASES[-4][0]])
def test_implicit_and_unfolded_forward_steps_agree(name, make):
    """The bench layer with the implicit forward and an implicit case with it switched off
    (materialized 1-bit unfolding, row-packed operands) both match the oracle's step."""
    from paper_2408_14267_gb300.layer import LayerStep
    w = make()
    ref = run_oracle(w)
    want = "implicit" not in name
    st = LayerStep(w, implicit=want)
    assert st.implicit == want
    st.dev_status.zero_()
    st.step()
    torch.cuda.synchronize()
    check_step(w, st, ref)

FOLD_CASES = [
    ("fold-resnet18-cifar-8192x2304x256-b4", lambda: wl.resnet18_cifar_conv()),
    ("fold-4x4-3x3-8-samples-per-tile", lambda: conv_case(6, 10, 4, 4, 20, 3, 1, 1, 4, SYS, seed=7)),
    ("fold-8x8-b8", lambda: conv_case(5, 40, 8, 8, 24, 3, 1, 1, 8, SYS, seed=8)),
    ("fold-2x2-topk", lambda: conv_case(40, 16, 2, 2, 8, 3, 1, 1, 2, TOP, seed=9)),
    ("fold-5x5-kernel-4x4-map", lambda: conv_case(5, 30, 4, 4, 16, 5, 1, 2, 4, BER, seed=10)),
    ("fold-stride2-16x16-to-8x8", lambda: conv_case(3, 12, 16, 16, 32, 3, 2, 1, 4, SYS, seed=11)),
]


@pytest.mark.parametrize("name,make", FOLD_CASES, ids=[c[0] for c in FOLD_CASES])
def test_conv_fold_parity(name, make):
    """grad_input with the Folder fused into the product equals the oracle's folded gradient."""
    from paper_2408_14267_gb300.layer import LayerStep
    w = make()
    ref = run_oracle(w)
    st = LayerStep(w, keep_acc=False)
    assert st.fold
    st.step()
    torch.cuda.synchronize()
    psq = ref["psq"]
    a_mag = np.zeros(ref["dx"].shape)
    c_mag = np.zeros(ref["dx"].shape)
    for s_, g in enumerate(psq["kept"]):
        a_mag[g] = np.abs(np.float64(psq["scale"][s_]) * ref["acc_fold"][g])
        c_mag[g] = np.abs(np.float64(psq["zero"][s_]) * ref["cs_fold"])
    assert_dequant_close(st.dx.cpu().numpy(), ref["dx"], a_mag, c_mag, "grad_input (fold)")
    dx = st.dx.cpu().numpy()
    for g in np.setdiff1d(np.arange(w["x"].shape[0]), psq["kept"]):
        assert np.all(dx[g] == 0)
    assert np.array_equal(st.y.cpu().numpy(), ref["y"])


@pytest.mark.parametrize("name,make", LINEAR_CASES, ids=[c[0] for c in LINEAR_CASES])
def test_linear_fused_dequant_parity(name, make):
    """Without the int32 copy, grad_input is dequantized in the GEMM epilogue; same results."""
    from paper_2408_14267_gb300.layer import LayerStep
    w = make()
    ref = run_oracle(w)
    st = LayerStep(w, keep_acc=False)
    st.step()
    torch.cuda.synchronize()
    assert np.array_equal(st.y.cpu().numpy(), ref["y"])
    a_mag = np.zeros(ref["dx"].shape)
    c_mag = np.zeros(ref["dx"].shape)
    psq, rpg = ref["psq"], st.rpg
    cs = om.colsum_sign(w["w"])
    for s_, g in enumerate(psq["kept"]):
        rows = slice(g * rpg, (g + 1) * rpg)
        a_mag[rows] = np.abs(np.float64(psq["scale"][s_]) * ref["acc_dx"][s_ * rpg:(s_ + 1) * rpg])
        c_mag[rows] = np.abs(np.float64(psq["zero"][s_]) * cs)[None, :]
    assert_dequant_close(st.dx.cpu().numpy(), ref["dx"], a_mag, c_mag, "grad_input (fused)")
    pruned = np.setdiff1d(np.arange(st.M // rpg), psq["kept"])
    dx = st.dx.cpu().numpy()
    for g in pruned:
        assert np.all(dx[g * rpg:(g + 1) * rpg] == 0)


@pytest.mark.parametrize("name,make", [CASES[0], CASES[1], CASES[9]], ids=[CASES[0][0], CASES[1][0], CASES[9][0]])
def test_concurrent_step_matches_serial(name, make):
    """The three-branch schedule (also captured in a CUDA graph) gives the serial step's results."""
    from paper_2408_14267_gb300.layer import LayerStep
    w = make()
    a = LayerStep(w, keep_acc=False)
    a.step()
    b = LayerStep(w, keep_acc=False)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        b.step_concurrent(s)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            b.step_concurrent(s)
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(a.y, b.y) and torch.equal(a.dx, b.dx) and torch.equal(a.dw, b.dw)


def test_single_branch_entry_point_matches_scq():
    """fqt1_agp_quantize_grad on one axis equals that branch of fqt1_scq_quantize."""
    from paper_2408_14267_gb300 import fqt1
    from paper_2408_14267_gb300.layer import LayerStep
    w = linear_case(64, 32, 40, 2, 4, SYS, seed=9)
    st = LayerStep(w)
    st.backward()
    for axis, ref in ((0, st.psq), (1, st.pcq)):
        n = st.M // st.rpg if axis == 0 else st.D
        p = st.p_s if axis == 0 else st.p_c
        rows = ref.capacity * (st.rpg if axis == 0 else 1)
        q = fqt1.QGradBuffers(n, ref.capacity, rows, st.D if axis == 0 else st.M)
        fqt1.agp_quantize_grad(st.gy, st.M, st.D, axis, st.gamma, p, q, st.ws, st.dev_status)
        torch.cuda.synchronize()
        c = ref.count()
        assert q.count() == c
        assert torch.equal(q.codes[:rows], ref.codes[:rows]) and torch.equal(q.p_hat, ref.p_hat)


def test_workspace_keys_restored_after_each_call():
    """Every quantizer call leaves its range keys at the 0xFF of fqt1_scq_workspace_init
    (the selection kernel resets each key it reads), so one workspace, initialised once,
    gives the results of a fresh one on repeated calls, other shapes and single branches."""
    from paper_2408_14267_gb300 import fqt1
    from paper_2408_14267_gb300 import workloads as wl
    from paper_2408_14267_gb300.layer import LayerStep
    steps = [LayerStep(wl.resnet18_cifar_conv()), LayerStep(wl.linear_small()),
             LayerStep(linear_case(100, 48, 72, 4, 2, SYS, seed=11))]
    ws = fqt1.scq_workspace(max(s.M for s in steps), max(s.D for s in steps), 0, 1, "cuda")

    def initialised(w):  # range keys 0xFF
        return bool((w == 255).all())

    def same(a, b, rows):
        c = a.count()
        assert c == b.count()
        for name in ("group_min", "group_range", "p_hat", "slot_of_group"):
            assert torch.equal(getattr(a, name), getattr(b, name)), name
        assert torch.equal(a.scale[:c], b.scale[:c]) and torch.equal(a.zero[:c], b.zero[:c])
        assert torch.equal(a.codes[: c * rows], b.codes[: c * rows])

    for st in steps + steps[:1]:
        st.dev_status.zero_()
        fqt1.scq_quantize(st.gy, st.M, st.D, st.gamma, st.p_s, st.p_c, st.psq, st.pcq, st.ws, st.dev_status)
        psq = fqt1.QGradBuffers(st.psq.n, st.psq.capacity, st.psq.capacity * st.rpg, st.D)
        pcq = fqt1.QGradBuffers(st.pcq.n, st.pcq.capacity, st.pcq.capacity, st.M)
        fqt1.scq_quantize(st.gy, st.M, st.D, st.gamma, st.p_s, st.p_c, psq, pcq, ws, st.dev_status)
        torch.cuda.synchronize()
        assert initialised(ws) and initialised(st.ws)
        same(psq, st.psq, st.rpg)
        same(pcq, st.pcq, 1)
        q = fqt1.QGradBuffers(st.pcq.n, st.pcq.capacity, st.pcq.capacity, st.M)
        fqt1.agp_quantize_grad(st.gy, st.M, st.D, 1, st.gamma, st.p_c, q, ws, st.dev_status)
        torch.cuda.synchronize()
        assert initialised(ws)
        same(q, st.pcq, 1)


@pytest.mark.parametrize("M,D,rpg,bits,mode", [(8192, 256, 64, 4, SYS), (250, 100, 5, 8, BER), (1024, 256, 4, 2, SYS),
                                              (60, 16, 60, 2, TOP)])
def test_scq_matches_single_branch_calls(M, D, rpg, bits, mode):
    """One fqt1_scq_quantize call (both groupings from one range pass and one rounding pass)
    equals two single-branch fqt1_agp_quantize_grad calls bit for bit, all outputs, also for M
    not a multiple of 4 (per-word rounding draws) and for every mask law."""
    from paper_2408_14267_gb300 import fqt1
    rng = np.random.default_rng(M + D)
    s_ = 10.0 ** rng.uniform(-2, 2, size=(M // rpg, 1, 1))
    g = torch.from_numpy((rng.laplace(0, 1e-3, (M // rpg, rpg, D)) * s_).reshape(M, D).astype(np.float32)).cuda()
    gamma = torch.from_numpy(rng.uniform(0.5, 2.0, D).astype(np.float32)).cuda()
    p_s, p_c = fqt1.AgpParams(bits, mode, 31, rpg), fqt1.AgpParams(bits, mode, 32, 1)
    cap_s, cap_c = fqt1.kept_capacity(M // rpg, bits, mode), fqt1.kept_capacity(D, bits, mode)
    bufs = lambda: (fqt1.QGradBuffers(M // rpg, cap_s, cap_s * rpg, D), fqt1.QGradBuffers(D, cap_c, cap_c, M))
    ws = fqt1.scq_workspace(M, D, 0, rpg, "cuda")
    st = torch.zeros(4, dtype=torch.int32, device="cuda")
    psq, pcq = bufs()
    for q in (psq, pcq):
        q.codes.fill_(0x5A)
    fqt1.scq_quantize(g, M, D, gamma, p_s, p_c, psq, pcq, ws, st)
    rs, rc = bufs()
    for q in (rs, rc):
        q.codes.fill_(0x5A)
    fqt1.agp_quantize_grad(g, M, D, 0, gamma, p_s, rs, ws, st)
    fqt1.agp_quantize_grad(g, M, D, 1, gamma, p_c, rc, ws, st)
    torch.cuda.synchronize()
    assert int(st[0].item()) == 0
    assert bool((ws == 255).all())
    for a, b in ((psq, rs), (pcq, rc)):
        for name in ("group_min", "group_range", "p_hat", "slot_of_group", "kept_idx", "kept_count", "codes"):
            assert torch.equal(getattr(a, name), getattr(b, name)), name
        c = a.count()
        assert torch.equal(a.scale[:c], b.scale[:c]) and torch.equal(a.zero[:c], b.zero[:c])


@pytest.mark.parametrize("rows,n", [(3, 5), (256, 2304), (17, 128), (40, 300), (1, 16), (70, 44), (33, 1000)])
def test_binarize_pack_e4m3_bytes(rows, n):
    """e4m3 bytes of the signs from the sign-pack pass (tile path for rows of a multiple of 4
    floats, packing + expansion otherwise) and from the expansion of packed signs: 0x38 for
    +1, 0xB8 for -1, zeros past the data, both orientations; the packed outputs unchanged."""
    from paper_2408_14267_gb300 import fqt1
    rng = np.random.default_rng(rows * 3 + n)
    x = rng.standard_normal((rows, n)).astype(np.float32)
    x[-1, -1] = 0.0
    xt = torch.from_numpy(x).cuda()
    rb = torch.empty(rows, fqt1.packed_words(n), dtype=torch.int32, device="cuda")
    cbits = torch.empty(n, fqt1.packed_words(rows), dtype=torch.int32, device="cuda")
    cs = torch.empty(n, dtype=torch.int32, device="cuda")
    re = torch.full((rows, fqt1.codes_ld(n)), 0x5A, dtype=torch.uint8, device="cuda")
    ce = torch.full((n, fqt1.codes_ld(rows)), 0x5A, dtype=torch.uint8, device="cuda")
    fqt1.binarize_pack_e4m3(xt, rows, n, n, rb, cbits, cs, re, ce)
    torch.cuda.synchronize()
    sgn = np.where(om.sign(x) > 0, 0x38, 0xB8).astype(np.uint8)
    r_, c_ = re.cpu().numpy(), ce.cpu().numpy()
    assert np.array_equal(r_[:, :n], sgn) and not r_[:, n:].any()
    assert np.array_equal(c_[:, :rows], sgn.T) and not c_[:, rows:].any()
    bits, _ = unpack_bits(rb, n)
    assert np.array_equal(bits, om.sign(x))
    assert np.array_equal(cs.cpu().numpy(), om.colsum_sign(x))


@pytest.mark.parametrize("rows,n", [(3, 5), (256, 2304), (17, 128), (40, 300), (1, 16)])
def test_expand_signs_e4m3_bytes(rows, n):
    """Packed signs -> e4m3 bytes: 0x38 for +1, 0xB8 for -1, zeros past the n columns."""
    from paper_2408_14267_gb300 import fqt1
    rng = np.random.default_rng(rows * 7 + n)
    x = rng.standard_normal((rows, n)).astype(np.float32)
    x[0, 0] = 0.0
    bits = torch.empty(rows, fqt1.packed_words(n), dtype=torch.int32, device="cuda")
    fqt1.binarize_pack(torch.from_numpy(x).cuda(), rows, n, n, bits, None, None)
    out = torch.full((rows, fqt1.codes_ld(n)), 0x5A, dtype=torch.uint8, device="cuda")
    fqt1.expand_signs_e4m3(bits, rows, n, out)
    torch.cuda.synchronize()
    o = out.cpu().numpy()
    assert np.array_equal(o[:, :n], np.where(om.sign(x) > 0, 0x38, 0xB8).astype(np.uint8))
    assert not o[:, n:].any()


@pytest.mark.parametrize("M,K,D,bias", [(8192, 2304, 256, False), (300, 200, 136, True), (64, 512, 512, True),
                                        (129, 1000, 40, False)])
def test_fwd_e4m3_weights_equal_packed(M, K, D, bias):
    """The forward product with sign(W) as e4m3 bytes loaded by TMA equals the packed-bit
    product bit for bit (acc and y), with ragged K, D and M."""
    from paper_2408_14267_gb300 import fqt1
    rng = np.random.default_rng(M + K + D)
    x = torch.from_numpy(rng.standard_normal((M, K)).astype(np.float32)).cuda()
    w = torch.from_numpy(rng.standard_normal((D, K)).astype(np.float32)).cuda()
    g = torch.from_numpy(rng.uniform(0.5, 2.0, D).astype(np.float32)).cuda()
    b = torch.from_numpy(rng.standard_normal(D).astype(np.float32)).cuda() if bias else None
    pk = lambda r: torch.empty(r, fqt1.packed_words(K), dtype=torch.int32, device="cuda")
    sx, sw = pk(M), pk(D)
    fqt1.binarize_pack(x, M, K, K, sx, None, None)
    fqt1.binarize_pack(w, D, K, K, sw, None, None)
    w8 = torch.empty(D, fqt1.codes_ld(K), dtype=torch.uint8, device="cuda")
    fqt1.expand_signs_e4m3(sw, D, K, w8)
    acc0, y0 = torch.empty(M, D, dtype=torch.int32, device="cuda"), torch.empty(M, D, device="cuda")
    acc1, y1 = torch.full((M, D), 3, dtype=torch.int32, device="cuda"), torch.full((M, D), 3.0, device="cuda")
    fqt1.fwd_gemm_bias(sx, sw, M, D, K, g, b, acc0, y0)
    fqt1.fwd_gemm_e4m3w(sx, w8, M, D, K, g, b, acc1, y1)
    torch.cuda.synchronize()
    assert torch.equal(acc0, acc1) and torch.equal(y0, y1)
    acc_ref, _ = om.forward(x.cpu().numpy(), w.cpu().numpy(), None)
    assert np.array_equal(acc1.cpu().numpy(), acc_ref)


@pytest.mark.parametrize("name,make", [CASES[1], FOLD_CASES[1], FOLD_CASES[2], FOLD_CASES[5]],
                         ids=[CASES[1][0], FOLD_CASES[1][0], FOLD_CASES[2][0], FOLD_CASES[5][0]])
def test_e4m3_weights_step_equals_packed_step(name, make):
    """A whole step with the e4m3 copies of sign(W) (forward and fused Folder products) equals
    the step on packed signs bit for bit."""
    from paper_2408_14267_gb300.layer import LayerStep
    w = make()
    a = LayerStep(w, keep_acc=False, e4m3_weights=True)
    b = LayerStep(w, keep_acc=False)
    assert a.w8 is not None and b.w8 is None
    for st in (a, b):
        st.dev_status.zero_()
        st.step()
    torch.cuda.synchronize()
    assert torch.equal(a.y, b.y) and torch.equal(a.dx, b.dx) and torch.equal(a.dw, b.dw)


E4M3X_CASES = [c for c in CASES if c[0] in ("linear-64x512x512-b2", "conv-resnet18-cifar-8192x2304x256-b4",
                                             "conv-same-8x8-ragged", "conv-same-16x16-5x5", "conv-same-4x8-1x1",
                                             "conv-same-8x16-7x7", "conv-same-4x64", "linear-b8-bernoulli",
                                             "linear-mixed-bits")]


@pytest.mark.parametrize("name,make", E4M3X_CASES, ids=[c[0] for c in E4M3X_CASES])
def test_e4m3_x_step_parity(name, make):
    """The step with e4m3 copies of sign(X_u) (the Unfolder's byte output, both products' sign
    operand straight from TMA) against the oracle: bytes, integer sums and outputs."""
    from paper_2408_14267_gb300.layer import LayerStep
    w = make()
    ref = run_oracle(w)
    st = LayerStep(w, keep_acc=True, fold=False, e4m3_x=True)
    assert st.e4m3_x and st.sx_row is None and st.sx_col is None
    st.dev_status.zero_()
    st.step()
    torch.cuda.synchronize()
    check_step(w, st, ref)


@pytest.mark.parametrize("name,make", [CASES[1], CASES[0], FOLD_CASES[2]], ids=[CASES[1][0], CASES[0][0],
                                                                             FOLD_CASES[2][0]])
def test_e4m3_x_step_equals_packed_step(name, make):
    """The benchmark's configuration (fused Folder, no int32 copies) with and without the e4m3
    copies of sign(X_u): identical y, dx and dW."""
    from paper_2408_14267_gb300.layer import LayerStep
    w = make()
    a = LayerStep(w, keep_acc=False, e4m3_weights=True, e4m3_x=True)
    b = LayerStep(w, keep_acc=False)
    assert a.e4m3_x and not b.e4m3_x
    for st in (a, b):
        st.dev_status.zero_()
        st.step()
    torch.cuda.synchronize()
    assert torch.equal(a.y, b.y) and torch.equal(a.dx, b.dx) and torch.equal(a.dw, b.dw)


def test_nonfinite_gradient_sets_status():
    from paper_2408_14267_gb300.layer import LayerStep
    w = linear_case(32, 32, 16, 1, 2, SYS, seed=10)
    w["gy"][5, 3] = np.nan
    st = LayerStep(w)
    st.dev_status.zero_()
    st.backward()
    torch.cuda.synchronize()
    assert int(st.dev_status[0].item()) & 0x100


@pytest.mark.parametrize("val", [float("-inf"), float("inf")])
def test_infinite_gradient_stays_in_bounds(val):
    """An infinite gradient value gives an infinite range, which breaks the fixed-point keep
    probabilities (every group would be kept).  The step must still flag the input, keep at
    most `capacity` groups per branch, and keep every kept id and slot in range."""
    from paper_2408_14267_gb300.layer import LayerStep
    w = linear_case(64, 64, 64, 1, 4, SYS, seed=12)
    w["gy"][5, 3] = val
    st = LayerStep(w)
    st.dev_status.zero_()
    st.step()
    torch.cuda.synchronize()
    assert int(st.dev_status[0].item()) & 0x100
    for q in (st.psq, st.pcq):
        cnt = q.count()
        assert 0 <= cnt <= q.capacity
        kid = q.kept_idx.cpu().numpy()
        assert np.all((kid[:cnt] >= 0) & (kid[:cnt] < q.n)) and np.all(kid[cnt:q.capacity] == -1)
        slots = q.slot_of_group.cpu().numpy()
        assert np.all((slots >= -1) & (slots < cnt))


@pytest.mark.parametrize("rows,cols,ld", [(77, 300, 304), (40, 128, 132), (3, 4, 8), (64, 256, 256), (33, 100, 103),
                                          (70, 45, 45)])
def test_binarize_pack_strided(rows, cols, ld):
    """Row bits, column bits and column sums of sign(x) for a strided [rows, cols] view (Sec. 5.1):
    rows of a multiple of 4 floats take the shared-memory tile path, the others the per-warp path."""
    from paper_2408_14267_gb300 import fqt1
    rng = np.random.default_rng(rows * 1000 + cols)
    full = rng.standard_normal((rows, ld)).astype(np.float32)
    full[:, :cols][rng.random((rows, cols)) < 0.05] = 0.0
    x = full[:, :cols]
    dev = torch.from_numpy(full).cuda()
    rw, cw = fqt1.packed_words(cols), fqt1.packed_words(rows)
    row_bits = torch.full((rows, rw), -1, dtype=torch.int32, device="cuda")
    col_bits = torch.full((cols, cw), -1, dtype=torch.int32, device="cuda")
    colsum = torch.full((cols,), 12345, dtype=torch.int32, device="cuda")
    fqt1.binarize_pack(dev, rows, cols, ld, row_bits, col_bits, colsum)
    torch.cuda.synchronize()
    s, pad = unpack_bits(row_bits, cols)
    assert np.array_equal(s, om.sign(x)) and not pad.any()
    sc, pad = unpack_bits(col_bits, rows)
    assert np.array_equal(sc, om.sign(x).T) and not pad.any()
    assert np.array_equal(colsum.cpu().numpy(), om.colsum_sign(x))


@pytest.mark.parametrize("M,K,N", [(512, 512, 512), (1024, 512, 1024), (2048, 512, 512)])
def test_table5_shapes_exact(M, K, N):
    """The two products bench.py --table5 times, on Table 5 shapes: sign(A) sign(B)^T (1-bit) and
    the kept quarter of A's rows as 4-bit codes times sign(B)^T (average 1-bit), int32 exact."""
    from paper_2408_14267_gb300 import fqt1
    rng = np.random.default_rng(M + N)
    a = rng.standard_normal((M, K)).astype(np.float32)
    b = rng.standard_normal((N, K)).astype(np.float32)
    g = (rng.standard_normal((M, K)) * np.exp(2 * rng.standard_normal((M, 1)))).astype(np.float32)
    dev = torch.device("cuda")
    wK = fqt1.packed_words(K)
    sa = torch.empty(M, wK, dtype=torch.int32, device=dev)
    sb = torch.empty(N, wK, dtype=torch.int32, device=dev)
    fqt1.binarize_pack(torch.from_numpy(a).cuda(), M, K, K, sa, None, None)
    fqt1.binarize_pack(torch.from_numpy(b).cuda(), N, K, K, sb, None, None)
    acc1 = torch.empty(M, N, dtype=torch.int32, device=dev)
    y = torch.empty(M, N, device=dev)
    fqt1.fwd_gemm(sa, sb, M, N, K, torch.ones(N, device=dev), acc1, y)
    assert np.array_equal(acc1.cpu().numpy(), om.int_matmul(om.sign(a), om.sign(b)))
    p = fqt1.AgpParams(4, SYS, 11, 1)
    cap = fqt1.kept_capacity(M, 4, SYS)
    q = fqt1.QGradBuffers(M, cap, cap, K, dev)
    ws = fqt1.scq_workspace(M, K, N, 1, dev)
    status = torch.zeros(4, dtype=torch.int32, device=dev)
    fqt1.agp_quantize_grad(torch.from_numpy(g).cuda(), M, K, 0, None, p, q, ws, status)
    acc4 = torch.empty(cap, N, dtype=torch.int32, device=dev)
    fqt1.bwd_input_gemm(q, sb, None, M, K, N, p, acc4, None)
    ref = om.agp_quantize(g, 0, 1, 4, SYS, 11)
    cnt = q.count()
    assert cnt == len(ref["kept"])
    assert np.array_equal(acc4.cpu().numpy()[:cnt], om.int_matmul(ref["codes"], om.sign(b)))


@pytest.mark.parametrize("M,K,D", [(300, 1000, 64), (257, 129, 70), (128, 2304, 256)])
def test_fwd_acc_only(M, K, D):
    """fqt1_fwd_gemm with y = NULL (and no Gamma) writes the int32 accumulators alone, on the
    tensor-core kernel: exact against the oracle (TMA stores when D is a multiple of 4, direct
    stores otherwise)."""
    from paper_2408_14267_gb300 import fqt1
    rng = np.random.default_rng(M * 7 + D)
    a = rng.standard_normal((M, K)).astype(np.float32)
    b = rng.standard_normal((D, K)).astype(np.float32)
    dev = torch.device("cuda")
    wK = fqt1.packed_words(K)
    sa = torch.empty(M, wK, dtype=torch.int32, device=dev)
    sb = torch.empty(D, wK, dtype=torch.int32, device=dev)
    fqt1.binarize_pack(torch.from_numpy(a).cuda(), M, K, K, sa, None, None)
    fqt1.binarize_pack(torch.from_numpy(b).cuda(), D, K, K, sb, None, None)
    acc = torch.full((M, D), 7777, dtype=torch.int32, device=dev)
    n0 = fqt1.kernel_launches()
    fqt1.fwd_gemm(sa, sb, M, D, K, None, acc, None)
    torch.cuda.synchronize()
    assert fqt1.kernel_launches() == n0 + 1
    assert np.array_equal(acc.cpu().numpy(), om.int_matmul(om.sign(a), om.sign(b)))


@pytest.mark.parametrize("name,make", [CASES[0], CASES[1]], ids=[CASES[0][0], CASES[1][0]])
def test_host_copy_step_matches_serial(name, make):
    """The step with its host copies (LayerStep.step_concurrent_host, the end-to-end form) gives
    the outputs of the serial step bit for bit, from inputs that reach the device only through
    its copies."""
    from paper_2408_14267_gb300.layer import LayerStep
    w = make()
    st = LayerStep(w, keep_acc=False)
    st.step()
    torch.cuda.synchronize()
    ref = [t.clone() for t in (st.y, st.dx, st.dw)]
    h_in = [t.detach().cpu().pin_memory() for t in (st.x, st.w, st.gy)]
    if st.gamma is not None:
        h_in.append(st.gamma.detach().cpu().pin_memory())
    for t in (st.x, st.w, st.gy, st.y, st.dx, st.dw):
        t.zero_()
    h_out = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in ref]
    st.step_concurrent_host(h_in, h_out)
    torch.cuda.synchronize()
    for h, r, what in zip(h_out, ref, ("y", "dx", "dw")):
        assert torch.equal(h, r.cpu()), what


@pytest.mark.parametrize("N,C,H,W,k,s,p", [(3, 64, 8, 8, 3, 1, 1), (2, 64, 32, 32, 3, 1, 1), (2, 32, 16, 16, 3, 2, 1),
                                           (2, 96, 7, 9, 3, 1, 1), (3, 64, 4, 4, 1, 1, 0), (2, 32, 20, 20, 7, 2, 3)])
def test_im2col_from_channels_last_planes(N, C, H, W, k, s, p):
    """Channels-last input: the plane bits equal the signs of x, and the Unfolder reading them
    writes the same rows, columns and column sums as the Unfolder reading x."""
    from paper_2408_14267_gb300 import fqt1
    rng = np.random.default_rng(N * C + H + k)
    x = rng.standard_normal((N, C, H, W)).astype(np.float32)
    x[0, :2, 0, 0] = 0.0
    xt = torch.from_numpy(x).cuda()
    xl = xt.contiguous(memory_format=torch.channels_last)
    pw = fqt1.plane_words(H, W)
    planes = torch.full((N * C * pw,), -1, dtype=torch.int32, device="cuda")
    fqt1.pack_planes_nhwc(xl, N, C, H, W, planes)
    Ho, Wo = om.conv_out_hw(H, W, k, k, s, p)
    M, K = N * Ho * Wo, C * k * k
    outs = []
    for use_planes in (False, True):
        rb = torch.full((M, fqt1.packed_words(K)), 7, dtype=torch.int32, device="cuda")
        cbits = torch.full((K, fqt1.packed_words(M)), 7, dtype=torch.int32, device="cuda")
        cs = torch.empty(K, dtype=torch.int32, device="cuda")
        if use_planes:
            fqt1.im2col_planes(planes, N, C, H, W, k, k, s, p, rb, cbits, cs)
        else:
            fqt1.im2col(xt, N, C, H, W, k, k, s, p, rb, cbits, cs)
        outs.append((rb, cbits, cs))
    torch.cuda.synchronize()
    w = planes.cpu().numpy().view(np.uint32).reshape(N, C, pw)
    bits = ((w[:, :, :, None] >> np.arange(32, dtype=np.uint32)) & 1).reshape(N, C, -1)
    assert np.array_equal(bits[:, :, :H * W].astype(np.int8) * 2 - 1, om.sign(x).reshape(N, C, H * W))
    assert not bits[:, :, H * W:].any()
    for a, b in zip(*outs):
        assert torch.equal(a, b)


@pytest.mark.parametrize("N,C,H,W,k,s,p", [(2, 3, 30, 30, 7, 2, 3), (2, 64, 28, 28, 1, 2, 0), (3, 16, 14, 14, 3, 2, 1),
                                           (2, 5, 13, 11, 3, 1, 1), (1, 32, 56, 56, 3, 1, 1), (4, 8, 9, 7, 1, 1, 0),
                                           (5, 37, 4, 4, 3, 1, 1), (9, 50, 2, 2, 3, 1, 1), (3, 11, 2, 4, 3, 1, 1),
                                           (3, 40, 15, 13, 1, 3, 0), (2, 33, 8, 9, 1, 1, 0), (5, 70, 7, 7, 1, 2, 0),
                                           (40, 70, 4, 4, 3, 1, 1), (70, 33, 2, 2, 3, 1, 1), (6, 45, 1, 1, 3, 1, 1),
                                           (9, 21, 1, 2, 3, 1, 1), (1, 29, 4, 4, 3, 1, 1)])
def test_pack_planes_nchw_and_unfold_from_planes(N, C, H, W, k, s, p):
    """Contiguous x: fqt1_pack_planes writes the signs of x as channel planes (any C, H W not a
    multiple of 32, bits past H W clear), and the Unfolder reading those planes writes the same
    rows, columns and column sums as the Unfolder reading x (the region-tile shape of the
    ResNet-18 stem, and the 1 x 1 downsamples, which the pointwise pass serves from x).  Maps of
    fewer than 32 pixels that divide 32 (4 x 4, 2 x 2, 1 x 2, 1 x 1): the Unfolder reading x takes
    each ballot over several whole planes; the cases span several row and column tiles, channel
    counts that leave a partial ballot per image, and a single image."""
    from paper_2408_14267_gb300 import fqt1
    rng = np.random.default_rng(N * C + H * 3 + k)
    x = rng.standard_normal((N, C, H, W)).astype(np.float32)
    x[0, 0, 0, :3] = 0.0
    xt = torch.from_numpy(x).cuda()
    pw = fqt1.plane_words(H, W)
    planes = torch.full((N * C * pw,), -1, dtype=torch.int32, device="cuda")
    fqt1.pack_planes(xt, N, C, H, W, planes)
    Ho, Wo = om.conv_out_hw(H, W, k, k, s, p)
    M, K = N * Ho * Wo, C * k * k
    path = fqt1.im2col_path(N, C, H, W, k, k, s, p)
    assert path in (1, 2, 3)
    outs = []
    for use_planes in (False, True):
        rb = torch.full((M, fqt1.packed_words(K)), 7, dtype=torch.int32, device="cuda")
        cbits = torch.full((K, fqt1.packed_words(M)), 7, dtype=torch.int32, device="cuda")
        cs = torch.empty(K, dtype=torch.int32, device="cuda")
        if use_planes:
            fqt1.im2col_planes(planes, N, C, H, W, k, k, s, p, rb, cbits, cs)
        else:
            fqt1.im2col(xt, N, C, H, W, k, k, s, p, rb, cbits, cs)
        outs.append((rb, cbits, cs))
    torch.cuda.synchronize()
    w = planes.cpu().numpy().view(np.uint32).reshape(N, C, pw)
    bits = ((w[:, :, :, None] >> np.arange(32, dtype=np.uint32)) & 1).reshape(N, C, -1)
    assert np.array_equal(bits[:, :, :H * W].astype(np.int8) * 2 - 1, om.sign(x).reshape(N, C, H * W))
    assert not bits[:, :, H * W:].any()
    for a, b in zip(*outs):
        assert torch.equal(a, b)
    # and both against the oracle's unfolded signs
    su, pad = unpack_bits(outs[1][0], K)
    assert np.array_equal(su, om.sign(om.unfold(x, k, k, s, p))) and not pad.any()


def test_im2col_path_query():
    """fqt1_im2col_path: whole-image tiles for the bench layer, region tiles for the ResNet-18
    ImageNet stem, the pointwise pass for 1 x 1 windows without padding (the downsamples), the
    gather for regions too large, -1 for invalid shapes."""
    from paper_2408_14267_gb300 import fqt1
    assert fqt1.im2col_path(128, 256, 8, 8, 3, 3, 1, 1) == 2
    assert fqt1.im2col_path(64, 3, 224, 224, 7, 7, 2, 3) == 1
    assert fqt1.im2col_path(64, 64, 56, 56, 1, 1, 2, 0) == 3
    assert fqt1.im2col_path(2, 256, 56, 56, 1, 1, 1, 0) == 3
    assert fqt1.im2col_path(1, 64, 512, 512, 3, 3, 1, 1) == 0
    assert fqt1.im2col_path(2, 4, 3, 3, 7, 7, 1, 0) == -1


def test_im2col_planes_rejects_gather_shapes():
    """Shapes served only by the gather Unfolder (which reads x itself) are unsupported from planes."""
    from paper_2408_14267_gb300 import fqt1
    N, C, H, W = 2, 256, 56, 56
    planes = torch.zeros(N * C * fqt1.plane_words(H, W), dtype=torch.int32, device="cuda")
    rb = torch.empty(N * H * W, fqt1.packed_words(C), dtype=torch.int32, device="cuda")
    with pytest.raises(fqt1.Fqt1Error, match="UNSUPPORTED"):
        fqt1.im2col_planes(planes, N, C, H, W, 1, 1, 1, 0, rb, None, None)


@pytest.mark.parametrize("name,make", FOLD_CASES, ids=[c[0] for c in FOLD_CASES])
def test_fold_channels_last_output(name, make):
    """The fused Folder writing dx channels-last (N, H, W, C) gives the NCHW result's values,
    pruned samples included."""
    from paper_2408_14267_gb300 import fqt1
    from paper_2408_14267_gb300.layer import LayerStep
    w = make()
    st = LayerStep(w, keep_acc=False)
    assert st.fold
    st.step()
    N, C, H, W, kh, kw = st.conv
    dx = torch.full((N, H, W, C), 3.0, device="cuda")
    fqt1.bwd_input_fold(st.psq, st.sw_col, st.cs_w, N, C, H, W, kh, kw, st.stride, st.pad, st.D, st.p_s, dx,
                        nhwc=True)
    torch.cuda.synchronize()
    assert torch.equal(dx.permute(0, 3, 1, 2), st.dx)


@pytest.mark.parametrize("name,make", [CASES[12], CASES[15], CASES[8], CASES[10], CASES[11]],
                         ids=[CASES[12][0], CASES[15][0], CASES[8][0], CASES[10][0], CASES[11][0]])
def test_col2im_channels_last_output(name, make):
    """The two-call Folder writing dx channels-last gives the NCHW result's values."""
    from paper_2408_14267_gb300 import fqt1
    from paper_2408_14267_gb300.layer import LayerStep
    w = make()
    st = LayerStep(w, keep_acc=True, fold=False)
    st.step()
    N, C, H, W, kh, kw = st.conv
    dx = torch.full((N, H, W, C), 3.0, device="cuda")
    fqt1.col2im(st.acc_dx, st.psq, st.cs_w, N, C, H, W, kh, kw, st.stride, st.pad, dx, nhwc=True)
    torch.cuda.synchronize()
    assert torch.equal(dx.permute(0, 3, 1, 2), st.dx)
