"""Pins of the oracle's stochastic rounding, AGP quantizer and SCQ factoring (Sec. 3.2, 5.2, 5.3, App. B/C)."""
import numpy as np
import pytest

from oracle import method as om

f32 = np.float32


def test_sr_unbiased_and_variance():
    """E[SR(t)] = t and Var[SR(t)] = p(1 - p) with p = t - floor(t) (App. B proposition)."""
    bits, trials = 4, 20000
    z, r = f32(-0.5), f32(2.0)
    xs = np.array([-0.5, -0.43, -0.11, 0.0, 0.2999, 0.77, 1.3, 1.5], dtype=f32)
    flat = np.arange(xs.size, dtype=np.uint64)
    q = np.stack([om.sr_codes(xs, z, r, bits, seed, 0, flat) for seed in range(trials)])
    B = f32(15)
    inv = B / r
    t = ((xs - z) * inv).astype(np.float64)
    frac = t - np.floor(t)
    assert np.all((q == np.floor(t)) | (q == np.floor(t) + 1))
    sd = np.sqrt(np.maximum(frac * (1 - frac), 1e-12) / trials)
    assert np.all(np.abs(q.mean(axis=0) - t) <= 5 * sd + 1e-9)
    var = q.var(axis=0)
    assert np.all(np.abs(var - frac * (1 - frac)) <= 0.02)
    assert q[:, 0].max() == 0 and q[:, -1].min() == 15   # x = Z -> 0, x = Z + R -> B


def test_sr_grid_points_exact_and_degenerate():
    z, r = f32(0.0), f32(3.0)
    xs = np.array([0, 1, 2, 3], dtype=f32)        # t = 0, 1, 2, 3 exactly for b = 2
    for seed in range(200):
        assert om.sr_codes(xs, z, r, 2, seed, 1, np.arange(4, dtype=np.uint64)).tolist() == [0, 1, 2, 3]
        assert om.sr_codes(xs, xs, f32(0), 2, seed, 1, np.arange(4, dtype=np.uint64)).tolist() == [0] * 4


def _dequant_psq(psq, M, D):
    """Dequantized AGP gradient (float64): (q S' + Z') on kept rows, 0 elsewhere."""
    out = np.zeros((M, D))
    rpg = psq["rows_per_group"]
    for s, g in enumerate(psq["kept"]):
        c = psq["codes"][s * rpg:(s + 1) * rpg].astype(np.float64)
        out[g * rpg:(g + 1) * rpg] = c * np.float64(psq["scale"][s]) + np.float64(psq["zero"][s])
    return out


def _dequant_pcq(pcq, M, D):
    out = np.zeros((M, D))
    for s, j in enumerate(pcq["kept"]):
        out[:, j] = pcq["codes"][s].astype(np.float64) * np.float64(pcq["scale"][s]) + np.float64(pcq["zero"][s])
    return out


@pytest.mark.parametrize("axis", [0, 1])
def test_agp_quantizer_unbiased(axis):
    """E[Q_PSQ^b(M G)] = G (Sec. 5.2): mean over seeds of the dequantized output."""
    rng = np.random.default_rng(9)
    M, D, rpg, bits, trials = 12, 6, 2, 2, 6000
    g = (rng.laplace(0, 1, (M, D)) * 10.0 ** rng.uniform(-1, 1, (M, 1))).astype(f32)
    acc = np.zeros((M, D))
    acc2 = np.zeros((M, D))
    for seed in range(trials):
        qd = om.agp_quantize(g, axis, rpg, bits, om.SYSTEMATIC, seed)
        d = _dequant_psq(qd, M, D) if axis == 0 else _dequant_pcq(qd, M, D)
        acc += d
        acc2 += d * d
    mean = acc / trials
    sd = np.sqrt(np.maximum(acc2 / trials - mean ** 2, 0) / trials)
    tol = 5 * sd + 1e-4 * np.abs(g)            # fp32 scale rounding ~1e-7 relative
    assert np.all(np.abs(mean - g) <= tol)


def test_eq24_variance_bound_topk():
    """Eq. 24: with the top-N/b groups kept, Var <= D / (4 B^2) sum_kept R_i^2, and the SR
    variance equals sum (R/B)^2 p(1-p) over kept elements."""
    rng = np.random.default_rng(2)
    M, D, bits, trials = 16, 32, 4, 3000
    g = (rng.standard_normal((M, D)) * 10.0 ** rng.uniform(-2, 1, (M, 1))).astype(f32)
    samples = np.stack([_dequant_psq(om.agp_quantize(g, 0, 1, bits, om.TOPK, s), M, D) for s in range(trials)])
    qd = om.agp_quantize(g, 0, 1, bits, om.TOPK, 0)
    kept = qd["kept"]
    B = (1 << bits) - 1
    total_var = samples.var(axis=0).sum()
    bound = D / (4 * B * B) * np.sum(qd["r"][kept].astype(np.float64) ** 2)
    assert total_var <= bound * 1.05
    inv = (f32(B) / qd["r"][kept]).astype(f32)
    t = ((g[kept] - qd["z"][kept][:, None]) * inv[:, None]).astype(np.float64)
    p = t - np.floor(t)
    expect = np.sum((qd["r"][kept].astype(np.float64)[:, None] / B) ** 2 * p * (1 - p))
    assert abs(total_var - expect) <= 0.08 * expect
    # the 1-bit PSQ bound of App. B is larger
    assert bound <= D / 4 * np.sum(qd["r"].astype(np.float64) ** 2)


def test_scq_factoring_and_bit_planes():
    """Sec. 5.3 / App. C: the scales factor out of the integer product, and the b-bit codes
    decompose losslessly into bit-planes multiplied by AND-popcount."""
    rng = np.random.default_rng(4)
    M, K, D, rpg = 12, 45, 10, 3
    x = rng.standard_normal((M, K)).astype(f32)
    w = rng.standard_normal((D, K)).astype(f32)
    g = (rng.standard_normal((M, D)) * 10.0 ** rng.uniform(-2, 1, (M, 1))).astype(f32)
    psq, pcq = om.scq_quantize(g, rpg, 4, om.SYSTEMATIC, 7, 2, om.SYSTEMATIC, 8)
    sw = np.where(w > 0, 1.0, -1.0)
    sx = np.where(x > 0, 1.0, -1.0)
    acc_dx, dx = om.bwd_input(psq, w, M)
    ref = _dequant_psq(psq, M, D) @ sw                 # dequantize first, float64 product
    a = np.abs(np.repeat(psq["scale"], rpg)[:, None].astype(np.float64) * acc_dx)
    mag = np.zeros_like(ref)
    for s, gid in enumerate(psq["kept"]):
        mag[gid * rpg:(gid + 1) * rpg] = a[s * rpg:(s + 1) * rpg] + abs(psq["zero"][s]) * np.abs(sw.sum(0))
    assert np.all(np.abs(dx - ref) <= 1e-6 * mag + 1e-30)
    pruned = np.setdiff1d(np.arange(M // rpg), psq["kept"])
    for gid in pruned:
        assert np.all(dx[gid * rpg:(gid + 1) * rpg] == 0)
    acc_dw, dw = om.bwd_weight(pcq, x, D)
    refw = (sx.T @ _dequant_pcq(pcq, M, D)).T
    magw = np.zeros_like(refw)
    for s, j in enumerate(pcq["kept"]):
        magw[j] = np.abs(np.float64(pcq["scale"][s]) * acc_dw[s]) + abs(pcq["zero"][s]) * np.abs(sx.sum(0))
    assert np.all(np.abs(dw - refw) <= 1e-6 * magw + 1e-30)
    # bit-planes: x = sum_i 2^(i-1) x^i, each plane through AND-popcount with +-1 operands
    planes = om.bit_planes(psq["codes"], 4)
    assert np.array_equal((planes.astype(np.int64) * (1 << np.arange(4))[:, None, None]).sum(0), psq["codes"])
    wbits = [sum(1 << j for j in range(D) if w[j, k] > 0) for k in range(K)]
    for r in range(planes.shape[1]):
        for k in range(K):
            tot = 0
            for p in range(4):
                a_bits = sum(1 << j for j in range(D) if planes[p, r, j])
                # {0,1} x {-1,+1}: sum a_j s_j = 2 popc(a & w) - popc(a)
                tot += (1 << p) * (2 * bin(a_bits & wbits[k]).count("1") - bin(a_bits).count("1"))
            assert tot == acc_dx[r, k]


def test_conv_grad_input_matches_transposed_conv():
    """Folder after the PSQ product == transposed convolution of the dequantized gradient."""
    import torch
    rng = np.random.default_rng(6)
    N, C, H, W, D, k, s, p = 4, 3, 7, 6, 5, 3, 2, 1
    x = rng.standard_normal((N, C, H, W)).astype(f32)
    w = rng.standard_normal((D, C, k, k)).astype(f32)
    Ho, Wo = om.conv_out_hw(H, W, k, k, s, p)
    gy = (rng.standard_normal((N * Ho * Wo, D)) * 10.0 ** rng.uniform(-2, 1, (N * Ho * Wo, 1))).astype(f32)
    res = om.layer_step_conv(x, w, np.ones(D, f32), gy, s, p, 2, om.SYSTEMATIC, 1, 2, om.SYSTEMATIC, 2)
    gd = _dequant_psq(res["psq"], N * Ho * Wo, D).reshape(N, Ho, Wo, D).transpose(0, 3, 1, 2)
    sw = np.where(w > 0, 1.0, -1.0)
    ref = torch.nn.functional.conv_transpose2d(torch.from_numpy(gd), torch.from_numpy(sw), stride=s, padding=p,
                                               output_padding=((H + 2 * p - k) % s, (W + 2 * p - k) % s)).numpy()
    scale = np.zeros(N)
    scale[res["psq"]["kept"]] = np.abs(res["psq"]["scale"])
    tol = 1e-6 * (scale[:, None, None, None] * np.abs(res["acc_fold"]) + np.abs(ref)) + 1e-30
    assert np.all(np.abs(res["dx"] - ref) <= tol)


def test_agp_variance_below_one_bit_psq():
    """Sec. 5.2 / App. B: on groups with heterogeneous ranges, AGP with b = 4 (a quarter of the
    groups kept at 4 bits, systematic masks) has a much smaller variance E||Q(G) - G||^2 than
    1-bit PSQ (every group at 1 bit), whose exact variance is sum R_i^2 p(1 - p) over the
    elements (SR variance with B = 1)."""
    rng = np.random.default_rng(12)
    M, D, rpg, trials = 32, 8, 1, 1500
    g = (rng.standard_normal((M, D)) * np.exp(2 * rng.standard_normal((M, 1)))).astype(f32)
    agp = np.stack([_dequant_psq(om.agp_quantize(g, 0, rpg, 4, om.SYSTEMATIC, s), M, D) for s in range(trials)])
    var_agp = ((agp - g.astype(np.float64)) ** 2).sum(axis=(1, 2)).mean()
    qd = om.agp_quantize(g, 0, rpg, 1, om.SYSTEMATIC, 0)
    t = ((g - qd["z"][:, None]) * (f32(1) / qd["r"])[:, None]).astype(np.float64)
    p = t - np.floor(t)
    var_psq = np.sum(qd["r"].astype(np.float64)[:, None] ** 2 * p * (1 - p))
    assert var_agp < 0.25 * var_psq
    # and the 1-bit PSQ variance formula itself against sampling
    psq = np.stack([_dequant_psq(om.agp_quantize(g, 0, rpg, 1, om.SYSTEMATIC, s), M, D) for s in range(400)])
    emp = ((psq - g.astype(np.float64)) ** 2).sum(axis=(1, 2)).mean()
    assert abs(emp - var_psq) <= 0.1 * var_psq
