"""Pins of the oracle's AGP keep probabilities and masks (Sec. 5.2, App. B)."""
import numpy as np
import pytest

from oracle import method as om

TWO32 = 2 ** 32


def _phat(P):
    return np.array(P, dtype=np.float64) / TWO32


def test_closed_form_when_no_cap_binds():
    """p_i = N R_i / (b R_total) (Sec. 5.2) when every such value is <= 1."""
    rng = np.random.default_rng(1)
    for n, b in [(64, 2), (64, 4), (37, 8), (100, 4)]:
        r = rng.uniform(1.0, 1.5, n).astype(np.float32)
        P, _ = om.agp_probabilities(r, b)
        ref = n * r.astype(np.float64) / (b * r.astype(np.float64).sum())
        assert ref.max() <= 1.0
        assert np.max(np.abs(_phat(P) - ref)) < 2.0 ** -30
        # budget: sum p = n / b up to the integer truncations (condition 1)
        assert n / b - n * 2.0 ** -31 <= _phat(P).sum() <= n / b


def test_equal_ranges_and_b1():
    r = np.full(48, 0.37, dtype=np.float32)
    for b in [2, 4, 8]:
        P, _ = om.agp_probabilities(r, b)
        assert all(p == TWO32 // b for p in P)
    P, _ = om.agp_probabilities(np.random.default_rng(0).random(20).astype(np.float32), 1)
    assert all(p == TWO32 for p in P)
    kept, p_hat, _ = om.select_groups(np.random.default_rng(0).random(20).astype(np.float32), 1, om.SYSTEMATIC, 3, 2)
    assert kept.tolist() == list(range(20)) and np.all(p_hat == 1.0)


def _waterfill_bisection(r, b):
    """Independent solver: find c with sum min(1, c r_i) = n/b by bisection (float64)."""
    r = r.astype(np.float64)
    n = r.size
    lo, hi = 0.0, 1.0
    while np.minimum(1.0, hi * r).sum() < n / b:
        hi *= 2
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        if np.minimum(1.0, mid * r).sum() < n / b:
            lo = mid
        else:
            hi = mid
    return np.minimum(1.0, hi * r)


@pytest.mark.parametrize("n,b", [(64, 2), (128, 4), (256, 4), (512, 8), (33, 4), (7, 2)])
def test_water_filling_matches_bisection(n, b):
    """Heavy-tailed ranges (4 decades) force caps: compare with an independent solver."""
    rng = np.random.default_rng(n + b)
    r = (10.0 ** rng.uniform(-2, 2, n)).astype(np.float32)
    P, _ = om.agp_probabilities(r, b)
    ph = _phat(P)
    ref = _waterfill_bisection(r, b)
    assert np.max(np.abs(ph - ref)) < 1e-8
    assert np.all(ph <= 1.0)
    # condition 3: larger range, never smaller probability
    o = np.argsort(r, kind="stable")
    assert np.all(np.diff(ph[o]) >= -1e-12)
    assert n / b - n * 2.0 ** -31 <= ph.sum() <= n / b


def test_zero_ranges_never_kept():
    r = np.array([0, 3, 0, 1, 0, 0, 2, 0], dtype=np.float32)
    P, _ = om.agp_probabilities(r, 2)
    assert [P[i] for i in (0, 2, 4, 5, 7)] == [0] * 5
    assert [P[i] for i in (1, 3, 6)] == [TWO32] * 3
    for seed in range(50):
        kept, _, _ = om.select_groups(r, 2, om.SYSTEMATIC, seed, 2)
        assert set(kept.tolist()) == {1, 3, 6}


def test_topk_keeps_largest():
    r = np.array([5, 1, 9, 9, 2, 7, 3, 0.5], dtype=np.float32)
    kept, p_hat, _ = om.select_groups(r, 4, om.TOPK, 0, 2)
    assert kept.tolist() == [2, 3]
    kept, _, _ = om.select_groups(r, 2, om.TOPK, 0, 2)
    assert kept.tolist() == [0, 2, 3, 5]


@pytest.mark.parametrize("mode", [om.SYSTEMATIC, om.BERNOULLI])
def test_mask_inclusion_frequencies(mode):
    """m_i ~ Bern(p^_i): inclusion frequency over many seeds matches p^ (binomial z-test)."""
    rng = np.random.default_rng(5)
    n, b, trials = 24, 4, 6000
    r = (10.0 ** rng.uniform(-1.5, 1.5, n)).astype(np.float32)
    P, _ = om.agp_probabilities(r, b)
    ph = _phat(P)
    cap = om.kept_capacity(n, b, mode)
    counts = np.zeros(n)
    for seed in range(trials):
        kept = om.agp_masks(P, seed, 2, mode)
        counts += kept
        if mode == om.SYSTEMATIC:
            # the bit budget: floor or ceil of sum p^ groups, never above the capacity
            assert int(np.floor(ph.sum())) <= kept.sum() <= int(np.ceil(ph.sum()))
        assert kept.sum() <= cap
    freq = counts / trials
    sd = np.sqrt(np.maximum(ph * (1 - ph), 1e-12) / trials)
    assert np.all(np.abs(freq - ph) <= 5 * sd + 1e-12)
    # unbiasedness of the mask: E[m_i / p^_i] = 1 for groups with p^ > 0
    nz = ph > 0
    assert np.all(np.abs(freq[nz] / ph[nz] - 1) <= 5 * sd[nz] / ph[nz] + 1e-12)
