"""Small worked cases of AGP and stochastic rounding, derived by hand from Sec. 5.2 and Sec. 3.2.

Each expected value below is worked out in the docstring from the definitions (water-filled
keep probabilities, systematic masks over one offset U, the stochastic-rounding threshold), so a
reader can check it with pen and paper. The only generator calls are to the oracle's Philox
word, itself pinned against Triton's independent implementation.
"""
import numpy as np

from oracle import method as om
from oracle.philox import uniform_u32

TWO32 = 1 << 32


def test_water_filling_with_one_binding_cap():
    """R = [8, 1, 1, 1, 1], b = 2: the budget is n / b = 2.5.

    Proportional probabilities 2.5 R / 12 give 1.67 for group 0, above 1, so group 0 is
    capped at p = 1 and the remaining 1.5 is shared by the four equal groups: p = 0.375 each.
    In fixed point: max R = 8 = 0.5 x 2^4, so E = 4 and R~ = R 2^36 = [2^39, 2^36 x 4];
    t = 0 fails (5 x 2^39 > 2 x 12 x 2^36), t = 1 holds (3 x 2^36 <= 2 x 4 x 2^36), so t* = 1
    and P = 3 x 2^36 x 2^32 / (2 x 4 x 2^36) = 3 x 2^29 for the others.
    """
    r = np.array([8, 1, 1, 1, 1], dtype=np.float32)
    assert om.fixed_point_ranges(r) == [1 << 39] + [1 << 36] * 4
    P, order = om.agp_probabilities(r, 2)
    assert P == [TWO32] + [3 << 29] * 4
    assert order == [0, 1, 2, 3, 4]
    assert sum(P) == 5 * TWO32 // 2


def test_no_cap_probabilities_and_systematic_masks_by_hand():
    """R = [4, 2, 1, 1], b = 2: p_i = n R_i / (b R_total) = R_i / 4 = [1, 1/2, 1/4, 1/4].

    P = [2^32, 2^31, 2^30, 2^30]. The systematic mask keeps group i when [C_i, C_i + P_i)
    holds a multiple of 2^32, with C_0 = U and C_{i+1} = C_i + P_i:
      group 0 always (P_0 = 2^32);
      group 1 iff U + 2^31 >= 2^32, i.e. U >= 2^31;
      group 2 iff U in [2^30, 2^31);
      group 3 iff U < 2^30.
    So exactly two groups are kept, and the second is fixed by U alone.
    """
    r = np.array([4, 2, 1, 1], dtype=np.float32)
    P, _ = om.agp_probabilities(r, 2)
    assert P == [TWO32, 1 << 31, 1 << 30, 1 << 30]
    seen = set()
    for seed in range(400):
        u = int(uniform_u32(seed, 2, np.uint64(0)))
        second = 1 if u >= 1 << 31 else (2 if u >= 1 << 30 else 3)
        kept, p_hat, _ = om.select_groups(r, 2, om.SYSTEMATIC, seed, 2)
        assert kept.tolist() == [0, second], seed
        assert p_hat.tolist() == [1.0, 0.5, 0.25, 0.25]
        seen.add(second)
    assert seen == {1, 2, 3}


def test_stochastic_rounding_thresholds_by_hand():
    """b = 2 (B = 3), Z = 0, R = 1: t = 3 x, floor and fraction are exact in fp32.

    x = 0 and x = 1 give t = 0 and 3: codes 0 and 3 whatever the draw.
    x = 0.5 gives t = 1.5: code 2 iff u = (w >> 8) 2^-24 < 0.5, i.e. w < 2^31, else 1.
    x = 0.25 gives t = 0.75: code 1 iff (w >> 8) < 0.75 x 2^24, i.e. w < 3 x 2^30, else 0.
    A zero range gives code 0.
    """
    x = np.array([0.0, 1.0, 0.5, 0.25], dtype=np.float32)
    seeds = range(64)
    for seed in seeds:
        idx = np.arange(4, dtype=np.uint64) + np.uint64(4 * seed)
        q = om.sr_codes(x, np.float32(0), np.float32(1), 2, seed, 0, idx)
        w = uniform_u32(seed, 0, idx).astype(np.int64)
        assert q[0] == 0 and q[1] == 3
        assert q[2] == (2 if w[2] < 1 << 31 else 1)
        assert q[3] == (1 if w[3] < 3 << 30 else 0)
    q = om.sr_codes(np.array([0.3, -2.0], np.float32), np.float32(0.3), np.float32(0), 4, 1, 0,
                    np.arange(2, dtype=np.uint64))
    assert q.tolist() == [0, 0]


def test_rescale_of_a_kept_group_by_hand():
    """S' = R / (B p^) and Z' = Z / p^ (Sec. 5.2, M = diag(m / p)): R = 1, Z = -0.5,
    p^ = 0.375, b = 2 give S' = 1 / 1.125 = 8/9 and Z' = -4/3, each rounded once to fp32."""
    s, z = om.group_scale(np.array([1.0], np.float32), np.array([-0.5], np.float32), np.array([0.375]), 2)
    assert s[0] == np.float32(8.0 / 9.0)
    assert z[0] == np.float32(-4.0 / 3.0)


def test_bernoulli_masks_by_hand():
    """The paper-literal mode draws m_i ~ Bern(p_i) independently: group i is kept iff its own
    32-bit word is below P_i. R = [2, 0, 1] with b = 1 keeps all (plain PSQ); with P built for
    b = 2 (n / b = 1.5): p = 1.5 R / 3 = [1, 0, 0.5] with no cap binding, so group 0 is always
    kept, group 1 never, and group 2 iff its word is below 2^31."""
    r = np.array([2, 0, 1], dtype=np.float32)
    kept, p_hat, _ = om.select_groups(r, 1, om.BERNOULLI, 0, 2)
    assert kept.tolist() == [0, 1, 2] and p_hat.tolist() == [1.0, 1.0, 1.0]
    P, _ = om.agp_probabilities(r, 2, om.BERNOULLI)
    assert P == [TWO32, 0, 1 << 31]
    seen = set()
    for seed in range(200):
        w2 = int(uniform_u32(seed, 3, np.uint64(2)))
        kept, _, _ = om.select_groups(r, 2, om.BERNOULLI, seed, 3)
        assert kept.tolist() == ([0, 2] if w2 < 1 << 31 else [0]), seed
        seen.add(len(kept))
    assert seen == {1, 2}
