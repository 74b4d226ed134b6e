"""Pins of the oracle's score branches and their fusion (Sec. 3.1,
Eqs. 8, 10 and 11)."""
from fractions import Fraction
import math

import numpy as np
import pytest

import synth
from fp64_ref import relshift_gather


def test_content_rank1_split(oracle_lib):
    # (Q + 1u^T) K^T = Q K^T + 1 (K u)^T exactly in integers (Eq. 8).
    lay = synth.draw(2, 3, 21, 32, seed=5)
    q = lay.q.astype(np.int64)
    k = lay.k.astype(np.int64)
    u = lay.u.astype(np.int64)
    want = np.einsum("bhid,bhjd->bhij", q, k) + np.einsum("bhjd,hd->bhj", k, u)[:, :, None, :]
    np.testing.assert_array_equal(oracle_lib.content_scores(lay.q, lay.k, lay.u), want)


def test_position_rank1_split(oracle_lib):
    lay = synth.draw(2, 3, 13, 32, seed=6)
    q = lay.q.astype(np.int64)
    p = lay.p.astype(np.int64)
    vb = lay.vb.astype(np.int64)
    bd = np.einsum("bhid,hrd->bhir", q, p) + np.einsum("hrd,hd->hr", p, vb)[None, :, None, :]
    np.testing.assert_array_equal(oracle_lib.position_scores(lay.q, lay.p, lay.vb),
                                  relshift_gather(bd))


def _fused_real(qc, qp, r_c, r_p):
    return r_c * qc.astype(np.float64) + r_p * qp.astype(np.float64)


@pytest.mark.parametrize("seed,T", [(1, 17), (2, 40), (3, 64)])
def test_fused_matches_eq10_real_ratios(oracle_lib, seed, T):
    # Eq. 11 is Eq. 10 with the real ratios replaced by dyadic m 2^-(31+s):
    # |r - m 2^-(31+s)| <= 2^-(32+s) and |qc|, |qp| < 2^23, so both round to
    # the same integer unless the real value lies within 2^-17 of a
    # half-integer; there they may differ by one.
    lay = synth.draw(1, 8, T, 128, seed=seed)
    root = math.sqrt(128)
    sc = lay.scales
    r_c = sc["S_Q"] * sc["S_K"] / (sc["S_s"] * root)
    r_p = sc["S_Q"] * sc["S_P"] / (sc["S_s"] * root)
    m_c, m_p, s = oracle_lib.dyadic_pair(r_c, r_p)
    qs = oracle_lib.fused_scores(lay.q, lay.k, lay.p, lay.u, lay.vb, m_c, m_p, s).astype(np.int64)
    qc = oracle_lib.content_scores(lay.q, lay.k, lay.u)
    qp = oracle_lib.position_scores(lay.q, lay.p, lay.vb)
    x = _fused_real(qc, qp, r_c, r_p)
    want = np.clip(np.floor(x + 0.5), -127, 127).astype(np.int64)
    near_tie = np.abs(x - np.floor(x) - 0.5) < 2.0 ** -17
    assert np.all(np.abs(qs - want) <= 1)
    np.testing.assert_array_equal(qs[~near_tie], want[~near_tie])
    assert (qs >= -127).all() and (qs <= 127).all()


def _one_score(oracle_lib, qval, m_c, s, m_p=0):
    q = np.array([[[[qval]]]], np.int8)
    k = np.ones((1, 1, 1, 1), np.int8)
    p = np.zeros((1, 1, 1), np.int8)
    z = np.zeros((1, 1), np.int8)
    return int(oracle_lib.fused_scores(q, k, p, z, z, m_c, m_p, s)[0, 0, 0, 0])


@pytest.mark.parametrize("qc,want", [(1, 1), (-1, 0), (3, 2), (-3, -1), (5, 3), (-5, -2), (2, 1), (-2, -1)])
def test_fused_rounding_ties_go_up(oracle_lib, qc, want):
    # m_c = 2^30 with s = 0 is the ratio 1/2: odd qc lands on an exact tie,
    # which rounds toward +infinity.
    assert _one_score(oracle_lib, qc, 2 ** 30, 0) == want


@pytest.mark.parametrize("s", [0, 5, 17, 31])
def test_fused_shift_exponent(oracle_lib, s):
    # m = 2^30 encodes the ratio 2^-(s+1) exactly: the score is the closed
    # form round(qc / 2^(s+1)), clamped to the int8 grid.
    for qc in (1, 7, 100, 127):
        val = qc * 2 ** 30
        ref = Fraction(val, 2 ** (31 + s))
        want = max(-127, min(127, math.floor(ref + Fraction(1, 2))))
        assert _one_score(oracle_lib, qc, 2 ** 30, s) == want


def test_fused_saturation_and_headroom(oracle_lib):
    # Adversarial all-+-127 inputs with the largest multipliers: the int64
    # accumulation must not wrap (results saturate with the right sign).
    T, dh = 8, 128
    ones = np.full((1, 1, T, dh), 127, np.int8)
    negs = np.full((1, 1, T, dh), -127, np.int8)
    p = np.full((1, 2 * T - 1, dh), 127, np.int8)
    u = np.full((1, dh), 127, np.int8)
    big = 2 ** 31 - 1
    for s in (0, 31):
        pos = oracle_lib.fused_scores(ones, ones, p, u, u, big, big, s)
        neg = oracle_lib.fused_scores(ones, negs, -p, u, u, big, big, s)
        if s == 0:
            assert (pos == 127).all() and (neg == -127).all()
        else:
            # 2^31 * 2 * 254*127*128 / 2^62 ~ 3.9e-3 -> rounds to 0
            assert (pos == 0).all() and (neg == 0).all()


def test_content_only_when_m_p_zero(oracle_lib):
    # m_p = 0 removes the position branch: the scores no longer depend on P.
    lay = synth.draw(1, 2, 12, 32, seed=9)
    other = synth.draw(1, 2, 12, 32, seed=10)
    a = oracle_lib.fused_scores(lay.q, lay.k, lay.p, lay.u, lay.vb, 2 ** 30, 0, 12)
    b = oracle_lib.fused_scores(lay.q, lay.k, other.p, lay.u, other.vb, 2 ** 30, 0, 12)
    np.testing.assert_array_equal(a, b)
    c = oracle_lib.fused_scores(lay.q, other.k, lay.p, other.u, lay.vb, 0, 2 ** 30, 12)
    d = oracle_lib.fused_scores(lay.q, lay.k, lay.p, lay.u, lay.vb, 0, 2 ** 30, 12)
    np.testing.assert_array_equal(c, d)
