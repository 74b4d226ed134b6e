"""Pins of the oracle's whole layer (Sec. 3.1 end to end) and of its offline
integer constants (Eq. 7, Eq. 11, I-BERT's exponential constants)."""
import math

import numpy as np
import pytest

import synth
from fp64_ref import attention_f64

# Stated agreement of the integer layer with the float64 rel-pos attention
# (Eqs. 8-9, real scales, fused score clipped to its grid, exact softmax,
# output quantised onto S_O), in output LSB: (max, mean) by the fineness of
# the score grid, q_ln2 = floor(ln2 / S_s).  The integer path rounds the
# fused score onto its int8 grid, approximates exp, and keeps probabilities
# on the grid 2^-8; on a coarse score grid the integer exponential dominates
# the error (see test_oracle_softmax.lsb_bound).
def layer_bound(q_ln2: int) -> tuple[float, float]:
    if q_ln2 >= 16:
        return 6, 0.85
    if q_ln2 >= 10:
        return 12, 1.0
    return 32, 3.0


CASES = [
    # (workload, B, T) - the workload's distribution at a size the oracle
    # finishes in seconds
    (0, 1, 64),
    (1, 1, 125),
    (2, 2, 250),
    (3, 1, 375),
    (4, 1, 300),
]


@pytest.mark.parametrize("w,B,T", CASES)
@pytest.mark.parametrize("seed", [17, 18, 19])
def test_layer_vs_float64_attention(oracle_lib, w, B, T, seed):
    W = synth.WORKLOADS[w]
    lay = synth.draw(B, W.H, T, W.dh, seed=1000 * w + seed, p_mode=W.p_mode,
                     dist=W.dist, masked=W.masked)
    c = oracle_lib.layer_constants(lay.scales, W.dh)
    got = oracle_lib.relpos_mhsa(lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb, c, lay.lengths)
    _, want, _, _ = attention_f64(lay, lay.lengths)
    err = np.abs(got.astype(np.int64) - want)
    mx, mean = layer_bound(c.softmax[0])
    assert err.max() <= mx, (c.softmax, err.max())
    assert err.mean() <= mean, (c.softmax, err.mean())
    assert (got != -128).all()


def test_layer_detects_dropped_terms(oracle_lib):
    # The float64 comparison is sharp enough to see a missing bias or a
    # mirrored relative shift: perturbing the inputs that way moves the
    # result far outside the stated bound.
    lay = synth.draw(1, 8, 96, 128, seed=4242, p_mode="sinusoid")
    c = oracle_lib.layer_constants(lay.scales, 128)
    _, want, _, _ = attention_f64(lay)
    for bad in ("u", "vb", "pflip"):
        q, k, v, p, u, vb = lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb
        if bad == "u":
            u = np.zeros_like(u)
        elif bad == "vb":
            vb = np.zeros_like(vb)
        else:
            p = np.ascontiguousarray(p[:, ::-1, :])
        got = oracle_lib.relpos_mhsa(q, k, v, p, u, vb, c)
        err = np.abs(got.astype(np.int64) - want)
        mx, mean = layer_bound(c.softmax[0])
        assert err.max() > mx and err.mean() > mean, (bad, err.max(), err.mean())


def test_masked_layer_equals_truncated_problem(oracle_lib):
    # Keys j >= len are excluded and rows i >= len output 0, while Phi still
    # indexes P with T.  So the first len rows equal the unmasked problem of
    # length len on Q,K,V[:len] and P rows T-len .. T+len-2.
    B, H, T, dh = 3, 2, 37, 64
    lens = np.array([37, 20, 1], np.int32)
    lay = synth.draw(B, H, T, dh, seed=77, lengths=lens)
    c = oracle_lib.layer_constants(lay.scales, dh)
    out = oracle_lib.relpos_mhsa(lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb, c, lens)
    for b, n in enumerate(lens):
        n = int(n)
        sl = lambda x: np.ascontiguousarray(x[b:b + 1, :, :n])
        p_n = np.ascontiguousarray(lay.p[:, T - n:T + n - 1])
        ref = oracle_lib.relpos_mhsa(sl(lay.q), sl(lay.k), sl(lay.v), p_n, lay.u, lay.vb, c)
        np.testing.assert_array_equal(out[b:b + 1, :, :n], ref)
        assert (out[b, :, n:] == 0).all()


def test_lengths_clamped(oracle_lib):
    B, H, T, dh = 3, 1, 9, 16
    lay = synth.draw(B, H, T, dh, seed=78)
    c = oracle_lib.layer_constants(lay.scales, dh)
    a = oracle_lib.relpos_mhsa(lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb, c,
                               np.array([-5, 0, 99], np.int32))
    b = oracle_lib.relpos_mhsa(lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb, c,
                               np.array([0, 0, T], np.int32))
    np.testing.assert_array_equal(a, b)
    assert (a[:2] == 0).all()


def test_single_frame_closed_form(oracle_lib):
    # T = 1: one key, probability 255, O = round(m_o 255 V 2^-(31+s_o)).
    lay = synth.draw(2, 3, 1, 128, seed=79)
    c = oracle_lib.layer_constants(lay.scales, 128)
    out = oracle_lib.relpos_mhsa(lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb, c)
    m_o, s_o = c.multipliers[2], c.shifts[1]
    x = m_o * 255 * lay.v.astype(np.int64)
    want = np.clip(np.floor_divide(x + 2 ** (30 + s_o), 2 ** (31 + s_o)), -127, 127)
    np.testing.assert_array_equal(out, want)


def test_workload_shifts_in_range():
    import oracle
    for w in range(5):
        c = oracle.layer_constants(synth.layer(w, 0).scales, 128) if w != 3 else \
            oracle.layer_constants(synth.draw(1, 8, 375, 128, 3000, p_mode="sinusoid").scales, 128)
        assert all(8 <= s <= 20 for s in c.shifts), c
        assert all(2 ** 30 <= m < 2 ** 31 for m in (max(c.multipliers[:2]), c.multipliers[2])), c


@pytest.mark.parametrize("ratio", [0.49, 1e-3, 3.1e-7, 2 ** -9, 2 ** -20 * 1.5, 1e-12])
def test_dyadic_encoding(ratio):
    import oracle
    m, s = oracle.dyadic(ratio)
    assert 0 <= s <= 31
    approx = m / 2.0 ** (31 + s)
    assert abs(approx - ratio) <= 2.0 ** -(32 + s) * (1 + 1e-12)
    if s < 31:
        assert 2 ** 30 <= m < 2 ** 31


def test_dyadic_exact_powers():
    import oracle
    assert oracle.dyadic(0.25) == (2 ** 30, 1)
    assert oracle.dyadic(2.0 ** -9) == (2 ** 30, 8)
    with pytest.raises(ValueError):
        oracle.dyadic(1.0)
    with pytest.raises(ValueError):
        oracle.dyadic(0.0)


def test_dyadic_pair_shares_shift():
    import oracle
    m_c, m_p, s = oracle.dyadic_pair(3e-3, 1e-3)
    assert 2 ** 30 <= m_c < 2 ** 31 and m_p < m_c
    assert abs(m_p / 2.0 ** (31 + s) - 1e-3) <= 2.0 ** -(32 + s)
