"""Pins of the oracle's whole layer (Sec. 3.1 end to end) and of its offline
integer constants (Eq. 7, Eq. 11, I-BERT's exponential constants)."""
import math

import numpy as np
import pytest

import synth
import ibert_bounds as ib
from fp64_ref import attention_f64

def derived_bound(lay, c, lengths=None):
    """Per-output bound of |O_int - O_ref| in output steps, derived from the
    roundings of the method (tests/ibert_bounds.py, step 6): the fused
    score's rounding onto its int8 grid, the integer exponential's floors and
    its halving every floor(ln2 / S_s) steps, the floor onto the probability
    grid 2^-8, and the two roundings onto the output grid.  O_ref is the
    float64 rel-pos attention of fp64_ref (real scales, fused score clipped
    to its grid, exact softmax, output quantised onto S_O)."""
    _, want, probs, scores = attention_f64(lay, lengths)
    r = lay.scales["S_V"] / lay.scales["S_O"]
    bound = ib.layer_output_bound(probs, scores, lay.v, lay.scales["S_s"], c.shifts[0], r,
                                  c.multipliers[2], c.shifts[1])
    return bound, want


def _check_layer(oracle_lib, lay):
    c = oracle_lib.layer_constants(lay.scales, lay.q.shape[-1])
    got = oracle_lib.relpos_mhsa(lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb, c, lay.lengths)
    bound, want = derived_bound(lay, c, lay.lengths)
    err = np.abs(got.astype(np.int64) - want)
    worst = np.unravel_index(np.argmax(err - bound), err.shape)
    assert (err <= bound).all(), (c.softmax, int(err[worst]), float(bound[worst]), worst)
    assert (got != -128).all()
    return err, bound


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
    _check_layer(oracle_lib, lay)


def _first_utterance(lay):
    return synth.Layer(q=lay.q[:1], k=lay.k[:1], v=lay.v[:1], p=lay.p, u=lay.u, vb=lay.vb,
                       lengths=None if lay.lengths is None else lay.lengths[:1],
                       scales=lay.scales)


# The benchmark's encoder layers on the coarsest score grids: layer 13
# (q_ln2 = 7), layers 1 and 2 (q_ln2 = 8), layer 7 (q_ln2 = 9); one
# utterance each, with the layer's own scales.
@pytest.mark.parametrize("index,q_ln2", [(13, 7), (1, 8), (2, 8), (7, 9)])
def test_encoder_layer_coarse_grid(oracle_lib, index, q_ln2):
    lay = _first_utterance(synth.layer(3, index))
    c = oracle_lib.layer_constants(lay.scales, 128)
    assert c.softmax[0] == q_ln2
    err, bound = _check_layer(oracle_lib, lay)
    # informative, not a pin: the error stays well inside the bound on average
    assert err.mean() <= bound.mean()


def test_layer_detects_dropped_terms(oracle_lib):
    # The derived bound is sharp enough to see a missing bias or a mirrored
    # relative shift: perturbing the inputs that way moves some outputs
    # outside it.
    lay = synth.draw(1, 8, 96, 128, seed=4242, p_mode="sinusoid")
    c = oracle_lib.layer_constants(lay.scales, 128)
    bound, want = derived_bound(lay, c)
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
        assert (err > bound).sum() > 100, (bad, int((err > bound).sum()))


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
