"""Pins of the oracle's integer softmax (I-BERT's integer exponential and
normalisation, which I-Parakeet uses for the attention, Sec. 2.2 and the
text after Eq. 11).  Constants from tests/golden/ibert_exp.txt."""
import math
import os

import numpy as np
import pytest

import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "ibert_exp.txt")


def _golden():
    vals = {}
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                k, v = line.split()
                vals[k] = float(v)
    return vals


def _grid_params(oracle_lib):
    out = []
    for w in range(5):
        lay = synth.layer(w, 0) if w != 3 else synth.draw(1, 8, 375, 128, 3000, p_mode="sinusoid")
        S = lay.scales["S_s"]
        out.append((S, oracle_lib.isoftmax_params(S)))
    for q in (5, 8, 16, 32, 100, 400):
        S = math.log(2) / (q + 0.25)
        out.append((S, oracle_lib.isoftmax_params(S)))
    return out


def test_constants_match_golden(oracle_lib):
    g = _golden()
    assert (oracle_lib.IBERT_A, oracle_lib.IBERT_B, oracle_lib.IBERT_C) == (g["a"], g["b"], g["c"])
    # the fitted polynomial is close to exp at both ends of [-ln2, 0]
    poly = lambda p: g["a"] * (p + g["b"]) ** 2 + g["c"]
    assert abs(poly(0.0) - 1.0) < 5e-4
    assert abs(poly(-math.log(2)) - 0.5) < 5e-4
    xs = np.linspace(-math.log(2), 0, 2001)
    assert np.max(np.abs(poly(xs) - np.exp(xs))) < 2.5e-3


def test_params_closed_form(oracle_lib):
    # On the grid S = ln2/10.5: q_ln2 = 10; q_b = floor(1.353/S); q_c = floor(0.344/(0.3585 S^2)).
    S = math.log(2) / 10.5
    q_ln2, q_b, q_c = oracle_lib.isoftmax_params(S)
    assert q_ln2 == 10
    assert q_b == math.floor(1.353 * 10.5 / math.log(2))
    assert q_c == math.floor(0.344 * 10.5 ** 2 / (0.3585 * math.log(2) ** 2))


def test_iexp_monotone_exhaustive(oracle_lib):
    for S, prm in _grid_params(oracle_lib):
        e = [oracle_lib.iexp(d, prm) for d in range(-254, 1)]
        assert all(a <= b for a, b in zip(e, e[1:])), (S, prm)
        assert e[-1] == prm[1] ** 2 + prm[2]          # d = 0: L(0) = q_b^2 + q_c


def test_iexp_halving_identity(oracle_lib):
    # Stepping d down by q_ln2 adds one to the shift: e(d - q_ln2) = floor(e(d) / 2).
    for S, prm in _grid_params(oracle_lib):
        q_ln2 = prm[0]
        for d in range(-254 + q_ln2, 1):
            assert oracle_lib.iexp(d - q_ln2, prm) == oracle_lib.iexp(d, prm) // 2


def test_iexp_polynomial_accuracy(oracle_lib):
    # For -q_ln2 < d <= 0 no shift happens and e(d) a S^2 approximates
    # exp(d S) up to the fit error (2.5e-3) plus the floors of q_b and q_c
    # (|dL| <= 2 (b/S) + 2 in units of a S^2).
    for S, prm in _grid_params(oracle_lib):
        q_ln2 = prm[0]
        bound = 2.5e-3 + (2 * 1.353 / S + 2) * 0.3585 * S * S
        for d in range(-q_ln2 + 1, 1):
            approx = oracle_lib.iexp(d, prm) * 0.3585 * S * S
            assert abs(approx - math.exp(d * S)) <= bound, (S, d)


def _softmax_f64(scores, S, valid):
    x = scores.astype(np.float64) * S
    n = scores.shape[-1]
    mask = np.arange(n)[None, :] < valid[:, None]
    x = np.where(mask, x, -np.inf)
    mx = np.max(x, axis=-1, keepdims=True)
    e = np.where(mask, np.exp(x - np.where(np.isfinite(mx), mx, 0)), 0.0)
    den = e.sum(-1, keepdims=True)
    return 256.0 * np.divide(e, den, out=np.zeros_like(e), where=den > 0)


# Stated bound of |a_j - 256 softmax_f64(S_s q_s)_j| in output LSB (grid
# 2^-8), by the fineness of the score grid.  The integer exponential halves
# every q_ln2 = floor(ln2 / S) steps instead of every ln2 / S, and q_b, q_c
# are floored; on a coarse int8 score grid that costs up to tens of LSB on
# a single probability, on a fine grid about one.
def lsb_bound(q_ln2: int) -> float:
    if q_ln2 >= 24:
        return 3.0
    if q_ln2 >= 16:
        return 10.0
    if q_ln2 >= 11:
        return 24.0
    return 64.0


@pytest.mark.parametrize("n", [1, 2, 7, 64, 375, 1500])
def test_softmax_vs_float64(oracle_lib, n):
    rng = np.random.default_rng(n)
    for S, prm in _grid_params(oracle_lib):
        for sig in (5, 30, 90):
            sc = np.clip(np.rint(rng.normal(0, sig, size=(40, n))), -127, 127).astype(np.int8)
            valid = rng.integers(1, n, size=40, endpoint=True).astype(np.int32)
            a = oracle_lib.isoftmax(sc, prm, valid).astype(np.float64)
            ref = _softmax_f64(sc, S, valid)
            err = np.abs(a - ref)
            assert err.max() <= lsb_bound(prm[0]), (S, prm, sig, err.max())
            assert err.mean() <= max(1.5, lsb_bound(prm[0]) / 8), (S, prm, sig, err.mean())


def test_softmax_row_sum_bounds(oracle_lib):
    # f = floor(2^32 / Sum), a_j = floor(e_j f / 2^24): the sum of a_j is at
    # most 256 and loses less than one per valid term plus ceil(Sum / 2^24).
    rng = np.random.default_rng(3)
    for S, prm in _grid_params(oracle_lib):
        for n in (1, 3, 50, 700):
            sc = np.clip(np.rint(rng.normal(0, 40, size=(30, n))), -127, 127).astype(np.int8)
            valid = rng.integers(1, n, size=30, endpoint=True).astype(np.int32)
            a = oracle_lib.isoftmax(sc, prm, valid).astype(np.int64)
            for r in range(30):
                nv = int(valid[r])
                row = sc[r, :nv].astype(np.int64)
                total = sum(oracle_lib.iexp(int(x - row.max()), prm) for x in row)
                s = int(a[r].sum())
                assert s <= 256
                assert s >= 256 - nv - math.ceil(total / 2 ** 24)
                assert (a[r, nv:] == 0).all()


def test_softmax_single_key_is_255(oracle_lib):
    for S, prm in _grid_params(oracle_lib):
        for x in (-127, 0, 5, 127):
            a = oracle_lib.isoftmax(np.array([[x]], np.int8), prm)
            assert a[0, 0] == 255   # 256 clamped onto the u8 grid


@pytest.mark.parametrize("n", [2, 3, 10, 64, 255, 256, 1000])
def test_softmax_uniform_closed_form(oracle_lib, n):
    # Equal scores: e_j = L(0), Sum = n L(0), a_j = floor(L(0) floor(2^32/(n L(0))) / 2^24).
    for S, prm in _grid_params(oracle_lib):
        L0 = prm[1] ** 2 + prm[2]
        want = (L0 * ((2 ** 32) // (n * L0))) >> 24
        a = oracle_lib.isoftmax(np.full((1, n), 17, np.int8), prm)
        assert (a == min(want, 255)).all()
        # floor(2^32 / (n L0)) loses less than L0 / 2^24 of the ideal 256 / n
        assert 256 / n - 1 - L0 / 2 ** 24 < int(a[0, 0]) <= 256 / n


def test_softmax_monotone_in_score(oracle_lib):
    rng = np.random.default_rng(4)
    for S, prm in _grid_params(oracle_lib):
        sc = np.clip(np.rint(rng.normal(0, 40, size=(20, 300))), -127, 127).astype(np.int8)
        a = oracle_lib.isoftmax(sc, prm)
        for r in range(20):
            order = np.argsort(sc[r], kind="stable")
            assert (np.diff(a[r][order].astype(np.int64)) >= 0).all()
