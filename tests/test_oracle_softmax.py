"""Pins of the oracle's integer softmax (I-BERT's integer exponential and
normalisation, which I-Parakeet uses for the attention, Sec. 2.2 and the
text after Eq. 11).  Constants from tests/golden/ibert_exp.txt; the error
bounds against the real exponential and softmax are derived step by step in
tests/ibert_bounds.py."""
import math
import os

import numpy as np
import pytest

import ibert_bounds as ib
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


# Score grids of the benchmark's encoder layers that are coarse (q_ln2 = 7,
# 8, 9): layer 13 (q_ln2 = 7), layers 1 and 2 (8, with frac(b / S) = 0.56
# and 0.68), layer 7 (9).  9 of the 24 layers have q_ln2 <= 9.
COARSE_LAYERS = (13, 1, 2, 7)
_COARSE = None
_GRIDS = None


def _coarse_grids():
    global _COARSE
    if _COARSE is None:
        out = [synth.layer(3, i).scales["S_s"] for i in COARSE_LAYERS]
        # q_ln2 = 7, 8, 9 with frac(b / S) on both sides of 1/2, so that a
        # rounded q_b differs from the floored one on some of them
        for q in (7, 8, 9):
            for f in (0.1, 0.5, 0.9):
                out.append(math.log(2) / (q + f))
        # b / S just above an integer (q_ln2 = 7, 8, 9): the floor of q_b
        # then loses almost nothing, and a q_c rounded up (frac(c / (a S^2))
        # = 0.885, 0.664, 0.926 here) shows above the fit
        for n, f in ((14, 0.01), (17, 0.01), (18, 0.005)):
            out.append(1.353 / (n + f))
        _COARSE = out
    return list(_COARSE)


def _grid_params(oracle_lib):
    global _GRIDS
    if _GRIDS is None:
        grids = []
        for w in range(5):
            lay = synth.layer(w, 0) if w != 3 else synth.draw(1, 8, 375, 128, 3000, p_mode="sinusoid")
            grids.append(lay.scales["S_s"])
        grids += _coarse_grids()
        for q in (5, 16, 32, 100, 400):
            grids.append(math.log(2) / (q + 0.25))
        _GRIDS = grids
    return [(S, oracle_lib.isoftmax_params(S)) for S in _GRIDS]


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


def test_params_worked_values(oracle_lib):
    # Worked by hand: S = ln2 / 8.5 gives ln2 / S = 8.5, b / S = 1.353 * 8.5 /
    # 0.693147 = 16.592 and c / (a S^2) = 0.344 * 72.25 / (0.3585 * 0.480453)
    # = 144.30: (q_ln2, q_b, q_c) = (8, 16, 144), each constant floored.
    # S = ln2 / 7.9: 7.9, 15.421, 124.64 -> (7, 15, 124).
    assert oracle_lib.isoftmax_params(math.log(2) / 8.5) == (8, 16, 144)
    assert oracle_lib.isoftmax_params(math.log(2) / 7.9) == (7, 15, 124)


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


def test_iexp_within_derived_bounds(oracle_lib):
    # Every value of the integer exponential against the real fit with the
    # error its floors allow (tests/ibert_bounds.py, steps 1-3): above it by
    # nothing (every floor rounds down), below it by less than
    # (2 a S (x + b)) 2^-z + a S^2.
    for S, prm in _grid_params(oracle_lib):
        d = np.arange(-254, 1)
        e = np.array([oracle_lib.iexp(int(x), prm) for x in d], dtype=np.float64)
        lo, hi = ib.iexp_bounds(S, d)
        got = e * ib.A * S * S
        assert (got <= hi * (1 + ib.REL)).all(), (S, prm, int(d[np.argmax(got - hi)]))
        assert (got > lo - ib.REL).all(), (S, prm, int(d[np.argmin(got - lo)]))


def test_iexp_derived_bounds_worked_value(oracle_lib):
    # S = ln2 / 8.5 (q_ln2 = 8): at d = 0 there is no shift and x = 0, so
    # a S^2 e(0) lies in (g(0) - 2 a b S - a S^2, g(0)] = (0.918781, 1.000273];
    # e(0) = 16^2 + 144 = 400 and 400 a S^2 = 0.953591.
    S = math.log(2) / 8.5
    lo, hi = ib.iexp_bounds(S, np.array([0.0]))
    assert abs(hi[0] - 1.000273) < 1e-6
    assert abs(lo[0] - 0.918781) < 1e-6
    assert oracle_lib.iexp(0, oracle_lib.isoftmax_params(S)) == 400
    assert lo[0] < 400 * 0.3585 * S * S <= hi[0]


@pytest.mark.parametrize("n", [1, 2, 7, 64, 375, 1500])
def test_softmax_vs_float64(oracle_lib, n):
    # Each probability within the derived bounds of tests/ibert_bounds.py
    # (steps 4-5) around 256 times the real softmax of the same scores.
    rng = np.random.default_rng(n)
    for S, prm in _grid_params(oracle_lib):
        for sig in (5, 30, 90):
            sc = np.clip(np.rint(rng.normal(0, sig, size=(40, n))), -127, 127).astype(np.int8)
            valid = rng.integers(1, n, size=40, endpoint=True).astype(np.int32)
            a = oracle_lib.isoftmax(sc, prm, valid).astype(np.float64)
            lower, upper, _ = ib.softmax_bounds(sc, S, valid)
            assert (a <= upper).all(), (S, prm, sig, float(np.max(a - upper)))
            assert (a >= lower).all(), (S, prm, sig, float(np.max(lower - a)))


def test_softmax_two_keys_coarse(oracle_lib):
    # Two keys q_ln2 grid steps apart on a coarse grid: the real weights are
    # 1 and exp(-q_ln2 S) (between 1/2 and 0.55), the integer ones L(0) and
    # floor(L(0) / 2).  The result lies within the derived bounds, and the
    # bounds are tight here: less than 5 steps wide.
    for S in _coarse_grids():
        prm = oracle_lib.isoftmax_params(S)
        sc = np.array([[100, 100 - prm[0]]], np.int8)
        valid = np.array([2], np.int32)
        a = oracle_lib.isoftmax(sc, prm, valid).astype(np.float64)
        lower, upper, _ = ib.softmax_bounds(sc, S, valid)
        assert ((lower <= a) & (a <= upper)).all(), (S, a, lower, upper)
        assert (upper - lower < 5).all(), (S, lower, upper)


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
