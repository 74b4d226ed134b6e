"""Pins of the integer LayerNorm oracle (Sec. 2.1, Eqs. 1-4; Sec. 2.2) against
the mathematics, not against itself:

* the integer square root equals Python's math.isqrt (exhaustive on small
  n, around every tested perfect square, random large n);
* the whole LayerNorm against a float64 LayerNorm of the dequantised input
  (within one step of the output grid, almost always equal);
* exact invariances: adding a constant to a row changes nothing, permuting
  the channels (with gamma and beta) permutes the output;
* closed forms: a constant row gives round(beta / S_y); a row of +a and -a
  halves normalises to +-1 exactly, giving round((+-gamma + beta) / S_y).
"""
import math

import numpy as np
import pytest

import oracle


def test_isqrt_matches_math_isqrt():
    for n in range(0, 200001):
        if n % 7 == 0 or n < 5000:
            assert oracle.isqrt(n) == math.isqrt(n)
    rng = np.random.default_rng(1)
    for k in list(rng.integers(1, 2 ** 31 - 1, size=300)) + [2 ** 31 - 1, 65536, 3]:
        k = int(k)
        for n in (k * k - 1, k * k, k * k + 1, k * k + 2 * k):
            if 0 <= n < 2 ** 62:
                assert oracle.isqrt(n) == math.isqrt(n), n
    for n in rng.integers(0, 2 ** 62, size=500):
        assert oracle.isqrt(int(n)) == math.isqrt(int(n))


def case(rows, d, seed, eps=1e-5):
    rng = np.random.default_rng(seed)
    x = np.clip(np.rint(rng.normal(rng.normal(0, 10), 35, size=(rows, d))), -127, 127).astype(np.int8)
    gamma = rng.uniform(0.3, 2.0, size=d) * rng.choice([-1.0, 1.0], size=d, p=[0.1, 0.9])
    beta = rng.normal(0.0, 0.5, size=d)
    s_x = rng.uniform(2.0, 6.0) / 127
    s_y = rng.uniform(3.0, 8.0) / 127
    return x, gamma, beta, s_x, s_y, eps


def float_layernorm(x, gamma, beta, s_x, s_y, eps):
    xr = x.astype(np.float64) * s_x
    mu = xr.mean(axis=-1, keepdims=True)
    var = ((xr - mu) ** 2).mean(axis=-1, keepdims=True)
    yr = gamma * (xr - mu) / np.sqrt(var + eps) + beta
    return np.clip(np.floor(yr / s_y + 0.5), -127, 127)


@pytest.mark.parametrize("d,seed", [(1024, 1), (1024, 2), (512, 3), (2048, 4), (80, 5)])
def test_layernorm_vs_float64(d, seed):
    x, gamma, beta, s_x, s_y, eps = case(64, d, seed)
    c = oracle.layernorm_constants(s_x, gamma, beta, s_y, eps)
    got = oracle.layernorm(x, c).astype(np.int64)
    ref = float_layernorm(x, gamma, beta, s_x, s_y, eps)
    diff = np.abs(got - ref)
    assert diff.max() <= 1
    assert (diff == 0).mean() > 0.99


def test_shift_invariance_is_exact():
    x, gamma, beta, s_x, s_y, eps = case(32, 1024, 6)
    x = np.clip(x, -100, 100).astype(np.int8)
    c = oracle.layernorm_constants(s_x, gamma, beta, s_y, eps)
    base = oracle.layernorm(x, c)
    for k in (-27, -1, 1, 13, 27):
        np.testing.assert_array_equal(oracle.layernorm((x.astype(np.int16) + k).astype(np.int8), c),
                                      base)


def test_channel_permutation():
    x, gamma, beta, s_x, s_y, eps = case(16, 1024, 7)
    perm = np.random.default_rng(8).permutation(1024)
    c = oracle.layernorm_constants(s_x, gamma, beta, s_y, eps)
    cp = oracle.layernorm_constants(s_x, gamma[perm], beta[perm], s_y, eps)
    np.testing.assert_array_equal(oracle.layernorm(np.ascontiguousarray(x[:, perm]), cp),
                                  oracle.layernorm(x, c)[:, perm])


def test_constant_row_gives_beta():
    d = 1024
    _, gamma, beta, s_x, s_y, eps = case(1, d, 9)
    c = oracle.layernorm_constants(s_x, gamma, beta, s_y, eps)
    for v in (-127, -3, 0, 5, 127):
        y = oracle.layernorm(np.full((1, d), v, np.int8), c).astype(np.int64)[0]
        np.testing.assert_array_equal(y, np.clip(np.floor(beta / s_y + 0.5), -127, 127))


def test_two_valued_row_normalises_to_one():
    d = 1024
    _, gamma, beta, s_x, s_y, _ = case(1, d, 10)
    c = oracle.layernorm_constants(s_x, gamma, beta, s_y, eps=0.0)
    assert c.eps_c == 0
    for a in (1, 7, 64, 127):
        row = np.where(np.arange(d) % 2 == 0, a, -a).astype(np.int8)[None, :]
        y = oracle.layernorm(row, c).astype(np.int64)[0]
        sign = np.where(np.arange(d) % 2 == 0, 1.0, -1.0)
        want = np.clip(np.floor((sign * gamma + beta) / s_y + 0.5), -127, 127)
        assert np.abs(y - want).max() <= 1
        assert (y == want).mean() > 0.99


def test_domain():
    c = oracle.layernorm_constants(0.03, np.ones(8), np.zeros(8), 0.03)
    with pytest.raises(oracle.OracleError):
        oracle.layernorm(np.zeros((2, 1), np.int8), oracle.NormConstants(c.eps_c, c.M[:1], c.B[:1], c.E[:1]))
    bad = oracle.NormConstants(c.eps_c, c.M, c.B, np.full(8, 63, np.int32))
    with pytest.raises(oracle.OracleError):
        oracle.layernorm(np.zeros((2, 8), np.int8), bad)


def test_epsilon_matters_for_small_variance():
    # rows of 0/1 values: the variance is comparable with epsilon
    rng = np.random.default_rng(11)
    d = 1024
    x = rng.integers(0, 2, size=(16, d)).astype(np.int8)
    gamma = rng.uniform(0.5, 1.5, size=d)
    beta = rng.normal(0.0, 0.2, size=d)
    s_x, s_y, eps = 0.02, 4.0 / 127, 2e-4
    c = oracle.layernorm_constants(s_x, gamma, beta, s_y, eps)
    got = oracle.layernorm(x, c).astype(np.int64)
    ref = float_layernorm(x, gamma, beta, s_x, s_y, eps)
    assert np.abs(got - ref).max() <= 1
    assert (got == ref).mean() > 0.98
