"""Pins of the oracle's remaining Conformer-block parts (Sec. 2.1 Eqs. 1-5,
Sec. 2.2, Sec. 3.2, Sec. 3.3) against the mathematics:

* residual addition: against the real-valued sum (one output step), exact
  closed forms with one input zero;
* GLU: GLU(z, z) is the Swish already pinned to Table 3; against the
  real-valued a sigma_hat(b) (one step) and the true a sigma(b); b beyond
  the clip point gives a or 0;
* depthwise convolution with folded BatchNorm: the integer accumulator
  against numpy brute force with zero padding at both ends (halving closed
  form on the output), against the real-valued convolution (one INT16 step);
* INT16 Swish: every one of the 65535 inputs against the real-valued
  approximation (one step) and the true Swish (Table 3's error + a step).
"""
import os

import numpy as np
import pytest

import oracle
from test_oracle_swish import golden, sw, sw_hat


def sig_hat(b):
    u = b / 2.0
    th = np.sign(u) * (oracle.SWISH_A * (np.minimum(np.abs(u), oracle.SWISH_C) - oracle.SWISH_C) ** 2 + 1.0)
    return (1.0 + th) / 2.0


def rnd(v):
    return np.floor(v + 0.5)


@pytest.mark.parametrize("alpha", [1.0, 0.5])
def test_residual_vs_real_sum(alpha):
    rng = np.random.default_rng(1)
    x = rng.integers(-127, 128, size=20000).astype(np.int8)
    y = rng.integers(-127, 128, size=20000).astype(np.int8)
    s_x, s_y = 0.05, 0.03
    s_z = (127 * s_x + alpha * 127 * s_y) / 127 * 0.8
    m_x, m_y, s = oracle.residual_params(s_x, s_y, s_z, alpha)
    got = oracle.residual(x, y, m_x, m_y, s).astype(np.int64)
    ref = np.clip(rnd((s_x * x + alpha * s_y * y.astype(np.float64)) / s_z), -127, 127)
    d = np.abs(got - ref)
    assert d.max() <= 1 and (d == 0).mean() > 0.99
    # one input zero: a single dyadic requantisation, exact
    z = oracle.residual(x, np.zeros_like(y), m_x, m_y, s).astype(np.int64)
    e = 31 + s
    np.testing.assert_array_equal(z, np.clip((m_x * x.astype(np.int64) + (1 << (e - 1))) >> e, -127, 127))


def test_glu_of_equal_halves_is_the_swish():
    z = np.arange(-127, 128, dtype=np.int8)
    for s_z, s_y in [(8 / 127, 8 / 127), (6 / 127, 5 / 127)]:
        p = oracle.swish_params(s_z, s_y)
        assert oracle.glu_params(s_z, s_z, s_y) == p
        ab = np.concatenate([z, z]).reshape(1, -1)
        np.testing.assert_array_equal(oracle.glu(ab, p)[0], oracle.swish(z, p))


@pytest.mark.parametrize("s_a,s_b,s_y", [(0.05, 0.06, 0.03), (0.02, 0.08, 0.01)])
def test_glu_vs_real(s_a, s_b, s_y):
    rng = np.random.default_rng(2)
    C = 512
    ab = rng.integers(-127, 128, size=(64, 2 * C)).astype(np.int8)
    p = oracle.glu_params(s_a, s_b, s_y)
    got = oracle.glu(ab, p).astype(np.int64)
    a = ab[:, :C] * s_a
    b = ab[:, C:].astype(np.float64) * s_b
    ref = np.clip(rnd(a * sig_hat(b) / s_y), -127, 127)
    # rounding the clip point q_c = round(2c/S_b) moves D by at most S_b/4, so
    # sigma moves by at most |a*| (S_b/8) (2c + S_b/4); the gain |a| / S_y
    # turns that into output steps, plus one step of final rounding
    dsig = abs(oracle.SWISH_A) * (s_b / 8) * (2 * oracle.SWISH_C + s_b / 4)
    d = np.abs(got - ref)
    assert (d <= 1 + np.abs(a) / s_y * dsig + 1e-9).all()
    assert (d == 0).mean() > 0.85
    # against the true sigmoid: |sigma_hat - sigma| <= Table 3's error / |x| bound
    true = a / (1.0 + np.exp(-b))
    inside = np.abs(true) < 120 * s_y
    err_sig = np.abs(sig_hat(np.linspace(-30, 30, 600001)) - 1 / (1 + np.exp(-np.linspace(-30, 30, 600001)))).max()
    assert np.abs(got * s_y - true)[inside].max() <= np.abs(a).max() * err_sig + s_y
    # saturation: b <= -q_c gives 0, b >= q_c gives round(a S_a / S_y)
    bb = ab[:, C:].astype(np.int64)
    assert (got[bb <= -p.q_c] == 0).all()
    hi = bb >= p.q_c
    assert np.abs(got[hi] - np.clip(rnd(a[hi] / s_y), -127, 127)).max() <= 1


def dw_acc_numpy(x, w, bias):
    B, T, C = x.shape
    K = w.shape[1]
    xp = np.zeros((B, T + K - 1, C), np.int64)
    xp[:, K // 2:K // 2 + T] = x
    acc = np.zeros((B, T, C), np.int64) + bias
    for k in range(K):
        acc += xp[:, k:k + T] * w[:, k].astype(np.int64)
    return acc


@pytest.mark.parametrize("T,K", [(1, 9), (5, 9), (64, 9), (37, 3), (20, 1)])
def test_dwconv_integer_part_vs_brute_force(T, K):
    rng = np.random.default_rng(T + K)
    B, C = 2, 96
    x = rng.integers(-127, 128, size=(B, T, C)).astype(np.int8)
    w = rng.integers(-127, 128, size=(C, K)).astype(np.int8)
    bias = rng.integers(-5000, 5000, size=C).astype(np.int32)
    m = np.full(C, 2 ** 30, np.int32)
    s = np.zeros(C, np.int32)
    got = oracle.dwconv(x, w, bias, m, s).astype(np.int64)
    acc = dw_acc_numpy(x, w, bias)
    np.testing.assert_array_equal(got, np.clip(np.floor_divide(acc + 1, 2), -32767, 32767))


def test_dwconv_vs_real_conv():
    rng = np.random.default_rng(9)
    B, T, C, K = 2, 50, 128, 9
    x = rng.integers(-127, 128, size=(B, T, C)).astype(np.int8)
    w = rng.integers(-127, 128, size=(C, K)).astype(np.int8)
    bias = rng.integers(-3000, 3000, size=C).astype(np.int32)
    s_x, s_w, s_y = 0.04, rng.uniform(0.001, 0.01, C), 64.0 / 32767
    m, s = oracle.linear_constants(s_x, s_w, np.full(C, s_y))
    got = oracle.dwconv(x, w, bias, m, s).astype(np.int64)
    real = dw_acc_numpy(x, w, bias) * (s_x * s_w)
    ref = np.clip(rnd(real / s_y), -32767, 32767)
    d = np.abs(got - ref)
    assert d.max() <= 1 and (d == 0).mean() > 0.99


@pytest.mark.parametrize("s_z,s_y", [(8 / 32767, 8 / 127), (12 / 32767, 6 / 127), (5 / 32767, 3 / 127)])
def test_swish16_every_input(s_z, s_y):
    p = oracle.swish16_params(s_z, s_y)
    z = np.arange(-32767, 32768, dtype=np.int16)
    got = oracle.swish16(z, p).astype(np.int64)
    x = z * s_z
    ref = np.clip(rnd(sw_hat(x, oracle.SWISH_A, oracle.SWISH_C) / s_y), -127, 127)
    d = np.abs(got - ref)
    assert d.max() <= 1 and (d == 0).mean() > 0.99
    inside = np.abs(sw(x)) <= 127 * s_y
    assert np.abs(got * s_y - sw(x))[inside].max() <= golden()["max_err"] + s_y
    assert got[z == 0].item() == 0
    assert (got[z.astype(np.int64) <= -p.q_c] == 0).all()


def test_swish16_domain():
    # q_one = round(1 / S_t) must stay below 2^31: input ranges below about 4
    with pytest.raises(ValueError):
        oracle.swish16_params(3 / 32767, 3 / 127)
