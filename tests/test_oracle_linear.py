"""Pins of the linear-layer oracle (Sec. 2.2, Eqs. 6-7) against what the
paper and the mathematics fix, not against the oracle itself:

* special cases with closed forms: the identity layer (W = 2 I, m = 2^30,
  n = 31 gives y = x), halving with ties toward +infinity (m = 2^30, n = 31
  is round(acc / 2)), the symmetric clamp;
* the integer product against numpy's int64 matmul (an independent route);
* the whole quantised layer against the real-valued layer it stands for
  (float64, dequantised inputs, quantised output): within one step of the
  output grid, almost always equal;
* the head-split layouts against plain numpy reshapes and transposes.
"""
import numpy as np
import pytest

import oracle
import synth

HALF_M = 2 ** 30          # m = 2^30 with s = 0: y = round(acc / 2)


def _halving(acc):
    # round(acc / 2) with ties toward +infinity, on the int8 grid
    return np.clip(np.floor_divide(acc + 1, 2), -127, 127).astype(np.int8)


def test_identity_layer():
    rng = np.random.default_rng(1)
    K = 256
    x = rng.integers(-127, 128, size=(3, 7, K), dtype=np.int8)
    w = (2 * np.eye(K)).astype(np.int8)
    m = np.full(K, HALF_M, np.int32)
    s = np.zeros(K, np.int32)
    np.testing.assert_array_equal(oracle.linear(x, w, None, m, s), x)


def test_product_matches_numpy_matmul():
    rng = np.random.default_rng(2)
    B, T, K, N = 2, 9, 384, 256
    x = rng.integers(-4, 5, size=(B, T, K), dtype=np.int8)
    w = rng.integers(-3, 4, size=(N, K), dtype=np.int8)
    bias = rng.integers(-40, 41, size=N).astype(np.int32)
    acc = x.reshape(-1, K).astype(np.int64) @ w.astype(np.int64).T + bias
    want = _halving(acc).reshape(B, T, N)
    got = oracle.linear(x, w, bias, np.full(N, HALF_M, np.int32), np.zeros(N, np.int32))
    np.testing.assert_array_equal(got, want)


def test_ties_round_up_and_clamp_is_symmetric():
    # one input channel carrying acc directly: x = acc, w = 1, m = 2^30
    acc = np.array([-127, -126, -5, -3, -1, 0, 1, 3, 5, 126, 127], np.int64)
    xs = acc.astype(np.int8).reshape(1, -1, 1)
    w = np.ones((1, 1), np.int8)
    m = np.array([HALF_M], np.int32)
    s = np.array([0], np.int32)
    got = oracle.linear(xs, w, None, m, s).reshape(-1)
    np.testing.assert_array_equal(got, _halving(acc))
    # ties: -3/2 -> -1, -1/2 -> 0, 1/2 -> 1, 3/2 -> 2
    got = oracle.linear(np.array([[[-3], [-1], [1], [3]]], np.int8), w, None, m, s).reshape(-1)
    np.testing.assert_array_equal(got, [-1, 0, 1, 2])
    # saturation: never -128
    big = oracle.linear(np.full((1, 1, 64), -127, np.int8), np.full((1, 64), 127, np.int8),
                        None, np.array([2 ** 31 - 1], np.int32), np.array([0], np.int32))
    assert big.item() == -127


@pytest.mark.parametrize("seed,groups", [(3, 1), (4, 3)])
def test_layer_vs_real_valued_layer(seed, groups):
    c = synth.linear(2, 40, 1024, 384, seed=seed, groups=groups)
    m, s = oracle.linear_constants(c.s_x, c.s_w, c.s_y_per_channel())
    got = oracle.linear(c.x, c.w, c.bias, m, s).astype(np.int64)
    # the real-valued layer: dequantise (Eq. 6), multiply, quantise onto S_y
    xr = c.x.astype(np.float64) * c.s_x
    wr = c.w.astype(np.float64) * c.s_w[:, None]
    br = c.bias.astype(np.float64) * c.s_x * c.s_w
    yr = xr.reshape(-1, xr.shape[-1]) @ wr.T + br
    ref = np.clip(np.floor(yr / c.s_y_per_channel()[None, :] + 0.5), -127, 127)
    diff = np.abs(got.reshape(ref.shape) - ref)
    assert diff.max() <= 1
    assert (diff == 0).mean() > 0.99


def test_head_split_layouts():
    rng = np.random.default_rng(5)
    B, T, K, N, G = 2, 11, 256, 768, 3
    x = rng.integers(-127, 128, size=(B, T, K), dtype=np.int8)
    w = rng.integers(-127, 128, size=(N, K), dtype=np.int8)
    bias = rng.integers(-1000, 1000, size=N).astype(np.int32)
    m = rng.integers(2 ** 30, 2 ** 31, size=N).astype(np.int32)
    s = rng.integers(8, 14, size=N).astype(np.int32)
    rows = oracle.linear(x, w, bias, m, s)
    # input in heads: [B, K/128, T, 128]
    xh = np.ascontiguousarray(x.reshape(B, T, K // 128, 128).transpose(0, 2, 1, 3))
    np.testing.assert_array_equal(oracle.linear(xh, w, bias, m, s, x_layout=oracle.HEADS), rows)
    # output in heads, G groups: [G, B, N/G/128, T, 128]
    yh = oracle.linear(x, w, bias, m, s, y_layout=oracle.HEADS, groups=G)
    want = rows.reshape(B, T, G, N // G // 128, 128).transpose(2, 0, 3, 1, 4)
    np.testing.assert_array_equal(yh, want)


def test_shapes_rejected():
    x = np.zeros((1, 2, 130), np.int8)
    w = np.zeros((128, 130), np.int8)
    m = np.full(128, HALF_M, np.int32)
    s = np.zeros(128, np.int32)
    with pytest.raises(oracle.OracleError):
        oracle.linear(np.zeros((1, 1, 2, 128), np.int8), np.zeros((128, 130), np.int8), None,
                      m, s, x_layout=oracle.HEADS)
    with pytest.raises(oracle.OracleError):
        oracle.linear(x, w, None, m, np.full(128, 32, np.int32))
    with pytest.raises(oracle.OracleError):
        oracle.linear(x, w, None, m, s, y_layout=oracle.HEADS, groups=3)
