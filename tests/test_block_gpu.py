"""Parity of the remaining Conformer-block kernels with the oracle (bit-exact):
residual additions (alone and fused into a projection), the GLU projection, the depthwise convolution with
folded BatchNorm on INT16 followed by the Swish."""
import numpy as np
import pytest

from guard import Guarded

import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def ip():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30846_gb300 as mod
    mod.load()
    return mod


@pytest.fixture(scope="module")
def orc():
    import oracle
    oracle.build()
    return oracle


def _d(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def assert_same(got, want):
    bad = got != want
    if bad.any():
        idx = np.argwhere(bad)[:5]
        raise AssertionError(f"{int(bad.sum())} of {got.size} differ; first at {idx.tolist()}: "
                             f"gpu {got[tuple(idx[0])]} oracle {want[tuple(idx[0])]}")


@pytest.mark.parametrize("n,alpha", [(16, 1.0), (1000, 0.5), (12000 * 1024 + 7, 0.5), (3, 1.0)])
def test_residual(ip, orc, n, alpha):
    rng = np.random.default_rng(n)
    x = rng.integers(-127, 128, size=n).astype(np.int8)
    y = rng.integers(-127, 128, size=n).astype(np.int8)
    m_x, m_y, s = orc.residual_params(0.05, 0.03, 0.06, alpha)
    g = Guarded(x.shape, torch.int8)
    got = ip.residual_i8(_d(x), _d(y), m_x, m_y, s, out=g.view).cpu().numpy()
    g.check()
    assert_same(got, orc.residual(x, y, m_x, m_y, s))


@pytest.mark.parametrize("B,T,K,N,alpha", [(1, 5, 128, 128, 1.0), (2, 130, 256, 384, 0.5),
                                           (3, 200, 1024, 256, 0.5), (32, 375, 1024, 1024, 1.0)])
def test_linear_residual(ip, orc, B, T, K, N, alpha):
    # the projection with the residual addition fused, against the oracle's
    # linear layer followed by its residual addition; the tile's last frames
    # (B T not a multiple of 128) and both column halves of every tile
    lc = synth.linear(B, T, K, N, seed=700 + T + N)
    m, s = orc.linear_constants(lc.s_x, lc.s_w, lc.s_y_per_channel())
    rng = np.random.default_rng(T + N)
    res = rng.integers(-127, 128, size=(B, T, N)).astype(np.int8)
    s_y = float(lc.s_y[0])
    rp = orc.residual_params(0.05, s_y, 1.2 * max(0.05, s_y), alpha)   # both ratios below 1
    want = orc.residual(res, orc.linear(lc.x, lc.w, lc.bias, m, s), *rp)
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    g = Guarded(want.shape, torch.int8)
    got = ip.linear_residual_i8(_d(lc.x), _d(lc.w), _d(lc.bias), _d(m), _d(s), _d(res), *rp,
                                out=g.view, workspace=ws)
    assert ip.status(ws) == 0
    g.check()
    assert_same(got.cpu().numpy(), want)


# Hand-picked constants at the edges of the residual's domain: the largest
# multipliers, the shortest and longest shifts, and (2^30, 2^30, 0), where
# (x + y) / 2 lands on a half step for every odd sum (the round-half-up tie).
EDGE_RESIDUAL = [(2 ** 31 - 1, 2 ** 31 - 1, 31), (2 ** 31 - 1, 1, 0), (1, 2 ** 31 - 1, 0),
                 (2 ** 30, 2 ** 30, 0), (2 ** 30, 2 ** 29, 1), (0, 2 ** 31 - 1, 31),
                 (12345, 2 ** 31 - 1, 7), (2 ** 31 - 1, 0, 30)]


@pytest.mark.parametrize("m_x,m_y,s_r", EDGE_RESIDUAL)
def test_residual_edge_constants(ip, orc, m_x, m_y, s_r):
    # every (x, y) pair of int8 values, bit for bit against the oracle
    v = np.arange(-128, 128, dtype=np.int16)
    x = np.repeat(v, 256).astype(np.int8)
    y = np.tile(v, 256).astype(np.int8)
    g = Guarded(x.shape, torch.int8)
    got = ip.residual_i8(_d(x), _d(y), m_x, m_y, s_r, out=g.view).cpu().numpy()
    g.check()
    assert_same(got, orc.residual(x, y, m_x, m_y, s_r))


@pytest.mark.parametrize("m_x,m_y,s_r", EDGE_RESIDUAL)
def test_linear_residual_edge_constants(ip, orc, m_x, m_y, s_r):
    B, T, K, N = 2, 70, 256, 256
    lc = synth.linear(B, T, K, N, seed=731)
    m, s = orc.linear_constants(lc.s_x, lc.s_w, lc.s_y_per_channel())
    rng = np.random.default_rng(s_r + 7)
    res = rng.integers(-128, 128, size=(B, T, N)).astype(np.int8)
    want = orc.residual(res, orc.linear(lc.x, lc.w, lc.bias, m, s), m_x, m_y, s_r)
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    g = Guarded(want.shape, torch.int8)
    got = ip.linear_residual_i8(_d(lc.x), _d(lc.w), _d(lc.bias), _d(m), _d(s), _d(res), m_x, m_y,
                                s_r, out=g.view, workspace=ws)
    assert ip.status(ws) == 0
    g.check()
    assert_same(got.cpu().numpy(), want)


def test_linear_residual_in_place(ip, orc):
    # res and y the same buffer: the residual stream updated in place
    B, T, K, N = 3, 130, 256, 384
    lc = synth.linear(B, T, K, N, seed=732)
    m, s = orc.linear_constants(lc.s_x, lc.s_w, lc.s_y_per_channel())
    res = np.random.default_rng(5).integers(-127, 128, size=(B, T, N)).astype(np.int8)
    rp = orc.residual_params(0.05, float(lc.s_y[0]), 1.2 * max(0.05, float(lc.s_y[0])), 0.5)
    want = orc.residual(res, orc.linear(lc.x, lc.w, lc.bias, m, s), *rp)
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    g = Guarded(res.shape, torch.int8)
    g.view.copy_(_d(res))
    got = ip.linear_residual_i8(_d(lc.x), _d(lc.w), _d(lc.bias), _d(m), _d(s), g.view, *rp,
                                out=g.view, workspace=ws)
    assert ip.status(ws) == 0
    g.check()
    assert got.data_ptr() == g.view.data_ptr()
    assert_same(got.cpu().numpy(), want)


def interleave(w):
    N2 = w.shape[0]
    C = N2 // 2
    out = np.empty_like(w)
    out[0::2] = w[:C]
    out[1::2] = w[C:]
    return out


@pytest.mark.parametrize("B,T,K,C", [(1, 5, 128, 64), (2, 130, 256, 192), (32, 375, 1024, 1024)])
def test_glu_projection(ip, orc, B, T, K, C):
    # the ConvBlock's first pointwise convolution, 2C outputs [a | b] -> C
    lc = synth.linear(B, T, K, 2 * C, seed=500 + T, groups=2)
    m, s = orc.linear_constants(lc.s_x, lc.s_w, lc.s_y_per_channel())
    g = orc.glu_params(float(lc.s_y[0]), float(lc.s_y[1]), 0.8 * float(lc.s_y[0]))
    ab = orc.linear(lc.x, lc.w, lc.bias, m, s)
    want = orc.glu(ab, g)
    perm = np.empty(2 * C, np.int64)
    perm[0::2] = np.arange(C)
    perm[1::2] = np.arange(C) + C
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    gd = Guarded(want.shape, torch.int8)
    got = ip.linear_glu_i8(_d(lc.x), _d(interleave(lc.w)), _d(lc.bias[perm]), _d(m[perm]),
                           _d(s[perm]), (g.q_c, g.q_one, g.m, g.s), out=gd.view, workspace=ws)
    assert ip.status(ws) == 0
    gd.check()
    assert_same(got.cpu().numpy(), want)


# C a multiple of 4 takes the four-channels-per-thread kernel (C = 300 and
# 260: a partly filled CTA), C = 258 and 66 the one-channel kernel.
@pytest.mark.parametrize("B,T,C,K", [(1, 1, 256, 9), (2, 33, 256, 9), (3, 100, 512, 5),
                                     (32, 375, 1024, 9), (1, 70, 300, 15), (2, 40, 256, 1),
                                     (2, 40, 256, 3), (1, 50, 256, 7), (1, 50, 256, 11),
                                     (1, 50, 256, 13), (2, 37, 260, 15), (1, 33, 4, 3),
                                     (1, 40, 258, 9), (2, 45, 66, 5)])
def test_dwconv_swish(ip, orc, B, T, C, K):
    rng = np.random.default_rng(T * C + K)
    x = rng.integers(-127, 128, size=(B, T, C)).astype(np.int8)
    w = rng.integers(-127, 128, size=(C, K)).astype(np.int8)
    bias = rng.integers(-20000, 20000, size=C).astype(np.int32)
    s_x, s_w = 0.04, rng.uniform(0.001, 0.01, C)
    s_bn = 40.0 / 32767                      # INT16 grid of the folded BatchNorm output
    m, s = orc.linear_constants(s_x, s_w, np.full(C, s_bn))
    p16 = orc.swish16_params(s_bn, 5.0 / 127)
    want = orc.swish16(orc.dwconv(x, w, bias, m, s), p16)
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    g = Guarded(want.shape, torch.int8)
    got = ip.dwconv_swish_i8(_d(x), _d(w), _d(bias), _d(m), _d(s),
                             (p16.q_c, p16.q_one, p16.m, p16.s), out=g.view, workspace=ws)
    assert ip.status(ws) == 0
    g.check()
    assert_same(got.cpu().numpy(), want)


def _dw_case(rng, B, T, C, K):
    x = rng.integers(-127, 128, size=(B, T, C)).astype(np.int8)
    w = rng.integers(-127, 128, size=(C, K)).astype(np.int8)
    bias = rng.integers(-20000, 20000, size=C).astype(np.int32)
    m, s = (rng.integers(1, 2 ** 31, size=C).astype(np.int32),
            rng.integers(10, 20, size=C).astype(np.int32))
    return x, w, bias, m, s


def test_dwconv_unaligned_buffers_take_the_one_channel_kernel(ip, orc):
    # x and y one byte off a 4-byte boundary (C a multiple of 4): the
    # one-channel kernel runs and gives the same bytes as the oracle
    rng = np.random.default_rng(77)
    B, T, C, K = 2, 50, 256, 9
    x, w, bias, m, s = _dw_case(rng, B, T, C, K)
    p16 = orc.swish16_params(40.0 / 32767, 5.0 / 127)
    want = orc.swish16(orc.dwconv(x, w, bias, m, s), p16)
    xs = torch.zeros(B * T * C + 1, dtype=torch.int8, device="cuda")
    xs[1:] = _d(x).flatten()
    ys = torch.zeros(B * T * C + 1, dtype=torch.int8, device="cuda")
    got = ip.dwconv_swish_i8(xs[1:].view(B, T, C), _d(w), _d(bias), _d(m), _d(s),
                             (p16.q_c, p16.q_one, p16.m, p16.s), out=ys[1:].view(B, T, C))
    assert_same(got.cpu().numpy(), want)
    assert int(ys[0]) == 0


@pytest.mark.parametrize("C", [256, 258])
def test_dwconv_extreme_constants(ip, orc, C):
    # multipliers 0, 1 and 2^31 - 1, shifts 0, 1, 30 and 31, biases at the
    # domain's edges, and Swish constants at the edges of theirs (q_one =
    # 2^31 - 1 with the largest q_c it allows; m_sw = 2^31 - 1 at s = 0 and
    # 31): every rounding and both clamps, in both kernels
    rng = np.random.default_rng(C)
    B, T, K = 1, 64, 9
    x = rng.integers(-127, 128, size=(B, T, C)).astype(np.int8)
    x[0, ::7] = 127
    x[0, 3::7] = -127
    w = rng.integers(-127, 128, size=(C, K)).astype(np.int8)
    w[::5] = 127
    mv = np.array([0, 1, 2 ** 31 - 1, 2 ** 30, 123456789], np.int64)
    sv = np.array([0, 1, 30, 31, 17], np.int64)
    bv = np.array([2 ** 30 - 1, -(2 ** 30 - 1), 0, 12345, -54321], np.int64)
    m = mv[rng.integers(0, 5, C)].astype(np.int32)
    s = sv[rng.integers(0, 5, C)].astype(np.int32)
    bias = bv[rng.integers(0, 5, C)].astype(np.int32)
    for p16 in (orc.Swish16Params(46340, 2 ** 31 - 1, 2 ** 31 - 1, 31),
                orc.Swish16Params(46340, 2 ** 31 - 1, 2 ** 31 - 1, 0),
                orc.Swish16Params(1, 1, 2 ** 31 - 1, 31),
                orc.Swish16Params(300, 90000, 1, 0)):
        want = orc.swish16(orc.dwconv(x, w, bias, m, s), p16)
        ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
        got = ip.dwconv_swish_i8(_d(x), _d(w), _d(bias), _d(m), _d(s),
                                 (p16.q_c, p16.q_one, p16.m, p16.s), workspace=ws)
        assert ip.status(ws) == 0
        assert_same(got.cpu().numpy(), want)


def test_dwconv_saturating_int16(ip, orc):
    # accumulators far beyond the INT16 grid: clamped before the Swish
    B, T, C, K = 1, 40, 256, 9
    x = np.full((B, T, C), 127, np.int8)
    x[:, ::2] = -127
    w = np.full((C, K), 127, np.int8)
    bias = np.zeros(C, np.int32)
    m = np.full(C, 2 ** 31 - 1, np.int32)
    s = np.zeros(C, np.int32)
    p16 = orc.swish16_params(40.0 / 32767, 5.0 / 127)
    want = orc.swish16(orc.dwconv(x, w, bias, m, s), p16)
    got = ip.dwconv_swish_i8(_d(x), _d(w), _d(bias), _d(m), _d(s),
                             (p16.q_c, p16.q_one, p16.m, p16.s))
    assert_same(got.cpu().numpy(), want)
