"""Seeded random sweeps of the Conformer block's other kernels through the C
ABI against the oracle, bit for bit (Sec. 2.1 Eqs. 1-5, Sec. 2.2 Eqs. 6-7,
Sec. 3.2 Eqs. 12-13, Sec. 3.3): the integer linear layer in each of its
variants (plain, fused Swish, fused GLU, fused residual addition) with
random shapes, input and output layouts, bias or none; the integer
LayerNorm with random row counts, widths and grids; the depthwise
convolution + INT16 BatchNorm + Swish with random shapes, kernel sizes,
per-channel constants and both of its kernels (C a multiple of 4 or not).
Guard bytes around every output catch a write outside it.
"""
import numpy as np
import pytest

import synth
from guard import Guarded

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


def assert_same(got, want, what):
    bad = got != want
    if bad.any():
        idx = np.argwhere(bad)[0].tolist()
        raise AssertionError(f"{what}: {int(bad.sum())} of {got.size} differ; first at {idx}")


def _interleave(w):
    C = w.shape[0] // 2
    out = np.empty_like(w)
    out[0::2] = w[:C]
    out[1::2] = w[C:]
    return out


@pytest.mark.parametrize("i", range(16))
def test_random_linear(ip, orc, i):
    rng = np.random.default_rng(70_000 + i)
    variant = ["plain", "plain", "swish", "glu", "residual"][i % 5]
    K = 128 * int(rng.integers(1, 17))
    G = 3 if (variant == "plain" and rng.integers(0, 2)) else 1
    N = 128 * G * int(rng.integers(1, 7 if G == 1 else 3))
    B = int(rng.integers(1, 6))
    T = int(rng.integers(1, 300))
    while B * T * K * N > 150_000_000 and T > 1:
        T //= 2
    bias = bool(rng.integers(0, 4))          # a quarter of the cases without bias
    x_layout = int(rng.integers(0, 2)) if variant == "plain" else 0
    y_layout = 1 if G == 3 else 0
    what = f"{variant} B={B} T={T} K={K} N={N} G={G} x_layout={x_layout}"
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    if variant == "glu":
        C = N
        lc = synth.linear(B, T, K, 2 * C, seed=80_000 + i, groups=2, bias=bias)
        m, s = orc.linear_constants(lc.s_x, lc.s_w, lc.s_y_per_channel())
        g = orc.glu_params(float(lc.s_y[0]), float(lc.s_y[1]),
                           float(2.0 ** rng.uniform(-1, 1)) * float(lc.s_y[0]))
        want = orc.glu(orc.linear(lc.x, lc.w, lc.bias, m, s), g)
        perm = np.empty(2 * C, np.int64)
        perm[0::2] = np.arange(C)
        perm[1::2] = np.arange(C) + C
        gd = Guarded(want.shape, torch.int8)
        ip.linear_glu_i8(_d(lc.x), _d(_interleave(lc.w)),
                         None if lc.bias is None else _d(lc.bias[perm]), _d(m[perm]), _d(s[perm]),
                         (g.q_c, g.q_one, g.m, g.s), out=gd.view, workspace=ws)
    else:
        lc = synth.linear(B, T, K, N, seed=80_000 + i, groups=G, bias=bias)
        m, s = orc.linear_constants(lc.s_x, lc.s_w, lc.s_y_per_channel())
        x = lc.x
        if x_layout == 1:
            x = np.ascontiguousarray(x.reshape(B, T, K // 128, 128).transpose(0, 2, 1, 3))
        z = orc.linear(x, lc.w, lc.bias, m, s, x_layout=x_layout, y_layout=y_layout, groups=G)
        bd = None if lc.bias is None else _d(lc.bias)
        if variant == "swish":
            s_z = float(lc.s_y[0])
            sw = orc.swish_params(s_z, float(2.0 ** rng.uniform(-1, 1)) * s_z)
            want = orc.swish(z, sw)
            gd = Guarded(want.shape, torch.int8)
            ip.linear_swish_i8(_d(x), _d(lc.w), bd, _d(m), _d(s), (sw.q_c, sw.q_one, sw.m, sw.s),
                               out=gd.view, workspace=ws)
        elif variant == "residual":
            res = rng.integers(-127, 128, size=(B, T, N)).astype(np.int8)
            s_y = float(lc.s_y[0])
            s_r = float(rng.uniform(0.02, 0.08))
            rp = orc.residual_params(s_r, s_y, 1.2 * max(s_r, s_y), float(rng.choice([0.5, 1.0])))
            want = orc.residual(res, z, *rp)
            gd = Guarded(want.shape, torch.int8)
            ip.linear_residual_i8(_d(x), _d(lc.w), bd, _d(m), _d(s), _d(res), *rp, out=gd.view,
                                  workspace=ws)
        else:
            want = z
            gd = Guarded(want.shape, torch.int8)
            ip.linear_i8(_d(x), _d(lc.w), bd, _d(m), _d(s), x_layout=x_layout, y_layout=y_layout,
                         groups=G, out=gd.view, workspace=ws)
    assert ip.status(ws) == 0, what
    gd.check()
    assert_same(gd.view.cpu().numpy(), want, what)


@pytest.mark.parametrize("i", range(8))
def test_random_layernorm(ip, orc, i):
    rng = np.random.default_rng(71_000 + i)
    d = 512 * int(rng.integers(1, 5))
    rows = int(rng.choice([int(rng.integers(1, 40)), int(rng.integers(40, 5000))]))
    x = np.clip(np.rint(rng.normal(rng.normal(0, 20), float(rng.uniform(2, 60)), size=(rows, d))),
                -127, 127).astype(np.int8)
    if rng.integers(0, 3) == 0:
        x[int(rng.integers(0, rows))] = int(rng.integers(-127, 128))   # a constant row
    gamma = rng.uniform(0.2, 2.5, size=d) * rng.choice([-1.0, 1.0], size=d, p=[0.1, 0.9])
    beta = rng.normal(0.0, 0.7, size=d)
    s_x, s_y = rng.uniform(1.0, 8.0) / 127, rng.uniform(2.0, 10.0) / 127
    eps = float(10.0 ** rng.uniform(-6, -3))
    c = orc.layernorm_constants(s_x, gamma, beta, s_y, eps)
    want = orc.layernorm(x, c)
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    g = Guarded(want.shape, torch.int8)
    ip.layernorm_i8(_d(x), _d(c.M), _d(c.B), _d(c.E), c.eps_c, out=g.view, workspace=ws)
    assert ip.status(ws) == 0
    g.check()
    assert_same(g.view.cpu().numpy(), want, f"layernorm rows={rows} d={d}")


@pytest.mark.parametrize("i", range(12))
def test_random_dwconv(ip, orc, i):
    rng = np.random.default_rng(72_000 + i)
    K = int(rng.choice([1, 3, 5, 7, 9, 11, 13, 15]))
    C = int(rng.integers(1, 300)) * (4 if i % 3 else 1) + (0 if i % 3 else int(rng.integers(0, 4)))
    B = int(rng.integers(1, 6))
    T = int(rng.integers(1, 400))
    x = rng.integers(-127, 128, size=(B, T, C)).astype(np.int8)
    w = rng.integers(-127, 128, size=(C, K)).astype(np.int8)
    bias = rng.integers(-(2 ** 20), 2 ** 20, size=C).astype(np.int32)
    m = rng.integers(0, 2 ** 31, size=C).astype(np.int32)
    s = rng.integers(0, 32, size=C).astype(np.int32)
    p16 = orc.swish16_params(float(rng.uniform(5, 80)) / 32767, float(rng.uniform(2, 8)) / 127)
    want = orc.swish16(orc.dwconv(x, w, bias, m, s), p16)
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    g = Guarded(want.shape, torch.int8)
    ip.dwconv_swish_i8(_d(x), _d(w), _d(bias), _d(m), _d(s), (p16.q_c, p16.q_one, p16.m, p16.s),
                       out=g.view, workspace=ws)
    assert ip.status(ws) == 0
    g.check()
    assert_same(g.view.cpu().numpy(), want, f"dwconv B={B} T={T} C={C} K={K}")
