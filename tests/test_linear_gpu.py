"""Parity of the integer linear layer on the GPU (through the C ABI) with the
CPU oracle: bit-exact on every output."""
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


def run_both(ip, orc, x, w, bias, m, s, x_layout=0, y_layout=0, groups=1):
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    want = orc.linear(x, w, bias, m, s, x_layout=x_layout, y_layout=y_layout, groups=groups)
    g = Guarded(want.shape, torch.int8)
    got = ip.linear_i8(_d(x), _d(w), None if bias is None else _d(bias), _d(m), _d(s),
                       x_layout=x_layout, y_layout=y_layout, groups=groups, out=g.view,
                       workspace=ws)
    st = ip.status(ws)
    g.check()
    return got.cpu().numpy(), want, st


def assert_same(got, want):
    bad = got != want
    if bad.any():
        idx = np.argwhere(bad)[:5]
        raise AssertionError(f"{int(bad.sum())} of {got.size} differ; first at {idx.tolist()}: "
                             f"gpu {got[tuple(idx[0])]} oracle {want[tuple(idx[0])]}")


def case(orc, B, T, K, N, seed, groups=1, bias=True):
    c = synth.linear(B, T, K, N, seed=seed, groups=groups, bias=bias)
    m, s = orc.linear_constants(c.s_x, c.s_w, c.s_y_per_channel())
    return c, m, s


@pytest.mark.parametrize("T", [1, 2, 127, 128, 129, 255, 300])
def test_ragged_frames(ip, orc, T):
    c, m, s = case(orc, 2, T, 256, 256, seed=40 + T)
    got, want, st = run_both(ip, orc, c.x, c.w, c.bias, m, s)
    assert st == 0
    assert_same(got, want)


@pytest.mark.parametrize("K,N", [(128, 128), (384, 640), (1024, 1024), (4096, 1024),
                                 (1024, 4096)])
def test_shapes(ip, orc, K, N):
    c, m, s = case(orc, 3, 77, K, N, seed=K + N)
    got, want, st = run_both(ip, orc, c.x, c.w, c.bias, m, s)
    assert st == 0
    assert_same(got, want)


@pytest.mark.parametrize("B,T,G", [(9, 1, 1), (5, 7, 3), (3, 50, 1), (7, 129, 3)])
def test_flat_tiles_across_utterances(ip, orc, B, T, G):
    # a 128-row tile of the flat frame axis spans several utterances
    c, m, s = case(orc, B, T, 256, 128 * G, seed=80 + T, groups=G)
    got, want, st = run_both(ip, orc, c.x, c.w, c.bias, m, s, y_layout=1, groups=G)
    assert st == 0
    assert_same(got, want)
    got, want, st = run_both(ip, orc, c.x, c.w, c.bias, m, s)    # row-major output (G = 1)
    assert st == 0
    assert_same(got, want)


def test_no_bias(ip, orc):
    c, m, s = case(orc, 2, 150, 512, 256, seed=7, bias=False)
    got, want, st = run_both(ip, orc, c.x, c.w, None, m, s)
    assert st == 0
    assert_same(got, want)


@pytest.mark.parametrize("G", [1, 3])
def test_head_split_output(ip, orc, G):
    c, m, s = case(orc, 3, 200, 1024, 384 * G, seed=60 + G, groups=G)
    got, want, st = run_both(ip, orc, c.x, c.w, c.bias, m, s, y_layout=1, groups=G)
    assert st == 0
    assert_same(got, want)


def test_head_split_input(ip, orc):
    c, m, s = case(orc, 2, 131, 1024, 256, seed=71)
    B, T, K = c.x.shape
    xh = np.ascontiguousarray(c.x.reshape(B, T, K // 128, 128).transpose(0, 2, 1, 3))
    got, want, st = run_both(ip, orc, xh, c.w, c.bias, m, s, x_layout=1)
    assert st == 0
    assert_same(got, want)


def test_extreme_values_longest_K(ip, orc):
    # +-128/127 everywhere, the largest K: the int32 accumulator stays exact
    rng = np.random.default_rng(3)
    K, N = 32768, 128
    x = rng.choice(np.array([-128, 127], np.int8), size=(1, 5, K))
    w = rng.choice(np.array([-128, 127], np.int8), size=(N, K))
    bias = rng.integers(-(2 ** 30) + 1, 2 ** 30, size=N).astype(np.int32)
    m = rng.integers(0, 2 ** 31, size=N).astype(np.int32)
    s = rng.integers(0, 32, size=N).astype(np.int32)
    got, want, st = run_both(ip, orc, x, w, bias, m, s)
    assert st == 0
    assert_same(got, want)


def test_constant_out_of_domain_is_reported(ip):
    x = torch.zeros((1, 4, 128), dtype=torch.int8, device="cuda")
    w = torch.zeros((128, 128), dtype=torch.int8, device="cuda")
    m = torch.full((128,), 2 ** 30, dtype=torch.int32, device="cuda")
    s = torch.zeros(128, dtype=torch.int32, device="cuda")
    s[5] = 40
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    ip.linear_i8(x, w, None, m, s, workspace=ws)
    assert ip.status(ws) == -7
    assert ip.status(ws) == 0       # read and cleared


def test_encoder_qkv_projection_full_size(ip, orc):
    # Q, K, V of one encoder layer: B=32, T=375, 1024 -> 3 x 1024, head-split
    c, m, s = case(orc, 32, 375, 1024, 3072, seed=3001, groups=3)
    got, want, st = run_both(ip, orc, c.x, c.w, c.bias, m, s, y_layout=1, groups=3)
    assert st == 0
    assert got.shape == (3, 32, 8, 375, 128)
    assert_same(got, want)


def test_encoder_output_projection_full_size(ip, orc):
    # the heads of the attention output [B, 8, T, 128] -> [B, T, 1024]
    c, m, s = case(orc, 32, 375, 1024, 1024, seed=3002)
    B, T, K = c.x.shape
    xh = np.ascontiguousarray(c.x.reshape(B, T, 8, 128).transpose(0, 2, 1, 3))
    got, want, st = run_both(ip, orc, xh, c.w, c.bias, m, s, x_layout=1)
    assert st == 0
    assert_same(got, want)


def swish_case(orc, B, T, K, N, seed):
    """FFN first projection: z on an int8 grid S_z (the linear layer's output
    grid), then the Swish onto S_y."""
    c = synth.linear(B, T, K, N, seed=seed)
    m, s = orc.linear_constants(c.s_x, c.s_w, c.s_y_per_channel())
    s_z = float(c.s_y[0])
    sw = orc.swish_params(s_z, 0.9 * s_z)
    return c, m, s, sw


def run_swish(ip, orc, c, m, s, sw):
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    z = orc.linear(c.x, c.w, c.bias, m, s)
    g = Guarded(z.shape, torch.int8)
    got = ip.linear_swish_i8(_d(c.x), _d(c.w), None if c.bias is None else _d(c.bias), _d(m),
                             _d(s), (sw.q_c, sw.q_one, sw.m, sw.s), out=g.view, workspace=ws)
    st = ip.status(ws)
    g.check()
    return got.cpu().numpy(), orc.swish(z, sw), st


@pytest.mark.parametrize("B,T,K,N", [(1, 1, 128, 128), (2, 77, 256, 384), (3, 200, 1024, 512)])
def test_linear_swish(ip, orc, B, T, K, N):
    c, m, s, sw = swish_case(orc, B, T, K, N, seed=900 + T)
    got, want, st = run_swish(ip, orc, c, m, s, sw)
    assert st == 0
    assert_same(got, want)


def test_ffn_first_projection_full_size(ip, orc):
    # FFN of one encoder block: B=32, T=375, 1024 -> 4096 with the Swish
    c, m, s, sw = swish_case(orc, 32, 375, 1024, 4096, seed=3003)
    got, want, st = run_swish(ip, orc, c, m, s, sw)
    assert st == 0
    assert_same(got, want)
