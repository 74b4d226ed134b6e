"""Parity of the integer LayerNorm on the GPU (through the C ABI) with the
CPU oracle: bit-exact on every output."""
import numpy as np
import pytest

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


def case(rows, d, seed, eps=1e-5, spread=35.0):
    rng = np.random.default_rng(seed)
    x = np.clip(np.rint(rng.normal(rng.normal(0, 10), spread, size=(rows, d))), -127, 127).astype(np.int8)
    gamma = rng.uniform(0.3, 2.0, size=d) * rng.choice([-1.0, 1.0], size=d, p=[0.1, 0.9])
    beta = rng.normal(0.0, 0.5, size=d)
    s_x, s_y = rng.uniform(2.0, 6.0) / 127, rng.uniform(3.0, 8.0) / 127
    return x, gamma, beta, s_x, s_y, eps


def run_both(ip, orc, x, gamma, beta, s_x, s_y, eps):
    c = orc.layernorm_constants(s_x, gamma, beta, s_y, eps)
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    got = ip.layernorm_i8(_d(x), _d(c.M), _d(c.B), _d(c.E), c.eps_c, workspace=ws)
    assert ip.status(ws) == 0
    return got.cpu().numpy(), orc.layernorm(x, c)


def assert_same(got, want):
    bad = got != want
    if bad.any():
        idx = np.argwhere(bad)[:5]
        raise AssertionError(f"{int(bad.sum())} of {got.size} differ; first at {idx.tolist()}: "
                             f"gpu {got[tuple(idx[0])]} oracle {want[tuple(idx[0])]}")


@pytest.mark.parametrize("d", [512, 1024, 1536, 2048])
@pytest.mark.parametrize("rows", [1, 7, 300])
def test_shapes(ip, orc, d, rows):
    assert_same(*run_both(ip, orc, *case(rows, d, seed=d + rows)))


def test_special_rows(ip, orc):
    d = 1024
    x, gamma, beta, s_x, s_y, _ = case(8, d, seed=5)
    x[0] = 0                                   # constant rows: sigma from epsilon only
    x[1] = -127
    x[2] = np.where(np.arange(d) % 2 == 0, 127, -127)
    x[3] = np.where(np.arange(d) == 0, 127, -127)   # one outlier
    x[4] = np.where(np.arange(d) % 2 == 0, 1, 0)
    for eps in (0.0, 1e-5, 1e-2):
        assert_same(*run_both(ip, orc, x, gamma, beta, s_x, s_y, eps))


def test_sigma_and_reciprocal_over_their_range(ip, orc):
    # sigma = isqrt(floor(sum c^2 / d) + eps_c) and f = floor(2^31 / sigma)
    # are Newton iterations in the kernel: rows with one to three nonzero
    # values (and constant rows) give floor(sum c^2 / d) = d sum q^2 -
    # (sum q)^2 over a wide spread, and eps_c from 0 to 2^40 (powers of two
    # and their neighbours, where the normalisation changes) moves sigma
    # from 1 to 2^20; every output against the oracle
    d, rows = 512, 2048
    rng = np.random.default_rng(12)
    x = np.zeros((rows, d), np.int8)
    for r in range(rows):
        k = int(rng.integers(0, 4))
        x[r, rng.choice(d, size=k, replace=False)] = rng.integers(-127, 128, size=k)
    x[::97] = rng.integers(-127, 128)
    _, gamma, beta, s_x, s_y, _ = case(1, d, seed=13)
    c = orc.layernorm_constants(s_x, gamma, beta, s_y, 1e-5)
    eps_values = [0, 1, 2, 3, 5, 2 ** 40]
    for k in range(2, 40, 3):
        eps_values += [2 ** k - 1, 2 ** k, 2 ** k + 1]
    eps_values += [int(v) for v in rng.integers(0, 2 ** 40, size=6)]
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    xd = _d(x)
    Md, Bd, Ed = _d(c.M), _d(c.B), _d(c.E)
    for eps_c in eps_values:
        got = ip.layernorm_i8(xd, Md, Bd, Ed, eps_c, workspace=ws)
        assert ip.status(ws) == 0
        want = orc.layernorm(x, orc.NormConstants(M=c.M, B=c.B, E=c.E, eps_c=eps_c))
        assert_same(got.cpu().numpy(), want)


def test_small_variance_rows(ip, orc):
    assert_same(*run_both(ip, orc, *case(64, 1024, seed=6, eps=2e-4, spread=0.6)))


def test_encoder_frames_full_size(ip, orc):
    # the LayerNorm before the attention of one block: B=32 x T=375 frames
    assert_same(*run_both(ip, orc, *case(32 * 375, 1024, seed=7)))


@pytest.mark.parametrize("mode", ["E31", "E32", "E62"])
def test_requant_shift_paths(ip, orc, mode):
    # The kernel shifts the high word of M n + B' when every E >= 32 (the
    # usual constants have E in the high 30s and 40s) and takes
    # floor(v / 2^31) first when some channel has E = 31.  Constants of
    # both kinds, at the ends of the domain, against the oracle with the
    # same constants.
    x, gamma, beta, s_x, s_y, eps = case(300, 1024, seed=11)
    c = orc.layernorm_constants(s_x, gamma, beta, s_y, eps)
    M, B, E = c.M.copy(), c.B.copy(), c.E.copy()
    ch = np.arange(0, 1024, 61)
    if mode == "E31":
        sh = E[ch] - 31
        M[ch] >>= sh
        B[ch] >>= sh
        E[ch] = 31
    elif mode == "E32":
        sh = E - 32
        M >>= sh
        B >>= sh
        E[:] = 32
    else:
        E[ch] = 62
        B[ch] = 0
    c2 = orc.NormConstants(M=M, B=B, E=E, eps_c=c.eps_c)
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    got = ip.layernorm_i8(_d(x), _d(M), _d(B), _d(E), c.eps_c, workspace=ws)
    assert ip.status(ws) == 0
    assert_same(got.cpu().numpy(), orc.layernorm(x, c2))


def test_constant_out_of_domain_is_reported(ip, orc):
    x, gamma, beta, s_x, s_y, eps = case(4, 512, seed=8)
    c = orc.layernorm_constants(s_x, gamma, beta, s_y, eps)
    E = c.E.copy()
    E[3] = 70
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    ip.layernorm_i8(_d(x), _d(c.M), _d(c.B), _d(E), c.eps_c, workspace=ws)
    assert ip.status(ws) == -7
