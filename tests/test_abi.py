"""Host-side checks of the C ABI (no GPU needed): the library builds, loads
and exports every function include/ip_mhsa.h declares; argument validation
returns the documented codes before any device work; the offline constant
helpers agree bit for bit with the oracle's; the kernel source carries no
floating-point type."""
import ctypes
import math
import os
import re

import numpy as np
import pytest

import paper_2609_30846_gb300 as ip

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "ip_mhsa.h")
CSRC = os.path.join(ROOT, "paper_2609_30846_gb300", "csrc")
KERNELS = os.path.join(CSRC, "ip_mhsa_kernels.cuh")
DEVICE_SOURCES = [os.path.join(CSRC, f) for f in
                  ("ip_mhsa_kernels.cuh", "ip_linear_kernels.cuh", "ip_norm_kernels.cuh",
                   "ip_ptx.cuh")]


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ip_[a-z0-9_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    return ip.load()


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert len(names) >= 10
    for n in names:
        assert hasattr(lib, n), f"{n} declared in include/ip_mhsa.h but not exported"
    assert set(names) == set(ip.EXPORTS)


def test_strerror_texts(lib):
    for code in range(-8, 1):
        assert ip.strerror(code)
    assert "unknown" in ip.strerror(-99)


def test_workspace_bytes(lib):
    assert ip.workspace_bytes(1, 8, 64) == 256   # the device status word
    for bad in [(1, 8, 0), (1, 8, ip.IP_MAX_T + 1), (-1, 8, 10)]:
        assert lib.ip_relpos_mhsa_workspace_bytes(*bad, 128) == 0
    assert lib.ip_relpos_mhsa_workspace_bytes(1, 8, 64, 64) == 0


def _call(lib, **over):
    buf = (ctypes.c_byte * 4096)()
    base = (ctypes.addressof(buf) + 255) // 256 * 256
    a = dict(q=base, k=base, v=base, p=base, u=base, vb=base,
             mult=(ctypes.c_int32 * 3)(2 ** 30, 2 ** 30, 2 ** 30),
             shifts=(ctypes.c_int32 * 2)(9, 8), sm=ip.SoftmaxParams(12, 24, 327),
             lens=None, B=1, H=1, T=4, dh=128, out=base, ws=base, wsb=1 << 20)
    a.update(over)
    return lib.ip_relpos_mhsa_i8(a["q"], a["k"], a["v"], a["p"], a["u"], a["vb"], a["mult"],
                                 a["shifts"], ctypes.byref(a["sm"]) if a["sm"] is not None else None,
                                 a["lens"], a["B"], a["H"], a["T"], a["dh"], a["out"], a["ws"],
                                 a["wsb"], None)


def test_validation_codes(lib):
    assert _call(lib, q=None) == -1
    assert _call(lib, sm=None) == -1
    assert _call(lib, ws=None) == -1
    assert _call(lib, T=0) == -2
    assert _call(lib, T=ip.IP_MAX_T + 1) == -2
    assert _call(lib, B=-1) == -2
    assert _call(lib, dh=64) == -4
    assert _call(lib, k=None) == -1
    assert _call(lib, B=70000) == -2
    buf = (ctypes.c_byte * 64)()
    odd = (ctypes.addressof(buf) + 15) // 16 * 16 + 8
    assert _call(lib, v=odd) == -3
    assert _call(lib, mult=(ctypes.c_int32 * 3)(-1, 0, 0)) == -7
    assert _call(lib, shifts=(ctypes.c_int32 * 2)(32, 8)) == -7
    assert _call(lib, shifts=(ctypes.c_int32 * 2)(9, -1)) == -7
    assert _call(lib, sm=ip.SoftmaxParams(0, 24, 327)) == -7      # q_ln2 < 1
    assert _call(lib, sm=ip.SoftmaxParams(5, 0, 1)) == -7         # L(0) = 1 < 2
    assert _call(lib, sm=ip.SoftmaxParams(5, 46341, 0)) == -7     # L(0) >= 2^31
    assert _call(lib, wsb=16) == -8
    # B = 0 or H = 0 is a valid empty problem: nothing is read or launched
    assert _call(lib, B=0) == 0
    assert _call(lib, B=0, q=None, out=None) == 0
    assert _call(lib, H=0, ws=None) == 0


def test_default_workspace_registration(lib):
    # ip_set_workspace validates without touching the device; a call that
    # passes no workspace takes the registered one (it then fails only on
    # the bad multiplier below, past every pointer check) and, with none
    # registered, reports the missing pointer.
    buf = (ctypes.c_byte * 1024)()
    base = (ctypes.addressof(buf) + 255) // 256 * 256
    bad_mult = (ctypes.c_int32 * 3)(-1, 0, 0)
    try:
        assert lib.ip_set_workspace(base + 16, 512) == -3
        assert lib.ip_set_workspace(base, 16) == -8
        assert _call(lib, ws=None, mult=bad_mult) == -1
        assert lib.ip_relpos_mhsa_status(None, None) == -1
        assert lib.ip_set_workspace(base, 512) == 0
        assert _call(lib, ws=None, mult=bad_mult) == -7
        assert _call(lib, ws=None, sm=None) == -1
        # an explicit workspace still wins over the registered one
        assert _call(lib, ws=base + 16, mult=bad_mult) == -3
    finally:
        assert lib.ip_set_workspace(None, 0) == 0
    assert _call(lib, ws=None, mult=bad_mult) == -1


def test_constants_match_oracle(lib):
    import oracle
    rng = np.random.default_rng(0)
    ratios = np.concatenate([10.0 ** rng.uniform(-18, -0.31, 400), [2.0 ** -9, 0.25, 0.49999]])
    for r in ratios:
        assert ip.dyadic_multiplier(float(r)) == oracle.dyadic(float(r)), r
    for _ in range(200):
        r_c, r_p = 10.0 ** rng.uniform(-6, -1, 2)
        assert ip.dyadic_pair(float(r_c), float(r_p)) == oracle.dyadic_pair(float(r_c), float(r_p))
    for S in 10.0 ** rng.uniform(-3.5, 0, 300):
        assert ip.isoftmax_params_from_scale(float(S)) == oracle.isoftmax_params(float(S)), S
    import synth
    for w in range(5):
        sc = synth.layer(w, 0).scales if w != 3 else synth.draw(1, 8, 375, 128, 3000, p_mode="sinusoid").scales
        c1 = ip.layer_constants(sc)
        c2 = oracle.layer_constants(sc, 128)
        assert (c1.multipliers, c1.shifts, c1.softmax) == (c2.multipliers, c2.shifts, c2.softmax)


def test_layer_constants_entry_point_matches_oracle(lib):
    # ip_relpos_layer_constants composes Eq. 11's and Eq. 7's ratios itself;
    # on random scales it agrees with the oracle's float64 composition, and
    # both refuse the same unencodable ones.
    import oracle
    rng = np.random.default_rng(11)
    agree = 0
    for _ in range(400):
        sc = dict(zip(("S_Q", "S_K", "S_P", "S_V", "S_s", "S_O"), 10.0 ** rng.uniform(-3, 0.3, 6)))
        dh = int(rng.choice([16, 64, 128]))
        try:
            want = oracle.layer_constants(sc, dh)
        except ValueError:
            want = None
        if want is None:
            with pytest.raises(ip.IpError):
                ip.layer_constants(sc, dh)
            continue
        got = ip.layer_constants(sc, dh)
        assert (got.multipliers, got.shifts, got.softmax) == \
            (want.multipliers, want.shifts, want.softmax), sc
        agree += 1
    assert agree > 100


def test_layer_constants_entry_point_errors(lib):
    m = (ctypes.c_int32 * 3)(7, 7, 7)
    sh = (ctypes.c_int32 * 2)(7, 7)
    sm = ip.SoftmaxParams(7, 7, 7)
    f = lib.ip_relpos_layer_constants
    assert f(0.01, 0.01, 0.01, 0.01, 0.1, 0.02, 128, None, sh, ctypes.byref(sm)) == -1
    for bad in ((0.0, 0.01, 0.01, 0.01, 0.1, 0.02, 128), (0.01, 0.01, 0.01, 0.01, -0.1, 0.02, 128),
                (0.01, 0.01, 0.01, float("inf"), 0.1, 0.02, 128), (0.01, 0.01, 0.01, 0.01, 0.1, 0.02, 0),
                (4.0, 4.0, 4.0, 0.01, 0.1, 0.02, 128)):   # the last: r_c >= 1/2, unencodable
        assert f(*bad, m, sh, ctypes.byref(sm)) == -7, bad
    assert tuple(m) == (7, 7, 7) and tuple(sh) == (7, 7) and sm.q_ln2 == 7   # untouched


def test_linear_constants_entry_point_matches_oracle(lib):
    import oracle
    rng = np.random.default_rng(12)
    for n in (1, 5, 64, 1000):
        s_x = float(10.0 ** rng.uniform(-3, -1))
        s_w = 10.0 ** rng.uniform(-4, -1, n)
        for s_y in (10.0 ** rng.uniform(-3, -1, n), float(10.0 ** rng.uniform(-2, -1))):
            got = ip.linear_constants(s_x, s_w, s_y)
            want = oracle.linear_constants(s_x, s_w, s_y)
            np.testing.assert_array_equal(got[0], want[0])
            np.testing.assert_array_equal(got[1], want[1])
    with pytest.raises(ip.IpError):
        ip.linear_constants(0.01, np.array([1e-3, -1e-3]), 0.01)
    with pytest.raises(ip.IpError):
        ip.linear_constants(0.01, np.array([], dtype=np.float64), 0.01)
    with pytest.raises(ip.IpError):
        ip.linear_constants(1.0, np.array([1.0]), 0.5)          # ratio 2, unencodable


def test_linear_residual_rejects_partial_overlap(lib):
    # res overlapping y other than exactly (in place) is refused before any
    # device work (the fake addresses are never dereferenced)
    P = ctypes.c_void_p
    fake = P(1 << 20)
    y = P(1 << 24)
    ws = P(1 << 21)

    def call(res):
        return lib.ip_linear_residual_i8(fake, fake, None, fake, fake, res, 1 << 30, 1 << 30, 0,
                                         1, 4, 256, 256, y, ws, 256, None)
    assert call(P((1 << 24) + 16)) == -7
    assert call(P((1 << 24) - 512)) == -7           # ends inside y
    assert call(P((1 << 24) + 512)) == -7           # starts inside y


def test_binding_holds_no_scale_arithmetic():
    # the binding marshals the scales to the C helpers; the ratios of Eq. 7
    # and Eq. 11 are composed behind the C ABI
    src = open(os.path.join(ROOT, "paper_2609_30846_gb300", "__init__.py")).read()
    for fn in ("def layer_constants", "def linear_constants"):
        start = src.index(fn)
        body = src[start:src.index("\ndef ", start + 1)]
        for pat in (r"sqrt", r"\* 256", r"/ \(", r"dyadic_multiplier\(", r"\bfor\s+\w+\s+in\b"):
            assert not re.search(pat, body), (fn, pat)


def test_constants_reject_bad_ratios(lib):
    with pytest.raises(ip.IpError):
        ip.dyadic_multiplier(1.0)
    with pytest.raises(ip.IpError):
        ip.dyadic_multiplier(-1e-3)
    with pytest.raises(ip.IpError):
        ip.isoftmax_params_from_scale(0.0)


@pytest.mark.parametrize("path", DEVICE_SOURCES, ids=os.path.basename)
def test_kernel_source_is_integer_only(path):
    text = open(path).read()
    code = re.sub(r"//[^\n]*", "", re.sub(r"/\*.*?\*/", "", text, flags=re.S))
    code = re.sub(r'"(\\.|[^"\\])*"', '""', code)          # drop string literals (PTX)
    for pat in (r"\bfloat\b", r"\bdouble\b", r"\b__half\b", r"\b__nv_bfloat16\b", r"\bhalf\b",
                r"__fdividef|__expf|\bexpf\b|\bexp\b\s*\(", r"\bsqrtf?\b", r"kind::f16|kind::tf32"):
        assert not re.search(pat, code), pat
    # No '/' or '%' by a run-time value: the compiler's integer division
    # would not be integer-only.  Divisions are the long-division helpers;
    # the remaining operators divide by compile-time powers of two.
    if path == KERNELS:
        assert "div_2pow32" in code and "iexp_neg" in code
    allowed = {"NSTAGE", "NK", "MROWS", "DH", "BK", "BM", "BN", "STAGES", "D", "NB",
               "16", "2", "4", "8", "32", "256"}
    for m in re.finditer(r"[^/*](/|%)\s*\(?\s*([A-Za-z_0-9]+)", code):
        if m.group(0).startswith("<") or m.group(1) == "/" and code[m.start(1) + 1] in "/*":
            continue
        tok = m.group(2)
        if tok.isdigit() and int(tok) & (int(tok) - 1) == 0:
            continue   # a literal power of two
        assert tok in allowed, f"run-time division by {tok!r}"


def test_linear_validation_codes(lib):
    P = ctypes.c_void_p
    fake = P(1 << 20)           # never dereferenced: every case fails validation first
    ws = P(1 << 21)

    def call(x_layout=0, y_layout=0, B=1, T=4, K=256, N=256, G=1, x=fake, w=fake, y=fake,
             m=fake, s=fake, bias=None, wsb=256, wsp=ws):
        return lib.ip_linear_i8(x, x_layout, w, bias, m, s, B, T, K, N, G, y, y_layout, wsp,
                                wsb, None)

    assert call(x_layout=2) == -7
    assert call(y_layout=-1) == -7
    assert call(K=200) == -2                     # not a multiple of 128
    assert call(K=65536) == -2                   # above IP_LINEAR_MAX_K
    assert call(N=64) == -2
    assert call(T=0) == -2
    assert call(y_layout=1, N=256, G=3) == -2    # N not a multiple of 128 G
    assert call(y_layout=0, G=2) == -2
    assert call(B=0, x=None, w=None, y=None) == 0   # empty batch: nothing touched
    assert call(w=None) == -1
    assert call(x=P((1 << 20) + 8)) == -3        # 16-byte alignment
    assert call(wsp=P((1 << 21) + 64)) == -3     # workspace 256-byte alignment
    assert call(wsb=128) == -8


def test_exact_division_constant():
    # udiv_magic: floor(n * (floor(2^64 / d) + 1) / 2^64) == floor(n / d) for
    # 0 <= n < 2^32, 2 <= d < 2^32 (d = 1 uses the constant 0 and returns n)
    rng = np.random.default_rng(0)
    ds = [2, 3, 5, 7, 24, 96, 375, 1500, 2 ** 16 + 1, 2 ** 31 - 1, 2 ** 32 - 1]
    ds += [int(v) for v in rng.integers(2, 2 ** 32, size=40)]
    for d in ds:
        M = (1 << 64) // d + 1
        ns = [0, 1, d - 1, d, d + 1, 2 * d - 1, 2 ** 32 - 1, (2 ** 32 - 1) // d * d,
              (2 ** 32 - 1) // d * d - 1]
        ns += [int(v) for v in rng.integers(0, 2 ** 32, size=200)]
        for n in ns:
            if 0 <= n < 2 ** 32:
                assert (n * M) >> 64 == n // d, (n, d)


@pytest.mark.parametrize("s_z,s_y", [(8 / 127, 8 / 127), (6 / 127, 7 / 127), (0.2, 0.05),
                                     (3e-3, 2e-3)])
def test_swish_constants_match_oracle(lib, s_z, s_y):
    import oracle
    want = oracle.swish_params(s_z, s_y)
    assert ip.swish_params_from_scales(s_z, s_y) == (want.q_c, want.q_one, want.m, want.s)


def test_swish_validation(lib):
    with pytest.raises(ip.IpError):
        ip.swish_params_from_scales(0.0, 0.1)
    with pytest.raises(ip.IpError):
        ip.swish_params_from_scales(1e-6, 0.1)      # q_one beyond 2^23
    P = ctypes.c_void_p
    fake = P(1 << 20)
    bad = ip.SwishParams(20, 100, 2 ** 30, 0)          # q_one < q_c^2
    assert lib.ip_linear_swish_i8(fake, fake, None, fake, fake, ctypes.byref(bad), 1, 4, 128, 128,
                                  fake, P(1 << 21), 256, None) == -7
    assert lib.ip_linear_swish_i8(fake, fake, None, fake, fake, None, 1, 4, 128, 128,
                                  fake, P(1 << 21), 256, None) == -1


@pytest.mark.parametrize("seed", [0, 1])
def test_layernorm_constants_match_oracle(lib, seed):
    import oracle
    rng = np.random.default_rng(seed)
    d = 1024
    gamma = rng.uniform(0.2, 2.0, d) * rng.choice([-1.0, 1.0], d)
    gamma[5] = 0.0
    beta = rng.normal(0, 0.5, d)
    s_x, s_y = rng.uniform(2, 6) / 127, rng.uniform(3, 8) / 127
    want = oracle.layernorm_constants(s_x, gamma, beta, s_y, 1e-5)
    got = ip.layernorm_constants(s_x, gamma, beta, s_y, 1e-5)
    assert got.eps_c == want.eps_c
    np.testing.assert_array_equal(got.M, want.M)
    np.testing.assert_array_equal(got.B, want.B)
    np.testing.assert_array_equal(got.E, want.E)


def test_layernorm_validation(lib):
    P = ctypes.c_void_p
    fake, ws = P(1 << 20), P(1 << 21)

    def call(rows=4, d=1024, eps=0, x=fake, M=fake, B=fake, E=fake, y=fake, wsp=ws, wsb=256):
        return lib.ip_layernorm_i8(x, rows, d, eps, M, B, E, y, wsp, wsb, None)

    assert call(d=80) == -4
    assert call(rows=-1) == -2
    assert call(eps=-1) == -7
    assert call(rows=0, x=None, y=None) == 0
    assert call(M=None) == -1
    assert call(B=P((1 << 20) + 4)) == -3
    assert call(wsb=16) == -8


def test_block_constants_match_oracle(lib):
    import oracle
    for args in [(0.05, 0.04, 0.06, 0.5), (0.03, 0.03, 0.04, 1.0)]:
        assert ip.residual_params(*args) == oracle.residual_params(*args)
    for args in [(0.05, 0.06, 0.03), (0.02, 0.08, 0.01)]:
        want = oracle.glu_params(*args)
        assert ip.glu_params(*args) == (want.q_c, want.q_one, want.m, want.s)
    for args in [(8 / 32767, 8 / 127), (20 / 32767, 5 / 127)]:
        want = oracle.swish16_params(*args)
        assert ip.swish16_params(*args) == (want.q_c, want.q_one, want.m, want.s)
    with pytest.raises(ip.IpError):
        ip.swish16_params(3 / 32767, 3 / 127)


def test_block_validation(lib):
    P = ctypes.c_void_p
    fake, ws = P(1 << 20), P(1 << 21)
    assert lib.ip_residual_i8(fake, fake, -1, 1, 1, 0, fake, None) == -2
    assert lib.ip_residual_i8(fake, fake, 16, -1, 1, 0, fake, None) == -7
    assert lib.ip_residual_i8(fake, fake, 16, 1, 1, 32, fake, None) == -7
    assert lib.ip_residual_i8(None, None, 0, 1, 1, 0, None, None) == 0
    assert lib.ip_residual_i8(P((1 << 20) + 8), fake, 16, 1, 1, 0, fake, None) == -3
    sw = ip.Swish16Params(100, 20000, 2 ** 30, 3)
    assert lib.ip_dwconv_swish_i8(fake, 1, 8, 64, fake, 8, fake, fake, fake, ctypes.byref(sw),
                                  fake, ws, 256, None) == -2      # even kernel
    bad = ip.Swish16Params(200, 20000, 2 ** 30, 3)               # q_one < q_c^2
    assert lib.ip_dwconv_swish_i8(fake, 1, 8, 64, fake, 9, fake, fake, fake, ctypes.byref(bad),
                                  fake, ws, 256, None) == -7
