"""The pins must catch plausible mistakes in the oracle.

Each case plants one mistake in a copy of the oracle's C source or of its
offline constants (on the CPU, in a temporary directory), rebuilds it there
and runs the fast pins against the copy in a subprocess: every mutant must
make at least one pin fail.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTANTS = {
    # mirrored relative shift (i - j instead of j - i)
    "phi_direction": ("int r = j - i + T - 1;", "int r = i - j + T - 1;"),
    # content branch without the u bias
    "drop_u": ("((int64_t)qi[d] + (int64_t)u[d]) * (int64_t)kj[d]",
               "((int64_t)qi[d]) * (int64_t)kj[d]"),
    # position branch without the v bias
    "drop_v": ("((int64_t)qi[d] + (int64_t)vb[d]) * (int64_t)pr[d]",
               "((int64_t)qi[d]) * (int64_t)pr[d]"),
    # truncation instead of rounding in Eq. 11 / Eq. 7
    "floor_not_round": ("return floor_div_pow2(x + ((int64_t)1 << (n - 1)), n);",
                        "return floor_div_pow2(x, n);"),
    # shift of 2^-n off by one
    "shift_off_by_one": ("return clamp_i8(round_shift(x, 31 + s_s));",
                         "return clamp_i8(round_shift(x, 30 + s_s));"),
    # exponential without the 2^-z factor
    "iexp_no_shift": ("return L >> z; /* L >= 0 */", "return L; /* L >= 0 */"),
    # exponential with the sign of q_b flipped
    "iexp_sign": ("int64_t t = p + sm->q_b;", "int64_t t = p - sm->q_b;"),
    # normaliser with the wrong output grid
    "softmax_grid": ("int64_t y = (e[j] * f) >> 24;", "int64_t y = (e[j] * f) >> 25;"),
    # masked keys still counted in the softmax
    "mask_keys": ("isoftmax_row(srow, len, len, sm, e, a);",
                  "for (int j = len; j < T; ++j) srow[j] = srow[0];\n        isoftmax_row(srow, T, T, sm, e, a);"),
    # transposed operand in A.V
    "av_transpose": ("acc += (int64_t)a[j] * (int64_t)vh[(size_t)j * dh + d];",
                     "acc += (int64_t)a[j] * (int64_t)vh[(size_t)d * dh + j % dh];"),
}

# mistakes planted in the linear-layer oracle (Eqs. 6-7)
LINEAR_MUTANTS = {
    # bias dropped
    "lin_drop_bias": ("int64_t acc = bias ? (int64_t)bias[n] : 0;", "int64_t acc = 0;"),
    # weights read transposed
    "lin_w_transposed": ("acc += xr[k] * (int64_t)wn[k];",
                         "acc += xr[k] * (int64_t)w[(size_t)k * N + n];"),
    # truncation instead of rounding
    "lin_floor": ("lin_floor_pow2((int64_t)m[n] * acc + ((int64_t)1 << (e - 1)), e)",
                  "lin_floor_pow2((int64_t)m[n] * acc, e)"),
    # shift one short
    "lin_shift": ("int e = 31 + s[n];", "int e = 30 + s[n];"),
    # asymmetric clamp (the int8 grid is symmetric, Eq. 6)
    "lin_clamp": ("if (v < -127) v = -127;\n            y[act_index",
                  "if (v < -128) v = -128;\n            y[act_index"),
    # head index of the head-split layout swapped with the frame
    "lin_heads": ("* heads + (size_t)(cc / 128)) * T + t) * 128",
                  "* T + t) * heads + (size_t)(cc / 128)) * 128"),
}

LINEAR_MUTANTS.update({
    # Swish with the sign of tanh dropped (sigma(x) = (1 + |tanh|) / 2)
    "swish_sign": ("int64_t t = (int64_t)p->q_one + sg * L;", "int64_t t = (int64_t)p->q_one + L;"),
    # Swish without the clip at c (the parabola turns back up)
    "swish_clip": ("int64_t dclip = (a < p->q_c ? a : p->q_c) - p->q_c;",
                   "int64_t dclip = a - p->q_c;"),
    # tanh = q_one + D^2 (sign of a lost)
    "swish_a_sign": ("int64_t L = (int64_t)p->q_one - dclip * dclip;",
                     "int64_t L = (int64_t)p->q_one + dclip * dclip;"),
    # x (1 + tanh) without the halving: output shift one short
    "swish_half": ("int e = 31 + p->s;\n    for", "int e = 30 + p->s;\n    for"),
})

LINEAR_PINS = ["tests/test_oracle_linear.py", "tests/test_oracle_swish.py"]

# mistakes planted in the LayerNorm oracle
NORM_MUTANTS = {
    # variance around 0 instead of the mean
    "ln_no_mean": ("int64_t c = (int64_t)d * q[i] - sum;\n            v += c * c;",
                   "int64_t c = (int64_t)d * q[i];\n            v += c * c;"),
    # output without subtracting the mean
    "ln_no_centre": ("int64_t c = (int64_t)d * q[i] - sum;\n            int64_t n",
                     "int64_t c = (int64_t)d * q[i];\n            int64_t n"),
    # mean square not divided by d
    "ln_var_div": ("ipo_isqrt(v / d + eps_c)", "ipo_isqrt(v / (d / 2) + eps_c)"),
    # epsilon dropped
    "ln_eps": ("ipo_isqrt(v / d + eps_c)", "ipo_isqrt(v / d)"),
    # square root one too large
    "ln_isqrt": ("if (next >= r) return r;", "if (next >= r) return r + 1;"),
    # reciprocal on the wrong grid
    "ln_recip": ("int64_t f = ((int64_t)1 << 31) / sigma;", "int64_t f = ((int64_t)1 << 30) / sigma;"),
}

NORM_PINS = ["tests/test_oracle_norm.py"]

# mistakes planted in the block oracle (residual, GLU, depthwise conv, INT16 Swish)
BLOCK_MUTANTS = {
    "res_drop_y": ("int64_t v = (int64_t)m_x * x[i] + (int64_t)m_y * y[i];",
                   "int64_t v = (int64_t)m_x * x[i];"),
    "glu_swap": ("int64_t a = ab[(size_t)r * 2 * C + c];\n            int64_t b = ab[(size_t)r * 2 * C + C + c];",
                 "int64_t b = ab[(size_t)r * 2 * C + c];\n            int64_t a = ab[(size_t)r * 2 * C + C + c];"),
    "glu_sign": ("int64_t t = (int64_t)p->q_one + sg * L;                   /* 1 + tanh */",
                 "int64_t t = (int64_t)p->q_one - sg * L;                   /* 1 + tanh */"),
    "dw_wrap": ("if (tt < 0 || tt >= T) continue;               /* zero padding */",
                "tt = (tt + T) % T;"),
    "dw_flip": ("acc += (int64_t)w[(size_t)c * K + k] * x",
                "acc += (int64_t)w[(size_t)c * K + (K - 1 - k)] * x"),
    "dw_no_bias": ("int64_t acc = bias[c];", "int64_t acc = 0;"),
    "sw16_clip": ("int64_t dclip = (mag < p->q_c ? mag : p->q_c) - p->q_c;\n        int64_t L = p->q_one",
                  "int64_t dclip = mag - p->q_c;\n        int64_t L = p->q_one"),
    "sw16_overflow": ("__int128 v = (__int128)p->m * (__int128)(q * t)",
                      "__int128 v = (__int128)(int64_t)((uint64_t)p->m * (uint64_t)(q * t))"),
}

BLOCK_PINS = ["tests/test_oracle_block.py"]

# mistakes in the offline softmax constants that show only on coarse score
# grids (q_ln2 = 7..9, where one grid step is a large share of ln2 and b):
# rounding instead of the floors of I-BERT's constants
CONST_MUTANTS = {
    "qb_round": ("q_b = math.floor(IBERT_B / S)", "q_b = math.floor(IBERT_B / S + 0.5)"),
    "qc_round": ("q_c = math.floor(IBERT_C / (IBERT_A * (S * S)))",
                 "q_c = math.floor(IBERT_C / (IBERT_A * (S * S)) + 0.5)"),
    "qln2_round": ("q_ln2 = math.floor(LN2 / S)", "q_ln2 = math.floor(LN2 / S + 0.5)"),
}

CONST_PINS = [
    "tests/test_oracle_softmax.py::test_iexp_within_derived_bounds",
    "tests/test_oracle_softmax.py::test_softmax_two_keys_coarse",
    "tests/test_oracle_layer.py::test_encoder_layer_coarse_grid",
]

PINS = [
    "tests/test_oracle_relshift.py",
    "tests/test_oracle_scores.py",
    "tests/test_oracle_softmax.py::test_iexp_within_derived_bounds",
    "tests/test_oracle_softmax.py::test_iexp_halving_identity",
    "tests/test_oracle_softmax.py::test_softmax_uniform_closed_form",
    "tests/test_oracle_softmax.py::test_softmax_single_key_is_255",
    "tests/test_oracle_layer.py::test_layer_vs_float64_attention",
    "tests/test_oracle_layer.py::test_masked_layer_equals_truncated_problem",
    "tests/test_oracle_layer.py::test_single_frame_closed_form",
]


def _copy_tree(dst):
    for name in ("oracle", "synth", "tests"):
        shutil.copytree(os.path.join(ROOT, name), os.path.join(dst, name),
                        ignore=shutil.ignore_patterns("*.so", "__pycache__", "*.tmp*"))


GROUPS = [(MUTANTS, PINS, "ipo_mhsa.c"), (LINEAR_MUTANTS, LINEAR_PINS, "ipo_linear.c"),
          (NORM_MUTANTS, NORM_PINS, "ipo_norm.c"), (BLOCK_MUTANTS, BLOCK_PINS, "ipo_block.c"),
          (CONST_MUTANTS, CONST_PINS, "consts.py")]


@pytest.mark.slow
@pytest.mark.parametrize("name", [n for g in GROUPS for n in sorted(g[0])])
def test_mutant_is_caught(tmp_path, name):
    table, pins, fname = next(g for g in GROUPS if name in g[0])
    old, new = table[name]
    _copy_tree(tmp_path)
    src = tmp_path / "oracle" / fname
    text = src.read_text()
    assert text.count(old) == 1, f"mutation site for {name} not found"
    src.write_text(text.replace(old, new))
    env = dict(os.environ, PYTHONPATH=str(tmp_path))
    res = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                          "-m", "not gpu and not slow"] + pins,
                         cwd=tmp_path, env=env, capture_output=True, text=True, timeout=600)
    assert res.returncode != 0, f"mutant {name} survived the pins:\n{res.stdout[-2000:]}"
    assert "failed" in res.stdout or "error" in res.stdout.lower()
