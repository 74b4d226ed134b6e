"""CPU oracle of one integer Conformer block (Sec. 2.1 Eqs. 1-5), composed
from the oracle's integer operations, with every integer constant derived
here from the declared grids.

TEST INFRASTRUCTURE ONLY (see the package docstring).

  Z1 = X  + 1/2 FFN1(LN1(X))          FFN = W2 Swish(W1 x)     (Eq. 1)
  Z2 = Z1 + MHSA(LN2(Z1))             rel-pos MHSA, Sec. 3.1   (Eq. 2)
  Z3 = Z2 + Conv(LN3(Z2))             PW2 Swish(BN(DW(GLU(PW1)))) (Eqs. 3, 5)
  H  = LN5(Z3 + 1/2 FFN2(LN4(Z3)))                             (Eq. 4)
"""
from __future__ import annotations

import numpy as np

from . import (HEADS, dwconv, glu, layernorm, linear, relpos_mhsa, residual, swish, swish16)
from .consts import (glu_params, layer_constants, layernorm_constants, linear_constants,
                     residual_params, swish16_params, swish_params)


def conformer_block(case, trace: dict | None = None) -> np.ndarray:
    """int8 output [B, T, D] of the block for the int8 input case.x; with
    `trace`, also the integer intermediates by name."""
    S = case.s
    B, T, D = case.x.shape
    keep = (lambda name, v: trace.__setitem__(name, v)) if trace is not None else (lambda n, v: None)

    def ln(name, x):
        q = case.ln[name]
        return layernorm(x, layernorm_constants(q.s_in, q.gamma, q.beta, q.s_out, q.eps))

    def lin(name, x, **kw):
        L = case.lin[name]
        m, s = linear_constants(L.s_in, L.s_w, L.s_out)
        return linear(x, L.w, L.bias, m, s, **kw)

    def ffn(pre, x, z_grid, h_grid):
        z = lin(pre + "a", x)
        keep(z_grid, z)
        h = swish(z, swish_params(S[z_grid], S[h_grid]))
        keep(h_grid, h)
        f = lin(pre + "b", h)
        keep(pre + "o", f)
        return f

    # Eq. 1
    a = ln("ln1", case.x)
    keep("ln1", a)
    f = ffn("ff1", a, "ff1z", "ff1h")
    z1 = residual(case.x, f, *residual_params(S["x"], S["ff1o"], S["z1"], 0.5))
    keep("z1", z1)
    # Eq. 2
    a = ln("ln2", z1)
    keep("ln2", a)
    qkv = lin("qkv", a, y_layout=HEADS, groups=3)
    keep("q", qkv[0]), keep("k", qkv[1]), keep("v", qkv[2])
    o = relpos_mhsa(qkv[0], qkv[1], qkv[2], case.p, case.u, case.vb,
                    layer_constants(case.attn_scales, qkv.shape[-1]))
    keep("o", o)
    o_rows = np.ascontiguousarray(o.transpose(0, 2, 1, 3)).reshape(B, T, D)
    mo = lin("out", o_rows)
    keep("mhsa", mo)
    z2 = residual(z1, mo, *residual_params(S["z1"], S["mhsa"], S["z2"], 1.0))
    keep("z2", z2)
    # Eqs. 3, 5
    a = ln("ln3", z2)
    keep("ln3", a)
    ab = lin("pw1", a)
    keep("pw1a", ab[..., :D]), keep("pw1b", ab[..., D:])
    g = glu(ab, glu_params(S["pw1a"], S["pw1b"], S["glu"]))
    keep("glu", g)
    m, s = linear_constants(S["glu"], case.dw_sw, np.full(D, S["bn"]))
    bn = dwconv(g, case.dw_w, case.dw_bias, m, s)
    keep("bn", bn)
    sw = swish16(bn, swish16_params(S["bn"], S["convsw"]))
    keep("convsw", sw)
    c = lin("pw2", sw)
    keep("conv", c)
    z3 = residual(z2, c, *residual_params(S["z2"], S["conv"], S["z3"], 1.0))
    keep("z3", z3)
    # Eq. 4
    a = ln("ln4", z3)
    keep("ln4", a)
    f = ffn("ff2", a, "ff2z", "ff2h")
    z4 = residual(z3, f, *residual_params(S["z3"], S["ff2o"], S["z4"], 0.5))
    keep("z4", z4)
    out = ln("ln5", z4)
    keep("out", out)
    return out
