"""Seeded synthetic Conformer block (Sec. 2.1, Eqs. 1-5) for the integer block
path: random real-valued weights of a Parakeet-CTC-0.6B-shaped block (d =
1024, 8 heads of 128, feed-forward 4096, depthwise kernel 9), quantised the
way Sec. 2.2 describes (Eq. 6: weights per output channel, activations per
tensor with min-max ranges), and calibrated offline by a float64 forward of
the real-valued block on the first utterances.  This module holds no
integer arithmetic of the method: only the real-valued model used for
calibration and the quantisation of the parameters.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

from . import sinusoid_relpos

D = 1024
H = 8
DH = 128
FF = 4096
KDW = 9


@dataclass
class QLinear:
    w: np.ndarray            # int8 [N, K]
    bias: np.ndarray | None  # int32 [N] on the grid S_in S_w
    s_w: np.ndarray          # [N]
    s_in: float
    s_out: np.ndarray        # [N] output grid of each channel


@dataclass
class QNorm:
    gamma: np.ndarray
    beta: np.ndarray
    s_in: float
    s_out: float
    eps: float = 1e-5


@dataclass
class BlockCase:
    x: np.ndarray                         # int8 [B, T, D] on s["x"]
    s: dict = field(default_factory=dict)  # activation grids
    ln: dict = field(default_factory=dict)        # name -> QNorm
    lin: dict = field(default_factory=dict)       # name -> QLinear
    p: np.ndarray | None = None           # int8 [H, 2T-1, DH]
    u: np.ndarray | None = None           # int8 [H, DH] on the Q grid
    vb: np.ndarray | None = None
    dw_w: np.ndarray | None = None        # int8 [D, KDW] (BatchNorm folded)
    dw_bias: np.ndarray | None = None     # int32 [D]
    dw_sw: np.ndarray | None = None       # [D]
    attn_scales: dict = field(default_factory=dict)
    ref_out: np.ndarray | None = None     # float64 block output of the calibration utterances
    calib: int = 0
    ref: dict = field(default_factory=dict)   # float64 intermediates of those utterances


def _qw(w: np.ndarray):
    """Per-output-channel int8 weights (Eq. 6, min-max per row)."""
    s = np.maximum(np.abs(w).max(axis=1), 1e-12) / 127.0
    return np.clip(np.rint(w / s[:, None]), -127, 127).astype(np.int8), s


def _grid(a: np.ndarray, levels: int = 127) -> float:
    return max(float(np.abs(a).max()), 1e-12) / levels


def _ln(x, g, b, eps):
    mu = x.mean(-1, keepdims=True)
    var = ((x - mu) ** 2).mean(-1, keepdims=True)
    return g * (x - mu) / np.sqrt(var + eps) + b


def _sig(x):
    return 1.0 / (1.0 + np.exp(-x))


def _attention(q, k, v, p, u, vb):
    """Real-valued rel-pos attention: q, k, v [B, H, T, DH], p [H, 2T-1, DH]."""
    B, Hh, T, dh = q.shape
    idx = np.arange(T)[None, :] - np.arange(T)[:, None] + T - 1     # [i, j] -> r
    out = np.empty_like(q)
    for h in range(Hh):
        ac = np.einsum("bid,bjd->bij", q[:, h] + u[h], k[:, h])
        bd_full = np.einsum("bid,rd->bir", q[:, h] + vb[h], p[h])
        bd = np.take_along_axis(bd_full, np.broadcast_to(idx, (B, T, T)), axis=2)
        sc = (ac + bd) / math.sqrt(dh)
        sc -= sc.max(-1, keepdims=True)
        a = np.exp(sc)
        a /= a.sum(-1, keepdims=True)
        out[:, h] = a @ v[:, h]
    return out, (ac + bd) / math.sqrt(dh)


def conformer_block(B: int, T: int, seed: int, calib: int = 2) -> BlockCase:
    """Integer parameters and grids of one block, and an int8 input batch."""
    g = np.random.Generator(np.random.PCG64(np.random.SeedSequence(seed)))

    def lin(n, k, bias=True, gain=1.0):
        w = g.standard_normal((n, k)) * (gain / math.sqrt(k))
        b = g.normal(0.0, 0.05, size=n) if bias else None
        return w, b

    def norm():
        return g.uniform(0.5, 1.5, size=D), g.normal(0.0, 0.1, size=D)

    R = {}
    R["ln1"], R["ln2"], R["ln3"], R["ln4"], R["ln5"] = (norm() for _ in range(5))
    R["ff1a"], R["ff1b"] = lin(FF, D), lin(D, FF)
    R["ff2a"], R["ff2b"] = lin(FF, D), lin(D, FF)
    R["qkv"] = lin(3 * D, D)
    R["pos"] = lin(D, D, bias=False)
    R["out"] = lin(D, D)
    R["pw1"] = lin(2 * D, D)
    R["pw2"] = lin(D, D)
    dw = g.standard_normal((D, KDW)) / math.sqrt(KDW)
    dw_b = g.normal(0.0, 0.05, size=D)
    # BatchNorm with a wide spread of per-channel scales (the reason for INT16)
    bn_g = np.exp(g.normal(0.0, 1.5, size=D))
    bn_b = g.normal(0.0, 0.2, size=D)
    bn_mu = g.normal(0.0, 0.1, size=D)
    bn_var = g.uniform(0.5, 2.0, size=D)
    fold = bn_g / np.sqrt(bn_var + 1e-5)
    dw_f = dw * fold[:, None]
    dwb_f = (dw_b - bn_mu) * fold + bn_b
    u = g.normal(0.0, 0.1, size=(H, DH))
    vb = g.normal(0.0, 0.1, size=(H, DH))

    X = g.standard_normal((B, T, D))
    pos = sinusoid_relpos(T, D).astype(np.float64)                  # [2T-1, D]

    # ---- float64 forward of the real-valued block on the first utterances
    A = {}
    xc = X[:calib]
    A["x"] = X
    a1 = _ln(xc, *R["ln1"], 1e-5); A["ln1"] = a1
    z = a1 @ R["ff1a"][0].T + R["ff1a"][1]; A["ff1z"] = z
    h = z * _sig(z); A["ff1h"] = h
    f = h @ R["ff1b"][0].T + R["ff1b"][1]; A["ff1o"] = f
    z1 = xc + 0.5 * f; A["z1"] = z1
    a2 = _ln(z1, *R["ln2"], 1e-5); A["ln2"] = a2
    qkv = a2 @ R["qkv"][0].T + R["qkv"][1]
    q, k, v = (qkv[..., i * D:(i + 1) * D].reshape(calib, T, H, DH).transpose(0, 2, 1, 3)
               for i in range(3))
    A["q"], A["k"], A["v"] = q, k, v
    P = (pos @ R["pos"][0].T).reshape(2 * T - 1, H, DH).transpose(1, 0, 2)
    A["p"] = P
    o, sc = _attention(q, k, v, P, u, vb)
    A["s"], A["o"] = sc, o
    orow = o.transpose(0, 2, 1, 3).reshape(calib, T, D)
    mo = orow @ R["out"][0].T + R["out"][1]; A["mhsa"] = mo
    z2 = z1 + mo; A["z2"] = z2
    a3 = _ln(z2, *R["ln3"], 1e-5); A["ln3"] = a3
    ab = a3 @ R["pw1"][0].T + R["pw1"][1]
    A["pw1a"], A["pw1b"] = ab[..., :D], ab[..., D:]
    gl = ab[..., :D] * _sig(ab[..., D:]); A["glu"] = gl
    gp = np.pad(gl, ((0, 0), (KDW // 2, KDW // 2), (0, 0)))
    bn = sum(gp[:, kk:kk + T] * dw_f[:, kk] for kk in range(KDW)) + dwb_f; A["bn"] = bn
    sw = bn * _sig(bn); A["convsw"] = sw
    c = sw @ R["pw2"][0].T + R["pw2"][1]; A["conv"] = c
    z3 = z2 + c; A["z3"] = z3
    a4 = _ln(z3, *R["ln4"], 1e-5); A["ln4"] = a4
    z = a4 @ R["ff2a"][0].T + R["ff2a"][1]; A["ff2z"] = z
    h = z * _sig(z); A["ff2h"] = h
    f = h @ R["ff2b"][0].T + R["ff2b"][1]; A["ff2o"] = f
    z4 = z3 + 0.5 * f; A["z4"] = z4
    A["out"] = _ln(z4, *R["ln5"], 1e-5)

    S = {name: _grid(a) for name, a in A.items() if name != "bn"}
    # The dyadic multipliers of the integer path only scale down (m 2^-(31+s)
    # < 1): a residual sum's grid is kept at least as coarse as the terms it
    # adds, and the INT16 grid of the BatchNorm output at least as coarse as
    # the accumulator grid of its widest channel.
    for z, terms in (("z1", (("x", 1.0), ("ff1o", 0.5))), ("z2", (("z1", 1.0), ("mhsa", 1.0))),
                     ("z3", (("z2", 1.0), ("conv", 1.0))), ("z4", (("z3", 1.0), ("ff2o", 0.5)))):
        S[z] = max(S[z], max(a * S[t] for t, a in terms) * 1.0001)
    dw_q, dw_s = _qw(dw_f)
    S["bn"] = max(_grid(A["bn"], 32767), S["glu"] * float(dw_s.max()) * 1.0001)   # INT16 (Sec. 3.3)

    case = BlockCase(np.clip(np.rint(X / S["x"]), -127, 127).astype(np.int8), S)
    case.ref_out, case.calib = A["out"], calib
    case.ref = {k: v for k, v in A.items() if k not in ("x", "s", "p")}
    case.ref["x"] = xc
    for name, src, dst in [("ln1", "x", "ln1"), ("ln2", "z1", "ln2"), ("ln3", "z2", "ln3"),
                           ("ln4", "z3", "ln4"), ("ln5", "z4", "out")]:
        case.ln[name] = QNorm(R[name][0], R[name][1], S[src], S[dst])

    def qlin(name, w, b, s_in, s_out):
        wq, sw_ = _qw(w)
        bq = None if b is None else np.clip(np.rint(b / (s_in * sw_)), -(2 ** 30 - 1),
                                              2 ** 30 - 1).astype(np.int32)
        case.lin[name] = QLinear(wq, bq, sw_, s_in, np.broadcast_to(np.asarray(s_out, float),
                                                                    (w.shape[0],)).copy())

    qlin("ff1a", *R["ff1a"], S["ln1"], S["ff1z"])
    qlin("ff1b", *R["ff1b"], S["ff1h"], S["ff1o"])
    qlin("qkv", *R["qkv"], S["ln2"], np.repeat([S["q"], S["k"], S["v"]], D))
    qlin("out", *R["out"], S["o"], S["mhsa"])
    qlin("pw1", *R["pw1"], S["ln3"], np.repeat([S["pw1a"], S["pw1b"]], D))
    qlin("pw2", *R["pw2"], S["convsw"], S["conv"])
    qlin("ff2a", *R["ff2a"], S["ln4"], S["ff2z"])
    qlin("ff2b", *R["ff2b"], S["ff2h"], S["ff2o"])
    case.p = np.ascontiguousarray(np.clip(np.rint(P / S["p"]), -127, 127).astype(np.int8))
    case.u = np.clip(np.rint(u / S["q"]), -127, 127).astype(np.int8)
    case.vb = np.clip(np.rint(vb / S["q"]), -127, 127).astype(np.int8)
    case.dw_w, case.dw_sw = dw_q, dw_s
    case.dw_bias = np.clip(np.rint(dwb_f / (S["glu"] * case.dw_sw)), -(2 ** 30 - 1),
                           2 ** 30 - 1).astype(np.int32)
    case.attn_scales = {"S_Q": S["q"], "S_K": S["k"], "S_V": S["v"], "S_P": S["p"],
                        "S_s": S["s"], "S_O": S["o"]}
    return case
