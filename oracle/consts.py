"""Offline integer constants of the oracle (float64 on the host, as the paper
precomputes its multipliers offline, Sec. 2.2 under Eq. 7).

TEST INFRASTRUCTURE ONLY (see the package docstring).

* Dyadic multipliers (Eq. 7, Eq. 11).  The paper writes a real ratio r as
  m 2^-n with n = 16.  Here the same dyadic form carries more bits: m is a
  31-bit integer, normalised into [2^30, 2^31) when possible, and the total
  right shift is n = 31 + s with 0 <= s <= 31 (so r = m 2^-(31+s)).
* Fused-branch pair (Eq. 11): m_c and m_p share one shift, taken from the
  larger ratio; the smaller multiplier is rounded on the same shift.
* I-BERT softmax constants (Kim et al., ICML 2021, integer-only exponential):
  exp(p) on [-ln2, 0] ~ a (p + b)^2 + c with a = 0.3585, b = 1.353,
  c = 0.344, and on the grid S: q_ln2 = floor(ln2/S), q_b = floor(b/S),
  q_c = floor(c / (a S^2)).
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

IBERT_A = 0.3585
IBERT_B = 1.353
IBERT_C = 0.344
LN2 = math.log(2.0)
SOFTMAX_BITS = 8          # attention probabilities on the grid 2^-8


def dyadic(ratio: float) -> tuple[int, int]:
    """(m, s) with m 2^-(31+s) the nearest such value to ``ratio`` and
    m in [2^30, 2^31) unless s had to be clipped to 31."""
    if not (ratio > 0.0) or not math.isfinite(ratio):
        raise ValueError(f"ratio must be positive and finite, got {ratio!r}")
    frac, exp = math.frexp(ratio)          # ratio = frac 2^exp, frac in [0.5, 1)
    s = -exp
    if s > 31:
        s = 31
        m = math.floor(ratio * 2.0 ** 62 + 0.5)
        return int(m), s
    if s < 0:
        raise ValueError(f"ratio {ratio!r} >= 1/2^0 cannot be encoded with s >= 0")
    m = math.floor(frac * 2.0 ** 31 + 0.5)
    if m == 2 ** 31:
        m, s = 2 ** 30, s - 1
        if s < 0:
            raise ValueError(f"ratio {ratio!r} rounds to 1")
    return int(m), int(s)


def dyadic_pair(r_c: float, r_p: float) -> tuple[int, int, int]:
    """(m_c, m_p, s) for the two branch ratios of Eq. 11 on one shared shift."""
    m_big, s = dyadic(max(r_c, r_p))
    scale = 2.0 ** (31 + s)
    m_c = int(math.floor(r_c * scale + 0.5))
    m_p = int(math.floor(r_p * scale + 0.5))
    if max(m_c, m_p) >= 2 ** 31:
        raise ValueError("multiplier overflow")
    return m_c, m_p, s


def isoftmax_params(S: float) -> tuple[int, int, int]:
    """(q_ln2, q_b, q_c) of I-BERT's integer exponential on the grid S."""
    q_ln2 = math.floor(LN2 / S)
    q_b = math.floor(IBERT_B / S)
    q_c = math.floor(IBERT_C / (IBERT_A * (S * S)))
    return int(q_ln2), int(q_b), int(q_c)


@dataclass(frozen=True)
class LayerConstants:
    multipliers: tuple[int, int, int]     # m_c, m_p, m_o
    shifts: tuple[int, int]               # s_s, s_o  (total shift 31 + s)
    softmax: tuple[int, int, int]         # q_ln2, q_b, q_c


def layer_constants(scales: dict, dh: int) -> LayerConstants:
    """Integer constants of one layer from its declared real scales.

    Eq. 11: r_c = S_Q S_K / (S_s sqrt(dh)), r_p = S_Q S_P / (S_s sqrt(dh)).
    Eq. 7 for A.V: r_o = 2^-8 S_V / S_O (probabilities on the grid 2^-8).
    """
    root = math.sqrt(dh)
    r_c = scales["S_Q"] * scales["S_K"] / (scales["S_s"] * root)
    r_p = scales["S_Q"] * scales["S_P"] / (scales["S_s"] * root)
    r_o = scales["S_V"] / (scales["S_O"] * 2.0 ** SOFTMAX_BITS)
    m_c, m_p, s_s = dyadic_pair(r_c, r_p)
    m_o, s_o = dyadic(r_o)
    return LayerConstants((m_c, m_p, m_o), (s_s, s_o), isoftmax_params(scales["S_s"]))


def linear_constants(s_x: float, s_w, s_y) -> tuple[np.ndarray, np.ndarray]:
    """Per-output-channel constants of Eq. 7: m[n], s[n] with
    m 2^-(31+s) the dyadic nearest to S_x S_w[n] / S_y[n] (weights carry one
    scale per channel, Sec. 2.2).  Returns int32 arrays (m, s)."""
    s_w = np.asarray(s_w, dtype=np.float64)
    s_y = np.broadcast_to(np.asarray(s_y, dtype=np.float64), s_w.shape)
    m = np.empty(s_w.shape, dtype=np.int32)
    s = np.empty(s_w.shape, dtype=np.int32)
    for n in range(s_w.size):
        m[n], s[n] = dyadic(float(s_x) * float(s_w[n]) / float(s_y[n]))
    return m, s


# Minimax fit of Eq. 13 (Sec. 3.2): tanh(u) ~ sgn(u) [a (min(|u|, c) - c)^2 + 1]
SWISH_A = -0.1240
SWISH_C = 2.4632


@dataclass(frozen=True)
class SwishParams:
    q_c: int
    q_one: int
    m: int
    s: int


def swish_params(s_z: float, s_y: float, a: float = SWISH_A, c: float = SWISH_C) -> SwishParams:
    """Integer constants of the Swish of Eqs. 12-13 for an int8 input on
    grid S_z and an int8 output on grid S_y (offline, float64): the clip
    point q_c = round(2c / S_z) of |z|, the 1 of the polynomial on its grid
    S_t = |a| (S_z/2)^2, q_one = round(1 / S_t), and the dyadic m 2^-(31+s)
    of S_z S_t / (2 S_y)."""
    if not (a < 0 and c > 0 and s_z > 0 and s_y > 0):
        raise ValueError("need a < 0, c > 0 and positive grids")
    s_t = abs(a) * (s_z / 2.0) ** 2
    q_c = int(math.floor(2.0 * c / s_z + 0.5))
    q_one = int(math.floor(1.0 / s_t + 0.5))
    m, s = dyadic(s_z * s_t / (2.0 * s_y))
    return SwishParams(q_c, q_one, m, s)


@dataclass(frozen=True)
class NormConstants:
    eps_c: int            # epsilon on the grid of c^2, c = d (q - mean)
    M: np.ndarray         # int32 [d]
    B: np.ndarray         # int64 [d]
    E: np.ndarray         # int32 [d], total right shift


def layernorm_constants(s_x: float, gamma, beta, s_y: float, eps: float = 1e-5) -> NormConstants:
    """Integer constants of the LayerNorm for an int8 input on grid S_x and
    an int8 output on S_y (offline, float64).  The normalised value reaches
    the affine step as n = (x - mean) / sqrt(var + eps) on the grid 2^-15;
    per channel y = (gamma_i 2^-15 n + beta_i) / S_y = (M_i n + B_i) 2^-E_i,
    with (|M_i|, E_i - 31) the dyadic of |gamma_i| 2^-15 / S_y (sign of
    gamma_i on M_i; gamma_i = 0 gives M_i = 0, E_i = 31) and B_i =
    round(beta_i / S_y 2^E_i).  eps_c = round(eps d^2 / S_x^2): var in units
    of c^2 / d where c = d (q - mean)."""
    gamma = np.asarray(gamma, dtype=np.float64)
    beta = np.asarray(beta, dtype=np.float64)
    d = gamma.size
    M = np.zeros(d, dtype=np.int32)
    E = np.full(d, 31, dtype=np.int32)
    B = np.zeros(d, dtype=np.int64)
    for i in range(d):
        g = float(gamma[i])
        if g != 0.0:
            m, s = dyadic(abs(g) * 2.0 ** -15 / s_y)
            M[i] = m if g > 0 else -m
            E[i] = 31 + s
        b = math.floor(float(beta[i]) / s_y * 2.0 ** int(E[i]) + 0.5)
        if abs(b) >= 2 ** 60:
            raise ValueError(f"beta/gamma ratio of channel {i} out of range")
        B[i] = b
    eps_c = int(math.floor(eps * d * d / (s_x * s_x) + 0.5))
    return NormConstants(eps_c, M, B, E)


def residual_params(s_x: float, s_y: float, s_z: float, alpha: float = 1.0) -> tuple[int, int, int]:
    """(m_x, m_y, s) of the residual addition z = x + alpha y (Eqs. 1-4) onto
    S_z: the dyadic pair of S_x / S_z and alpha S_y / S_z on one shift."""
    return dyadic_pair(s_x / s_z, alpha * s_y / s_z)


def glu_params(s_a: float, s_b: float, s_y: float, a: float = SWISH_A,
               c: float = SWISH_C) -> SwishParams:
    """Constants of GLU(a, b) = a sigma(b), sigma(b) = (1 + tanh(b/2)) / 2
    with the minimax tanh: q_c, q_one on the grid of b, and the dyadic of
    S_a S_t / (2 S_y), S_t = |a| (S_b/2)^2."""
    s_t = abs(a) * (s_b / 2.0) ** 2
    q_c = int(math.floor(2.0 * c / s_b + 0.5))
    q_one = int(math.floor(1.0 / s_t + 0.5))
    m, s = dyadic(s_a * s_t / (2.0 * s_y))
    return SwishParams(q_c, q_one, m, s)


@dataclass(frozen=True)
class Swish16Params:
    q_c: int
    q_one: int
    m: int
    s: int


def swish16_params(s_z: float, s_y: float, a: float = SWISH_A, c: float = SWISH_C) -> Swish16Params:
    """Swish constants for an INT16 input grid S_z (the BatchNorm output of
    Sec. 3.3) onto an int8 grid S_y; as swish_params."""
    p = swish_params(s_z, s_y, a, c)
    if not (1 <= p.q_c < 2 ** 16 and 1 <= p.q_one < 2 ** 31 and p.q_one >= p.q_c ** 2):
        raise ValueError(f"INT16 grid {s_z!r} outside the Swish domain (q_c={p.q_c}, q_one={p.q_one})")
    return Swish16Params(p.q_c, p.q_one, p.m, p.s)
