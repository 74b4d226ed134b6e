"""Derived error bounds of the integer softmax against the real one.

The attention of Sec. 3.1 (after Eq. 11) takes its softmax from I-BERT
(Sec. 2.2, last paragraph): an integer exponential built from the
second-order fit g(x) = a (x + b)^2 + c of exp on [-ln2, 0], with the three
constants q_ln2 = floor(ln2 / S), q_b = floor(b / S), q_c = floor(c / (a S^2))
on the score grid S, then a division by the row sum onto the grid 2^-8.
This module writes out how far that can land from the real exponential and
softmax, step by step, so that the oracle's tests compare against bounds
that follow from the algorithm's roundings instead of measured tolerances.
It uses only the real constants (tests/golden/ibert_exp.txt), numpy and the
float64 reference; it shares nothing with the oracle or the GPU path.

Derivation, for an integer score difference d <= 0 and S < b - ln2:

1. Range reduction: q = floor(ln2 / S), z = floor(-d / q), p = d + z q in
   (-q, 0], so x = p S lies in (-ln2, 0].
2. Polynomial: since q_b and q_c are floored, q_b S = b - beta S and
   q_c a S^2 = c - gamma a S^2 with beta, gamma in [0, 1).  With x + b - S > 0,
       g(x) - 2 a S (x + b) < a S^2 ((p + q_b)^2 + q_c) <= g(x).
   The upper side is one-sided: every floor rounds down.
3. Shift: e = floor(L / 2^z) lies in (L 2^-z - 1, L 2^-z].
4. Against exp(d S) = e^x 2^(-z q S / ln2): the method evaluates
   ghat(x) = a (x + u)^2 + w with u = q_b S in (b - S, b] and w = q_c a S^2 in
   (c - a S^2, c], the same u and w for every key of a row.  So the factor
   kappa = ghat(0) / g(0) is common to all keys and cancels in the softmax;
   what is left is the shape F(x) = ghat(x) / ghat(0), which grows with w
   (for x <= 0) and, in u, has its extremes at the ends of the interval or
   where w = a u (x + u).  The normalised ratio
   rho(d) = e a S^2 / (kappa exp(d S)) then lies in [lo(d), hi(d)]:
       hi = g(0) F_max(x) / e^x * D,
       lo = g(0) F_min(x) / e^x * D - a S^2 e^(-d S) / kappa_min,
   D = 2^(-z (1 - q S / ln2)) <= 1: the integer exponential halves every q
   grid steps instead of every ln2 / S (the floor in q_ln2), so it decays
   faster by D.  On a coarse grid (q_ln2 = 7..9) D falls to about 0.9 within
   two halvings: with the score rounding of the layer (step 6) this is the
   largest error term there.
5. Normalisation: with p_j the real softmax of the same scores,
   e_j / sum_k e_k = p_j rho_j / rho_bar, rho_bar = sum_k p_k rho_k; f =
   floor(2^32 / sum) and a_j = min(255, floor(e_j f / 2^24)) give
       256 e_j / sum - 1 - e_j / 2^24 < a_j <= 256 e_j / sum,  a_j >= 0.
   rho_j / rho_bar grows with rho_j and falls with the other terms, so
       a_j <= 256 p_j hi_j / (p_j hi_j + sum_{k != j} p_k lo_k)
       a_j >= 256 p_j lo_j / (p_j lo_j + sum_{k != j} p_k hi_k) - 1 - L0 / 2^24
   with L0 = g(0) / (a S^2) >= every e_j.
6. Layer output (Eq. 9 then Eq. 7): the integer fused score q_j differs from
   the real score s_j / S by at most 1/2 + eps (rounding of Eq. 11, eps the
   dyadic multipliers' error), which multiplies each key's weight by at most
   e^(+-(1/2 + eps) S) (the row maximum's share is common to all keys and
   cancels) and moves the integer difference d_j within 1 + 2 eps of the real
   one.  With r = S_V / S_O, M = m_o 2^-(31+s_o) and Vbar = sum p_j V_j,
       |O_int - O_ref| <= r [ sum_j p_j |rho_j - c| |V_j - Vbar| / rho_bar
                              + sum_j min(1/256 + L0/2^32, e_j / sum) |V_j| ]
                          + |256 M - r| 127 + 1
   for any constant c (the first term rewrites sum_j p_j (rho_j - rho_bar) V_j),
   the second is the floor onto the 2^-8 grid (a probability loses less than
   one step, and never more than itself), the last two are the output
   multiplier's error and the two roundings onto the output grid.
"""
from __future__ import annotations

import math
import os

import numpy as np

LN2 = math.log(2.0)
_GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "ibert_exp.txt")


def _golden():
    vals = {}
    with open(_GOLDEN) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                k, v = line.split()
                vals[k] = float(v)
    return vals["a"], vals["b"], vals["c"]


A, B, C = _golden()
REL = 1e-9          # float64 evaluation slack of the bounds themselves


def g(x):
    """The real fit of exp on [-ln2, 0]."""
    return A * (x + B) ** 2 + C


def _reduce(S: float, d: np.ndarray):
    if not (0 < S < B - LN2):
        raise ValueError(f"the bounds need 0 < S < b - ln2, got S = {S}")
    q = math.floor(LN2 / S)
    z = np.floor(-d / q)
    x = (d + z * q) * S
    return q, z, x


def iexp_bounds(S: float, d) -> tuple[np.ndarray, np.ndarray]:
    """Steps 1-3: (lo, hi) with lo < e(d) a S^2 <= hi for integers d <= 0."""
    d = np.asarray(d, dtype=np.float64)
    q, z, x = _reduce(S, d)
    sh = 2.0 ** (-z)
    hi = g(x) * sh
    lo = (g(x) - 2 * A * S * (x + B)) * sh - A * S * S
    return lo, hi


def _shape_range(S: float, x: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """Extremes of F(x) = ghat(x) / ghat(0) over u in [b - S, b] and
    w in [c - a S^2, c] (step 4)."""
    def F(u, w):
        return (A * (x + u) ** 2 + w) / (A * u * u + w)

    out = []
    for w, pick in ((C - A * S * S, np.minimum), (C, np.maximum)):
        best = pick(F(B - S, w), F(B, w))
        # stationary point in u: a u^2 + a x u - w = 0
        ustar = (-A * x + np.sqrt(A * A * x * x + 4 * A * w)) / (2 * A)
        inside = (ustar > B - S) & (ustar < B)
        best = np.where(inside, pick(best, F(np.clip(ustar, B - S, B), w)), best)
        out.append(best)
    return out[0], out[1]


def kappa_min(S: float) -> float:
    """Smallest common factor ghat(0) / g(0) the floors allow."""
    return (A * (B - S) ** 2 + C - A * S * S) / g(0.0)


def rho_bounds(S: float, d) -> tuple[np.ndarray, np.ndarray]:
    """Step 4: (lo, hi) of rho(d) = e(d) a S^2 / (kappa exp(d S)), lo >= 0."""
    d = np.asarray(d, dtype=np.float64)
    q, z, x = _reduce(S, d)
    drift = 2.0 ** (-z * (1.0 - q * S / LN2))
    f_lo, f_hi = _shape_range(S, x)
    hi = g(0.0) * f_hi / np.exp(x) * drift
    lo = g(0.0) * f_lo / np.exp(x) * drift - A * S * S * np.exp(-d * S) / kappa_min(S)
    return np.maximum(lo, 0.0), hi


def l0(S: float) -> float:
    """Upper bound of every e_j: L(0) = q_b^2 + q_c <= g(0) / (a S^2)."""
    return g(0.0) / (A * S * S)


def _prob_bounds(p: np.ndarray, lo: np.ndarray, hi: np.ndarray, S: float):
    """Step 5 from per-key ratio ranges; p, lo, hi [..., n].  Returns the
    bounds (lower, upper) of a_j and the upper bound of e_j / sum."""
    plo, phi = p * lo, p * hi
    s_lo = plo.sum(-1, keepdims=True)
    s_hi = phi.sum(-1, keepdims=True)
    den_up = phi + (s_lo - plo)
    den_dn = plo + (s_hi - phi)
    share_up = np.divide(phi, den_up, out=np.where(p > 0, 1.0, 0.0), where=den_up > 0)
    share_dn = np.divide(plo, den_dn, out=np.zeros_like(p), where=den_dn > 0)
    upper = np.minimum(255.0, 256.0 * share_up) * (1 + REL) + REL
    lower = 256.0 * share_dn * (1 - REL) - 1.0 - l0(S) / 2.0 ** 24 - REL
    return lower, upper, share_up


def softmax_f64(scores: np.ndarray, S: float, valid: np.ndarray) -> np.ndarray:
    """Real softmax of S * scores over the first valid[r] keys of each row."""
    x = scores.astype(np.float64) * S
    n = scores.shape[-1]
    mask = np.arange(n)[None, :] < valid[:, None]
    x = np.where(mask, x, -np.inf)
    mx = np.max(x, axis=-1, keepdims=True)
    e = np.where(mask, np.exp(x - np.where(np.isfinite(mx), mx, 0)), 0.0)
    den = e.sum(-1, keepdims=True)
    return np.divide(e, den, out=np.zeros_like(e), where=den > 0)


def softmax_bounds(scores: np.ndarray, S: float, valid: np.ndarray):
    """Bounds (lower, upper) of the integer softmax a_j of int8 score rows
    [rows, n] with valid[r] keys, and the real softmax times 256."""
    p = softmax_f64(scores, S, valid)
    n = scores.shape[-1]
    mask = np.arange(n)[None, :] < valid[:, None]
    sc = scores.astype(np.int64)
    mx = np.max(np.where(mask, sc, -10 ** 6), axis=-1, keepdims=True)
    d = np.where(mask, sc - mx, 0)
    lo, hi = rho_bounds(S, d)
    lo = np.where(mask, lo, 0.0)
    hi = np.where(mask, hi, 0.0)
    lower, upper, _ = _prob_bounds(p, lo, hi, S)
    lower = np.where(mask, lower, 0.0)
    upper = np.where(mask, upper, 0.0)
    return lower, upper, 256.0 * p


def layer_output_bound(probs: np.ndarray, scores: np.ndarray, v: np.ndarray, S: float,
                       s_s: int, r: float, m_o: int, s_o: int, row_block: int = 64) -> np.ndarray:
    """Step 6: bound of |O_int - O_ref| per output [B, H, T, dh], in output
    steps.  probs and scores are the float64 reference's softmax and clipped
    real scores [B, H, T, T] (masked keys: probability 0, score -inf); v is
    the int8 V [B, H, T, dh]."""
    Bn, H, T, dh = v.shape
    eps = 2.0 ** (23 - 32 - s_s)        # |qc| + |qp| < 2^23 (int8 inputs, d_k = 128)
    half = 0.5 + eps + REL
    fin = np.isfinite(scores)
    smax = np.max(np.where(fin, scores, -np.inf), axis=-1, keepdims=True)
    smax = np.where(np.isfinite(smax), smax, 0.0)
    dreal = np.where(fin, (scores - smax) / S, 0.0)
    # the integer difference lies within 1 + 2 eps of the real one, in [-254, 0]
    table = np.arange(-254, 1, dtype=np.float64)
    t_lo, t_hi = rho_bounds(S, table)
    first = np.clip(np.floor(dreal - 1 - 2 * eps), -254, 0)
    last = np.clip(np.ceil(dreal + 1 + 2 * eps), -254, 0)
    lo = np.full(dreal.shape, np.inf)
    hi = np.full(dreal.shape, -np.inf)
    for off in range(4):
        cand = first + off
        use = cand <= last
        idx = (np.clip(cand, -254, 0) + 254).astype(np.int64)
        lo = np.where(use, np.minimum(lo, t_lo[idx]), lo)
        hi = np.where(use, np.maximum(hi, t_hi[idx]), hi)
    sf = math.exp(half * S)
    lo = np.where(fin, lo / sf, 0.0)
    hi = np.where(fin, hi * sf, 0.0)
    p = probs
    _, _, share_up = _prob_bounds(p, lo, hi, S)
    r_lo = np.sum(p * lo, axis=-1, keepdims=True)
    c = np.sum(p * (lo + hi) / 2, axis=-1, keepdims=True)
    dev = p * np.maximum(hi - c, c - lo)
    dev = np.divide(dev, r_lo, out=np.zeros_like(dev), where=r_lo > 0)
    floor_loss = np.minimum(1.0 / 256 + l0(S) / 2.0 ** 32, share_up)
    vf = v.astype(np.float64)
    vbar = np.einsum("bhij,bhjd->bhid", p, vf)
    term1 = np.empty_like(vbar)
    for b in range(Bn):
        for h in range(H):
            for i0 in range(0, T, row_block):
                i1 = min(T, i0 + row_block)
                diff = np.abs(vf[b, h][None, :, :] - vbar[b, h, i0:i1][:, None, :])
                term1[b, h, i0:i1] = np.einsum("ij,ijd->id", dev[b, h, i0:i1], diff)
    term2 = np.einsum("bhij,bhjd->bhid", floor_loss, np.abs(vf))
    M = m_o / 2.0 ** (31 + s_o)
    return r * (term1 + term2) * (1 + REL) + abs(256 * M - r) * 127 + 1 + REL
