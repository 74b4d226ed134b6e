"""Real-valued relative-positional attention (Eqs. 8-9 in float64).

This is the floating-point definition the integer method approximates
(Sec. 3.1): dequantise the int8 inputs with their declared scales, form the
content and position branches, realign the position branch with the
relative shift, scale by 1/sqrt(d_k), take an exact softmax over the valid
keys, multiply by V and quantise the result onto the output grid (Eq. 6).
It shares nothing with the integer oracle and serves to pin it.
"""
from __future__ import annotations

import numpy as np


def relshift_gather(bd: np.ndarray) -> np.ndarray:
    """Phi as a gather: out[..., i, j] = bd[..., i, j - i + T - 1]."""
    T = bd.shape[-2]
    i = np.arange(T)[:, None]
    j = np.arange(T)[None, :]
    return np.take_along_axis(bd, np.broadcast_to(j - i + T - 1, bd.shape[:-2] + (T, T)), axis=-1)


def attention_f64(lay, lengths=None, clip_scores=True):
    """Float64 attention of one layer.

    With ``clip_scores`` the fused real score is clipped to the range of its
    int8 grid, +-127 S_s (the clip of Eq. 6), before the softmax.
    Returns (O_real, O quantised onto S_O, probabilities, scores)."""
    sc = lay.scales
    B, H, T, dh = lay.q.shape
    q = lay.q.astype(np.float64) * sc["S_Q"]
    k = lay.k.astype(np.float64) * sc["S_K"]
    v = lay.v.astype(np.float64) * sc["S_V"]
    p = lay.p.astype(np.float64) * sc["S_P"]
    u = lay.u.astype(np.float64) * sc["S_Q"]
    vb = lay.vb.astype(np.float64) * sc["S_Q"]
    ac = np.einsum("bhid,bhjd->bhij", q + u[None, :, None, :], k)
    bd = np.einsum("bhid,hrd->bhir", q + vb[None, :, None, :], p)
    s = (ac + relshift_gather(bd)) / np.sqrt(dh)
    if clip_scores:
        lim = 127 * sc["S_s"]
        s = np.clip(s, -lim, lim)
    if lengths is None:
        lengths = np.full(B, T)
    lens = np.clip(np.asarray(lengths), 0, T)
    keymask = np.arange(T)[None, :] < lens[:, None]                 # [B, T]
    s = np.where(keymask[:, None, None, :], s, -np.inf)
    mx = np.max(s, axis=-1, keepdims=True)
    mx = np.where(np.isfinite(mx), mx, 0.0)
    e = np.exp(s - mx)
    den = np.sum(e, axis=-1, keepdims=True)
    a = np.divide(e, den, out=np.zeros_like(e), where=den > 0)
    o = np.einsum("bhij,bhjd->bhid", a, v)
    rowmask = (np.arange(T)[None, :] < lens[:, None])[:, None, :, None]
    o = np.where(rowmask, o, 0.0)
    oq = np.clip(np.rint(o / sc["S_O"]), -127, 127).astype(np.int64)
    return o, oq, a, s
