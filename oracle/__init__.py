"""CPU oracle of the integer-only relative-positional MHSA (I-Parakeet, Sec. 3.1).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import this package.  It shares no
code with the GPU library: the arithmetic lives in ``ipo_mhsa.c`` (plain
int64 C, built here with gcc) and the offline integer constants in
``consts.py`` (float64, as the paper precomputes them offline, Eq. 7 and
Eq. 11).  Every function cites the passage it follows.

Pins: ``tests/test_oracle_*.py`` check this oracle against what the paper
and the mathematics fix (the literal Transformer-XL relative-shift route,
a float64 relative-position attention, closed forms of the integer softmax
and brute force on tiny inputs).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

from .consts import (IBERT_A, IBERT_B, IBERT_C, LayerConstants, dyadic,
                     dyadic_pair, isoftmax_params, layer_constants, linear_constants,
                     SWISH_A, SWISH_C, SwishParams, swish_params, NormConstants,
                     layernorm_constants, residual_params, glu_params, Swish16Params,
                     swish16_params)

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRCS = [os.path.join(_HERE, f) for f in ("ipo_mhsa.c", "ipo_linear.c", "ipo_norm.c", "ipo_block.c")]
_HDRS = [os.path.join(_HERE, f) for f in ("ipo_mhsa.h", "ipo_linear.h", "ipo_norm.h", "ipo_block.h")]
_LIB = os.path.join(_HERE, "libipo_mhsa.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the C oracle into ``oracle/libipo_mhsa.so`` (gcc, OpenMP)."""
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= max(
            os.path.getmtime(f) for f in _SRCS + _HDRS):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-Wall",
           "-Wextra", "-o", tmp] + _SRCS
    subprocess.run(cmd, check=True, cwd=_HERE)
    os.replace(tmp, _LIB)
    return _LIB


class _Params(ctypes.Structure):
    _fields_ = [("q_ln2", ctypes.c_int32), ("q_b", ctypes.c_int32),
                ("q_c", ctypes.c_int32)]


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            i32 = ctypes.c_int32
            lib.ipo_relpos_mhsa_i8.argtypes = [P] * 10 + [ctypes.c_int] * 4 + [P]
            lib.ipo_content_scores_i32.argtypes = [P, P, P] + [ctypes.c_int] * 4 + [P]
            lib.ipo_position_scores_i32.argtypes = [P, P, P] + [ctypes.c_int] * 4 + [P]
            lib.ipo_fused_scores_i8.argtypes = [P] * 5 + [i32, i32, i32] + [ctypes.c_int] * 4 + [P]
            lib.ipo_iexp.argtypes = [i32, P]
            lib.ipo_iexp.restype = ctypes.c_int64
            lib.ipo_isoftmax_u8.argtypes = [P, P, ctypes.c_int, ctypes.c_int, P, P]
            lib.ipo_set_threads.argtypes = [ctypes.c_int]
            lib.ipo_linear_i8.argtypes = [P, ctypes.c_int, P, P, P, P] + [ctypes.c_int] * 5 + [
                P, ctypes.c_int]
            lib.ipo_linear_i8.restype = ctypes.c_int
            lib.ipo_swish_i8.argtypes = [P, ctypes.c_longlong, P, P]
            lib.ipo_swish_i8.restype = ctypes.c_int
            LL = ctypes.c_longlong
            lib.ipo_residual_i8.argtypes = [P, P, LL, i32, i32, i32, P]
            lib.ipo_glu_i8.argtypes = [P, LL, ctypes.c_int, P, P]
            lib.ipo_dwconv_i16.argtypes = [P, ctypes.c_int, ctypes.c_int, ctypes.c_int, P,
                                           ctypes.c_int, P, P, P, P]
            lib.ipo_swish_i16.argtypes = [P, LL, P, P]
            for f in (lib.ipo_residual_i8, lib.ipo_glu_i8, lib.ipo_dwconv_i16, lib.ipo_swish_i16):
                f.restype = ctypes.c_int
            lib.ipo_isqrt.argtypes = [ctypes.c_int64]
            lib.ipo_isqrt.restype = ctypes.c_int64
            lib.ipo_layernorm_i8.argtypes = [P, ctypes.c_longlong, ctypes.c_int, ctypes.c_int64,
                                             P, P, P, P]
            lib.ipo_layernorm_i8.restype = ctypes.c_int
            for f in (lib.ipo_relpos_mhsa_i8, lib.ipo_content_scores_i32,
                      lib.ipo_position_scores_i32, lib.ipo_fused_scores_i8,
                      lib.ipo_isoftmax_u8, lib.ipo_set_threads):
                f.restype = ctypes.c_int
            _lib = lib
    return _lib


def _ptr(a: np.ndarray | None):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


def _params(c: LayerConstants) -> _Params:
    return _Params(*c.softmax)


class OracleError(RuntimeError):
    pass


def _check(rc: int, what: str):
    if rc != 0:
        raise OracleError(f"{what} returned {rc}")


def set_threads(n: int) -> int:
    """OpenMP threads for :func:`relpos_mhsa` (<= 0: all available)."""
    return _load().ipo_set_threads(n)


def relpos_mhsa(q, k, v, p, u, vb, c: LayerConstants, lengths=None) -> np.ndarray:
    """Whole integer rel-pos MHSA layer (Eqs. 8-11, I-BERT softmax, Eq. 9 and
    Eq. 7), int8 [B, H, T, dh]."""
    lib = _load()
    B, H, T, dh = q.shape
    out = np.empty_like(q)
    mult = np.array(c.multipliers, dtype=np.int32)
    sh = np.array(c.shifts, dtype=np.int32)
    sm = _params(c)
    lens = None if lengths is None else np.ascontiguousarray(lengths, dtype=np.int32)
    rc = lib.ipo_relpos_mhsa_i8(_ptr(q), _ptr(k), _ptr(v), _ptr(p), _ptr(u), _ptr(vb),
                                _ptr(mult), _ptr(sh), ctypes.addressof(sm), _ptr(lens),
                                B, H, T, dh, _ptr(out))
    _check(rc, "ipo_relpos_mhsa_i8")
    return out


def content_scores(q, k, u) -> np.ndarray:
    """A^c = (Q + 1u^T) K^T of Eq. 8, int32 [B, H, T, T]."""
    B, H, T, dh = q.shape
    out = np.empty((B, H, T, T), dtype=np.int32)
    _check(_load().ipo_content_scores_i32(_ptr(q), _ptr(k), _ptr(u), B, H, T, dh, _ptr(out)),
           "ipo_content_scores_i32")
    return out


def position_scores(q, p, vb) -> np.ndarray:
    """Phi((Q + 1v^T) P^T) of Eq. 8 through the static index map, int32 [B, H, T, T]."""
    B, H, T, dh = q.shape
    out = np.empty((B, H, T, T), dtype=np.int32)
    _check(_load().ipo_position_scores_i32(_ptr(q), _ptr(p), _ptr(vb), B, H, T, dh, _ptr(out)),
           "ipo_position_scores_i32")
    return out


def fused_scores(q, k, p, u, vb, m_c: int, m_p: int, s_s: int) -> np.ndarray:
    """Eq. 11 fused integer scores on the int8 grid, [B, H, T, T] (no mask)."""
    B, H, T, dh = q.shape
    out = np.empty((B, H, T, T), dtype=np.int8)
    _check(_load().ipo_fused_scores_i8(_ptr(q), _ptr(k), _ptr(p), _ptr(u), _ptr(vb),
                                       m_c, m_p, s_s, B, H, T, dh, _ptr(out)),
           "ipo_fused_scores_i8")
    return out


def iexp(d: int, softmax: tuple[int, int, int]) -> int:
    """I-BERT integer exponential of one integer d <= 0."""
    sm = _Params(*softmax)
    return int(_load().ipo_iexp(int(d), ctypes.addressof(sm)))


def isoftmax(scores: np.ndarray, softmax: tuple[int, int, int], valid=None) -> np.ndarray:
    """I-BERT integer softmax along the last axis of int8 scores; ``valid``
    gives per-row valid-key counts (default: all).  u8 on the grid 2^-8."""
    s = np.ascontiguousarray(scores, dtype=np.int8)
    n = s.shape[-1]
    rows = s.size // n
    if valid is None:
        valid = np.full(rows, n, dtype=np.int32)
    valid = np.ascontiguousarray(np.broadcast_to(valid, s.shape[:-1]).reshape(rows), dtype=np.int32)
    out = np.empty(s.shape, dtype=np.uint8)
    sm = _Params(*softmax)
    _check(_load().ipo_isoftmax_u8(_ptr(s), _ptr(valid), rows, n, ctypes.addressof(sm), _ptr(out)),
           "ipo_isoftmax_u8")
    return out


ROWS = 0
HEADS = 1


def linear(x, w, bias, m, s, *, x_layout: int = ROWS, y_layout: int = ROWS, groups: int = 1,
           B: int | None = None, T: int | None = None) -> np.ndarray:
    """Integer linear layer of Eqs. 6-7 (per-channel m, s; optional int32
    bias on the accumulator grid), int8.  ``x``: [B, T, K] (ROWS) or
    [B, K/128, T, 128] (HEADS); ``w``: [N, K].  Output [B, T, N] (ROWS) or
    [G, B, N/G/128, T, 128] (HEADS)."""
    x = np.ascontiguousarray(x, dtype=np.int8)
    w = np.ascontiguousarray(w, dtype=np.int8)
    N, K = w.shape
    if x_layout == ROWS:
        B, T, _ = x.shape
    else:
        B, _, T, _ = x.shape
    m = np.ascontiguousarray(m, dtype=np.int32)
    s = np.ascontiguousarray(s, dtype=np.int32)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.int32)
    if y_layout == ROWS:
        y = np.empty((B, T, N), dtype=np.int8)
    else:
        y = np.empty((groups, B, N // groups // 128, T, 128), dtype=np.int8)
    _check(_load().ipo_linear_i8(_ptr(x), x_layout, _ptr(w), _ptr(b), _ptr(m), _ptr(s),
                                 B, T, K, N, groups, _ptr(y), y_layout), "ipo_linear_i8")
    return y


class _Swish(ctypes.Structure):
    _fields_ = [("q_c", ctypes.c_int32), ("q_one", ctypes.c_int32), ("m", ctypes.c_int32),
                ("s", ctypes.c_int32)]


def swish(z, p: SwishParams) -> np.ndarray:
    """Integer minimax Swish (Eqs. 12-13) of int8 values on grid S_z, int8
    on grid S_y (constants from :func:`swish_params`)."""
    z = np.ascontiguousarray(z, dtype=np.int8)
    y = np.empty_like(z)
    prm = _Swish(p.q_c, p.q_one, p.m, p.s)
    _check(_load().ipo_swish_i8(_ptr(z), z.size, ctypes.addressof(prm), _ptr(y)), "ipo_swish_i8")
    return y


class _Swish16(ctypes.Structure):
    _fields_ = [("q_c", ctypes.c_int32), ("q_one", ctypes.c_int64), ("m", ctypes.c_int32),
                ("s", ctypes.c_int32)]


def residual(x, y, m_x: int, m_y: int, s: int) -> np.ndarray:
    """Residual addition of two int8 tensors onto one int8 grid (Eqs. 1-4)."""
    x = np.ascontiguousarray(x, dtype=np.int8)
    y = np.ascontiguousarray(y, dtype=np.int8)
    assert x.shape == y.shape
    z = np.empty_like(x)
    _check(_load().ipo_residual_i8(_ptr(x), _ptr(y), x.size, m_x, m_y, s, _ptr(z)),
           "ipo_residual_i8")
    return z


def glu(ab, p: SwishParams) -> np.ndarray:
    """Gated linear unit a sigma(b) over the last axis [a | b] of int8 ab."""
    ab = np.ascontiguousarray(ab, dtype=np.int8)
    C2 = ab.shape[-1]
    rows = ab.size // C2
    y = np.empty(ab.shape[:-1] + (C2 // 2,), dtype=np.int8)
    prm = _Swish(p.q_c, p.q_one, p.m, p.s)
    _check(_load().ipo_glu_i8(_ptr(ab), rows, C2 // 2, ctypes.addressof(prm), _ptr(y)),
           "ipo_glu_i8")
    return y


def dwconv(x, w, bias, m, s) -> np.ndarray:
    """Depthwise convolution over time with folded BatchNorm onto INT16,
    x int8 [B, T, C], w int8 [C, K]."""
    x = np.ascontiguousarray(x, dtype=np.int8)
    w = np.ascontiguousarray(w, dtype=np.int8)
    B, T, C = x.shape
    K = w.shape[1]
    y = np.empty((B, T, C), dtype=np.int16)
    b = np.ascontiguousarray(bias, dtype=np.int32)
    m = np.ascontiguousarray(m, dtype=np.int32)
    s = np.ascontiguousarray(s, dtype=np.int32)
    _check(_load().ipo_dwconv_i16(_ptr(x), B, T, C, _ptr(w), K, _ptr(b), _ptr(m), _ptr(s),
                                  _ptr(y)), "ipo_dwconv_i16")
    return y


def swish16(z, p: "Swish16Params") -> np.ndarray:
    """Integer Swish of INT16 values onto int8."""
    z = np.ascontiguousarray(z, dtype=np.int16)
    y = np.empty(z.shape, dtype=np.int8)
    prm = _Swish16(p.q_c, p.q_one, p.m, p.s)
    _check(_load().ipo_swish_i16(_ptr(z), z.size, ctypes.addressof(prm), _ptr(y)),
           "ipo_swish_i16")
    return y


def isqrt(n: int) -> int:
    """floor(sqrt(n)) of the oracle's integer Newton iteration, 0 <= n < 2^62."""
    return int(_load().ipo_isqrt(int(n)))


def layernorm(x, c: "NormConstants") -> np.ndarray:
    """Integer LayerNorm over the last axis (d channels) of int8 x; constants
    from :func:`layernorm_constants`."""
    x = np.ascontiguousarray(x, dtype=np.int8)
    d = x.shape[-1]
    rows = x.size // d
    y = np.empty_like(x)
    M = np.ascontiguousarray(c.M, dtype=np.int32)
    B = np.ascontiguousarray(c.B, dtype=np.int64)
    E = np.ascontiguousarray(c.E, dtype=np.int32)
    _check(_load().ipo_layernorm_i8(_ptr(x), rows, d, int(c.eps_c), _ptr(M), _ptr(B), _ptr(E),
                                    _ptr(y)), "ipo_layernorm_i8")
    return y


__all__ = ["build", "linear", "swish", "isqrt", "layernorm", "layernorm_constants",
           "NormConstants", "residual", "glu", "dwconv", "swish16", "residual_params",
           "glu_params", "swish16_params", "Swish16Params", "swish_params", "SwishParams", "SWISH_A", "SWISH_C", "linear_constants", "ROWS", "HEADS", "relpos_mhsa", "content_scores", "position_scores",
           "fused_scores", "iexp", "isoftmax", "set_threads", "dyadic",
           "dyadic_pair", "isoftmax_params", "layer_constants", "LayerConstants",
           "IBERT_A", "IBERT_B", "IBERT_C", "OracleError"]
