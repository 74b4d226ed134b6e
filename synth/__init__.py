"""Seeded synthetic workloads for the integer relative-positional MHSA.

This module draws inputs only.  It holds none of the attention arithmetic:
it produces int8 tensors shaped like the Conformer encoder of a
Parakeet-CTC-0.6B model (d_model = 1024, 8 heads of 128, Sec. 2.1) together
with the real-valued quantisation scales that an offline calibration would
declare for them (Eq. 6, min-max ranges).  Both the CPU oracle and the CUDA
path consume exactly what this module returns; each turns the declared
scales into its own integer constants.

Recipe (numpy PCG64 streams spawned from SeedSequence(seed), seed =
1000 * config + layer unless given):

* Q, K, V, u, v : round(N(0, 30^2)) clipped to [-127, 127]
  (long-form workload: Q, K, V = round(t_3 * 25) clipped to [-127, 127]).
* P : the tiny workload draws it like Q.  The others build it the way the
  model does (Sec. 3.1): the 2T-1 sinusoidal relative-position embeddings
  (row r <-> relative distance T-1-r, d = 1024), quantised to int8 with
  S = 1/127, projected through a seeded int8 W_pos [1024, 1024] ~
  round(N(0, 20^2)), requantised to int8 by its min-max range and split into
  8 heads of 128.
* lengths (masked workload): uniform integers in [T/2, T].
* declared scales: alpha_X ~ U[2, 6] for X in {Q, K, V, P}, S_X = alpha_X/127
  (u and v live on Q's grid).  S_s, the fused-score grid, is the min-max
  range estimated from second moments (kappa_s * sigma, kappa_s ~ U[3.5, 5]),
  so that a few scores saturate at +-127.  S_O = kappa_O * S_V with
  kappa_O ~ U[1.0625, 1.9375] keeps the output requantisation shift at 8.
"""
from __future__ import annotations

import math
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field

import numpy as np

D_MODEL = 1024
N_HEADS = 8
D_HEAD = 128


@dataclass(frozen=True)
class Workload:
    """One named workload: shape and input distribution."""
    key: int
    name: str
    B: int
    T: int
    layers: int = 1
    H: int = N_HEADS
    dh: int = D_HEAD
    p_mode: str = "sinusoid"      # "random" | "sinusoid"
    dist: str = "normal"          # "normal" | "t3"
    masked: bool = False

    @property
    def R(self) -> int:
        return 2 * self.T - 1

    def useful_ops(self) -> int:
        """Useful integer ops of the whole workload: 6 * dh * T^2 per (b, h)
        per layer (content, position and attn.V products, one MAC = 2 ops)."""
        return 6 * self.dh * self.T * self.T * self.B * self.H * self.layers

    def describe(self) -> str:
        return (f"{self.name}: B={self.B} H={self.H} dh={self.dh} T={self.T} "
                f"layers={self.layers} P={self.p_mode} dist={self.dist} "
                f"masked={self.masked}")


WORKLOADS = {
    0: Workload(0, "tiny-T64", B=1, T=64, p_mode="random"),
    1: Workload(1, "utt10s-T125", B=1, T=125),
    2: Workload(2, "batch20s-masked-T250", B=16, T=250, masked=True),
    3: Workload(3, "encoder24-B32-T375", B=32, T=375, layers=24),
    4: Workload(4, "longform-T1500-t3", B=4, T=1500, dist="t3"),
}


@dataclass
class Layer:
    """Inputs of one attention layer.  Arrays are C-contiguous numpy."""
    q: np.ndarray            # int8 [B, H, T, dh]
    k: np.ndarray            # int8 [B, H, T, dh]
    v: np.ndarray            # int8 [B, H, T, dh]
    p: np.ndarray            # int8 [H, 2T-1, dh]
    u: np.ndarray            # int8 [H, dh]
    vb: np.ndarray           # int8 [H, dh]
    lengths: np.ndarray | None   # int32 [B] or None (all T)
    scales: dict = field(default_factory=dict)   # declared real scales

    @property
    def shape(self):
        B, H, T, dh = self.q.shape
        return B, H, T, dh


_NCHUNK = 16          # fixed split of every large draw (independent of threads)
_POOL = None


def _pool():
    global _POOL
    if _POOL is None:
        _POOL = ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 1))
    return _POOL


def _draw_int8(seq: np.random.SeedSequence, shape, dist: str, scale: float) -> np.ndarray:
    """int8 draw of `shape`: round(N(0,1) * scale) or round(t_3 * scale),
    clipped to [-127, 127]; filled in _NCHUNK pieces, each from its own
    child seed, on a thread pool (numpy releases the GIL while drawing)."""
    n = int(np.prod(shape))
    out = np.empty(n, dtype=np.int8)
    kids = seq.spawn(_NCHUNK)
    bounds = [n * c // _NCHUNK for c in range(_NCHUNK + 1)]

    def fill(c):
        lo, hi = bounds[c], bounds[c + 1]
        if hi <= lo:
            return
        g = np.random.Generator(np.random.PCG64(kids[c]))
        if dist == "normal":
            x = g.standard_normal(hi - lo, dtype=np.float32)
        else:
            x = g.standard_t(3, size=hi - lo).astype(np.float32)
        x *= np.float32(scale)
        np.rint(x, out=x)
        np.clip(x, -127, 127, out=x)
        out[lo:hi] = x.astype(np.int8)

    if n >= 1 << 20:
        list(_pool().map(fill, range(_NCHUNK)))
    else:
        for c in range(_NCHUNK):
            fill(c)
    return out.reshape(shape)


def sinusoid_relpos(T: int, d: int = D_MODEL) -> np.ndarray:
    """Sinusoidal embeddings of the 2T-1 relative distances, row r <->
    distance T-1-r, interleaved sin/cos with frequencies 10000^(-2k/d)."""
    pos = (T - 1 - np.arange(2 * T - 1, dtype=np.float64))[:, None]
    freq = np.power(10000.0, -np.arange(0, d, 2, dtype=np.float64) / d)[None, :]
    pe = np.empty((2 * T - 1, d), dtype=np.float64)
    pe[:, 0::2] = np.sin(pos * freq)
    pe[:, 1::2] = np.cos(pos * freq)
    return pe


def _projected_p(seq: np.random.SeedSequence, T: int, H: int, dh: int) -> np.ndarray:
    d = H * dh
    e = np.rint(sinusoid_relpos(T, d) * 127.0)                 # int8 grid, S = 1/127
    w = _draw_int8(seq, (d, d), "normal", 20.0).astype(np.float64)
    acc = e @ w.T                                              # exact: |acc| < 2^53
    amax = float(np.max(np.abs(acc)))
    p = np.clip(np.rint(acc * (127.0 / amax)), -127, 127).astype(np.int8)
    return np.ascontiguousarray(p.reshape(2 * T - 1, H, dh).transpose(1, 0, 2))


def _rms(x: np.ndarray) -> float:
    """Root mean square of an int8 array, exact (integer sums below 2^53)."""
    flat = x.reshape(-1)
    total = 0.0
    step = 1 << 22
    for lo in range(0, flat.size, step):
        xf = flat[lo:lo + step].astype(np.float64)
        total += float(np.dot(xf, xf))
    return math.sqrt(total / max(flat.size, 1))


def draw(B: int, H: int, T: int, dh: int, seed: int, *, p_mode: str = "random",
         dist: str = "normal", masked: bool = False,
         lengths: np.ndarray | None = None) -> Layer:
    """Draw one layer of inputs of an arbitrary shape."""
    root = np.random.SeedSequence(seed)
    s_q, s_k, s_v, s_u, s_vb, s_p, s_len, s_sc = root.spawn(8)
    shape = (B, H, T, dh)
    if dist == "t3":
        q, k, v = (_draw_int8(sq, shape, "t3", 25.0) for sq in (s_q, s_k, s_v))
    elif dist == "normal":
        q, k, v = (_draw_int8(sq, shape, "normal", 30.0) for sq in (s_q, s_k, s_v))
    else:
        raise ValueError(f"unknown distribution {dist!r}")
    u = _draw_int8(s_u, (H, dh), "normal", 30.0)
    vb = _draw_int8(s_vb, (H, dh), "normal", 30.0)
    if p_mode == "random":
        p = _draw_int8(s_p, (H, 2 * T - 1, dh), "normal", 30.0)
    elif p_mode == "sinusoid":
        p = _projected_p(s_p, T, H, dh)
    else:
        raise ValueError(f"unknown P mode {p_mode!r}")
    if lengths is None and masked:
        g = np.random.Generator(np.random.PCG64(s_len))
        lengths = g.integers(T // 2, T, size=B, endpoint=True).astype(np.int32)
    elif lengths is not None:
        lengths = np.ascontiguousarray(lengths, dtype=np.int32)

    rng = np.random.Generator(np.random.PCG64(s_sc))
    a_q, a_k, a_v, a_p = (float(x) for x in rng.uniform(2.0, 6.0, size=4))
    s_q, s_k, s_v, s_p = a_q / 127, a_k / 127, a_v / 127, a_p / 127
    # Second-moment estimate of the real fused score (Q+u)K^T + (Q+v)P^T,
    # divided by sqrt(dh); its min-max range is taken as kappa_s sigma.
    rq = _rms(q)
    sig_c = math.sqrt(dh) * math.hypot(rq, _rms(u)) * _rms(k) * s_q * s_k
    sig_p = math.sqrt(dh) * math.hypot(rq, _rms(vb)) * _rms(p) * s_q * s_p
    sigma = math.hypot(sig_c, sig_p) / math.sqrt(dh)
    kappa_s = float(rng.uniform(3.5, 5.0))
    s_s = kappa_s * sigma / 127
    s_o = float(rng.uniform(1.0625, 1.9375)) * s_v
    scales = dict(S_Q=s_q, S_K=s_k, S_V=s_v, S_P=s_p, S_s=s_s, S_O=s_o)
    return Layer(q=q, k=k, v=v, p=p, u=u, vb=vb, lengths=lengths, scales=scales)


def layer(workload: int | Workload, index: int = 0, seed: int | None = None) -> Layer:
    """Inputs of layer `index` of a named workload."""
    w = WORKLOADS[workload] if isinstance(workload, int) else workload
    if seed is None:
        seed = 1000 * w.key + index
    return draw(w.B, w.H, w.T, w.dh, seed, p_mode=w.p_mode, dist=w.dist,
                masked=w.masked)



# ------------------------------------------------------------ linear layers

@dataclass
class LinearCase:
    """Inputs of one integer linear layer (Eqs. 6-7): int8 activations x
    [B, T, K], int8 weights w [N, K] (one row per output channel), an int32
    bias on the accumulator grid S_x S_w[n] (or None), and the declared
    scales: S_x, per-channel S_w [N], and S_y per output group (the G
    stacked projections of a head-split output each have their own grid)."""
    x: np.ndarray
    w: np.ndarray
    bias: np.ndarray | None
    s_x: float
    s_w: np.ndarray
    s_y: np.ndarray          # [G]
    groups: int = 1

    def s_y_per_channel(self) -> np.ndarray:
        N = self.w.shape[0]
        return np.repeat(self.s_y, N // self.groups)


def linear(B: int, T: int, K: int, N: int, seed: int, *, groups: int = 1,
           bias: bool = True, dist: str = "normal", calib_frames: int = 256) -> LinearCase:
    """Seeded linear-layer case shaped like the encoder's projections
    (d = 1024 in and out; Q, K, V stacked as three groups).

    x: round(N(0, 30^2)) (or t_3 * 25) clipped to [-127, 127]; w row n:
    round(N(0, sigma_n^2)), sigma_n ~ U[15, 45], clipped; S_x = alpha_x/127
    with alpha_x ~ U[2, 6]; S_w[n] = alpha_n/127 with alpha_n ~ U[0.05,
    0.3]; real bias ~ N(0, 0.5^2) put on the accumulator grid; S_y of each
    group = the min-max of the real output over the first `calib_frames`
    frames / 127 (the offline calibration of Eq. 6)."""
    seq = np.random.SeedSequence(seed)
    kx, kw, kb, ks = seq.spawn(4)
    x = _draw_int8(kx, (B, T, K), dist, 30.0 if dist == "normal" else 25.0)
    g = np.random.Generator(np.random.PCG64(ks))
    sig = g.uniform(15.0, 45.0, size=N)
    gw = np.random.Generator(np.random.PCG64(kw))
    wf = gw.standard_normal((N, K), dtype=np.float32) * sig[:, None].astype(np.float32)
    w = np.clip(np.rint(wf), -127, 127).astype(np.int8)
    s_x = g.uniform(2.0, 6.0) / 127.0
    s_w = g.uniform(0.05, 0.3, size=N) / 127.0
    bq = None
    if bias:
        gb = np.random.Generator(np.random.PCG64(kb))
        real = gb.normal(0.0, 0.5, size=N)
        bq = np.clip(np.rint(real / (s_x * s_w)), -(2**30 - 1), 2**30 - 1).astype(np.int32)
    # calibration: real output of the first frames, float64
    frames = x.reshape(-1, K)[:max(1, min(calib_frames, B * T))].astype(np.float64)
    acc = frames @ w.astype(np.float64).T
    if bq is not None:
        acc += bq.astype(np.float64)
    yr = acc * (s_x * s_w)[None, :]
    per = N // groups
    s_y = np.array([max(np.abs(yr[:, gi * per:(gi + 1) * per]).max(), 1e-30) / 127.0
                    for gi in range(groups)])
    return LinearCase(x, w, bq, float(s_x), s_w, s_y, groups)


# ------------------------------------------------------------ LayerNorm

@dataclass
class NormCase:
    """Inputs of one integer LayerNorm: int8 frames x [rows, d] on grid S_x
    (the residual stream), real per-channel gamma and beta, the output grid
    S_y and epsilon."""
    x: np.ndarray
    gamma: np.ndarray
    beta: np.ndarray
    s_x: float
    s_y: float
    eps: float = 1e-5


def norm(rows: int, d: int, seed: int, eps: float = 1e-5) -> NormCase:
    """Seeded LayerNorm case: each frame round(N(mu_r, 35^2)) clipped to
    +-127 with a per-frame offset mu_r ~ N(0, 10^2); gamma ~ U[0.3, 2] with
    10 % negative, beta ~ N(0, 0.5^2); S_x = alpha/127, alpha ~ U[2, 6];
    S_y = alpha_y/127, alpha_y ~ U[3, 8] (a normalised output stays within
    a few units)."""
    g = np.random.Generator(np.random.PCG64(np.random.SeedSequence(seed)))
    mu = g.normal(0.0, 10.0, size=(rows, 1)).astype(np.float32)
    xf = g.standard_normal((rows, d), dtype=np.float32) * np.float32(35.0) + mu
    x = np.clip(np.rint(xf), -127, 127).astype(np.int8)
    gamma = g.uniform(0.3, 2.0, size=d) * g.choice([-1.0, 1.0], size=d, p=[0.1, 0.9])
    beta = g.normal(0.0, 0.5, size=d)
    return NormCase(x, gamma, beta, g.uniform(2.0, 6.0) / 127, g.uniform(3.0, 8.0) / 127, eps)
