"""Integer-only relative-positional MHSA (I-Parakeet, Sec. 3.1) on GB300.

A thin Python binding over the C ABI of ``include/ip_mhsa.h``: argument
marshalling only.  Every step of the attention runs in the CUDA kernels of
``libipmhsa.so``; there is no CPU fallback, and a missing or unloadable
library raises :class:`LibraryError`.  PyTorch serves for device memory and
streams only.
"""
from __future__ import annotations

import ctypes
import threading
from dataclasses import dataclass

from . import build as _build

IP_DH = 128
IP_MAX_T = 2048

ERRORS = {
    0: "IP_OK", -1: "IP_ERR_NULL", -2: "IP_ERR_SHAPE", -3: "IP_ERR_ALIGN",
    -4: "IP_ERR_UNSUPPORTED", -5: "IP_ERR_CUDA", -6: "IP_ERR_TIMEOUT",
    -7: "IP_ERR_PARAM", -8: "IP_ERR_WORKSPACE",
}

EXPORTS = (
    "ip_relpos_mhsa_workspace_bytes", "ip_relpos_mhsa_i8", "ip_relpos_mhsa_status",
    "ip_relpos_mhsa_host_arena_bytes", "ip_relpos_mhsa_i8_host", "ip_strerror",
    "ip_debug_set_timeout_cycles", "ip_debug_set_stall_injection", "ip_dyadic_multiplier",
    "ip_dyadic_pair",
    "ip_isoftmax_params_from_scale", "ip_probe_int8_mma", "ip_relpos_mhsa_i8_noalloc",
    "ip_debug_set_split_mode", "ip_debug_set_wide_sums", "ip_linear_i8", "ip_linear_swish_i8", "ip_swish_params_from_scales",
    "ip_layernorm_i8", "ip_layernorm_constants", "ip_relpos_mhsa_i8_ex", "ip_residual_i8",
    "ip_residual_params", "ip_linear_glu_i8", "ip_glu_params", "ip_dwconv_swish_i8",
    "ip_swish16_params_from_scales", "ip_relpos_mhsa_i8_host_async", "ip_relpos_mhsa_host_status",
    "ip_set_workspace", "ip_probe_int8_mix", "ip_linear_residual_i8",
    "ip_relpos_layer_constants", "ip_linear_constants", "ip_relpos_mhsa_noalloc_status",
)

ROWS = 0    # IP_LAYOUT_ROWS:  [B][T][C]
HEADS = 1   # IP_LAYOUT_HEADS: [G][B][C/G/128][T][128]


class LibraryError(RuntimeError):
    """The GPU library could not be built or loaded."""


class IpError(RuntimeError):
    """A library call returned an IP_ERR_* code."""

    def __init__(self, fn: str, code: int, text: str):
        super().__init__(f"{fn}: {ERRORS.get(code, code)} ({text})")
        self.code = code


class SwishParams(ctypes.Structure):
    _fields_ = [("q_c", ctypes.c_int32), ("q_one", ctypes.c_int32), ("m", ctypes.c_int32),
                ("s", ctypes.c_int32)]


class Swish16Params(ctypes.Structure):
    _fields_ = [("q_c", ctypes.c_int32), ("q_one", ctypes.c_longlong), ("m", ctypes.c_int32),
                ("s", ctypes.c_int32)]


class SoftmaxParams(ctypes.Structure):
    _fields_ = [("q_ln2", ctypes.c_int32), ("q_b", ctypes.c_int32), ("q_c", ctypes.c_int32)]


_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile libipmhsa.so for sm_103a (nvcc) and return its path."""
    return _build.build(force=force)


def load(build_if_missing: bool = True) -> ctypes.CDLL:
    """Load libipmhsa.so and declare the C signatures."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        try:
            path = _build.build() if build_if_missing else _build.LIB
            lib = ctypes.CDLL(path)
        except Exception as exc:  # noqa: BLE001 - reported with context
            raise LibraryError(f"cannot build or load the GPU library: {exc}") from exc
        P = ctypes.c_void_p
        I = ctypes.c_int
        i32p = ctypes.POINTER(ctypes.c_int32)
        lib.ip_relpos_mhsa_workspace_bytes.argtypes = [I, I, I, I]
        lib.ip_relpos_mhsa_workspace_bytes.restype = ctypes.c_size_t
        lib.ip_relpos_mhsa_host_arena_bytes.argtypes = [I, I, I, I]
        lib.ip_relpos_mhsa_host_arena_bytes.restype = ctypes.c_size_t
        sig = [P] * 6 + [P, P, ctypes.POINTER(SoftmaxParams), P] + [I] * 4 + [P, P, ctypes.c_size_t, P]
        lib.ip_relpos_mhsa_i8.argtypes = sig
        lib.ip_relpos_mhsa_i8.restype = I
        lib.ip_relpos_mhsa_i8_host.argtypes = sig
        lib.ip_relpos_mhsa_i8_host.restype = I
        lib.ip_relpos_mhsa_i8_noalloc.argtypes = sig[:15] + [P]
        lib.ip_relpos_mhsa_i8_noalloc.restype = I
        lib.ip_relpos_mhsa_noalloc_status.argtypes = [P]
        lib.ip_relpos_mhsa_noalloc_status.restype = I
        lib.ip_relpos_mhsa_status.argtypes = [P, P]
        lib.ip_relpos_mhsa_status.restype = I
        lib.ip_set_workspace.argtypes = [P, ctypes.c_size_t]
        lib.ip_set_workspace.restype = I
        lib.ip_strerror.argtypes = [I]
        lib.ip_strerror.restype = ctypes.c_char_p
        lib.ip_debug_set_timeout_cycles.argtypes = [ctypes.c_longlong]
        lib.ip_debug_set_timeout_cycles.restype = I
        lib.ip_debug_set_stall_injection.argtypes = [I]
        lib.ip_debug_set_stall_injection.restype = I
        lib.ip_debug_set_split_mode.argtypes = [I]
        lib.ip_debug_set_split_mode.restype = I
        lib.ip_debug_set_wide_sums.argtypes = [I]
        lib.ip_debug_set_wide_sums.restype = I
        lib.ip_dyadic_multiplier.argtypes = [ctypes.c_double, i32p, i32p]
        lib.ip_dyadic_multiplier.restype = I
        lib.ip_dyadic_pair.argtypes = [ctypes.c_double, ctypes.c_double, i32p, i32p, i32p]
        lib.ip_dyadic_pair.restype = I
        lib.ip_isoftmax_params_from_scale.argtypes = [ctypes.c_double, ctypes.POINTER(SoftmaxParams)]
        lib.ip_isoftmax_params_from_scale.restype = I
        D_ = ctypes.c_double
        lib.ip_relpos_layer_constants.argtypes = [D_] * 6 + [I, P, P, ctypes.POINTER(SoftmaxParams)]
        lib.ip_relpos_layer_constants.restype = I
        lib.ip_linear_constants.argtypes = [D_, ctypes.POINTER(D_), ctypes.POINTER(D_), I,
                                            ctypes.POINTER(ctypes.c_int32),
                                            ctypes.POINTER(ctypes.c_int32)]
        lib.ip_linear_constants.restype = I
        lib.ip_relpos_mhsa_i8_ex.argtypes = [P] * 6 + [P, P, ctypes.POINTER(SoftmaxParams), P] + [
            I] * 4 + [P, I, P, ctypes.c_size_t, P]
        lib.ip_relpos_mhsa_i8_ex.restype = I
        lib.ip_relpos_mhsa_i8_host_async.argtypes = lib.ip_relpos_mhsa_i8_host.argtypes
        lib.ip_relpos_mhsa_i8_host_async.restype = I
        lib.ip_relpos_mhsa_host_status.argtypes = [P, I, I, I, I, P]
        lib.ip_relpos_mhsa_host_status.restype = I
        lib.ip_linear_i8.argtypes = [P, I, P, P, P, P, I, I, I, I, I, P, I, P, ctypes.c_size_t, P]
        lib.ip_linear_i8.restype = I
        lib.ip_linear_swish_i8.argtypes = [P, P, P, P, P, ctypes.POINTER(SwishParams), I, I, I, I,
                                           P, P, ctypes.c_size_t, P]
        lib.ip_linear_swish_i8.restype = I
        lib.ip_swish_params_from_scales.argtypes = [ctypes.c_double, ctypes.c_double,
                                                    ctypes.POINTER(SwishParams)]
        lib.ip_swish_params_from_scales.restype = I
        LL = ctypes.c_longlong
        lib.ip_layernorm_i8.argtypes = [P, LL, I, LL, P, P, P, P, P, ctypes.c_size_t, P]
        lib.ip_layernorm_i8.restype = I
        D = ctypes.c_double
        lib.ip_layernorm_constants.argtypes = [D, P, P, I, D, D, ctypes.POINTER(LL), P, P, P]
        lib.ip_layernorm_constants.restype = I
        i32p_ = ctypes.POINTER(ctypes.c_int32)
        lib.ip_residual_i8.argtypes = [P, P, ctypes.c_longlong, I, I, I, P, P]
        lib.ip_residual_i8.restype = I
        lib.ip_residual_params.argtypes = [D, D, D, D, i32p_, i32p_, i32p_]
        lib.ip_residual_params.restype = I
        lib.ip_linear_glu_i8.argtypes = [P, P, P, P, P, ctypes.POINTER(SwishParams), I, I, I, I, P,
                                         P, ctypes.c_size_t, P]
        lib.ip_linear_glu_i8.restype = I
        lib.ip_linear_residual_i8.argtypes = [P, P, P, P, P, P, I, I, I, I, I, I, I, P, P,
                                              ctypes.c_size_t, P]
        lib.ip_linear_residual_i8.restype = I
        lib.ip_glu_params.argtypes = [D, D, D, ctypes.POINTER(SwishParams)]
        lib.ip_glu_params.restype = I
        lib.ip_dwconv_swish_i8.argtypes = [P, I, I, I, P, I, P, P, P, ctypes.POINTER(Swish16Params),
                                           P, P, ctypes.c_size_t, P]
        lib.ip_dwconv_swish_i8.restype = I
        lib.ip_swish16_params_from_scales.argtypes = [D, D, ctypes.POINTER(Swish16Params)]
        lib.ip_swish16_params_from_scales.restype = I
        lib.ip_probe_int8_mma.argtypes = [I, I, P, P]
        lib.ip_probe_int8_mma.restype = ctypes.c_longlong
        lib.ip_probe_int8_mix.argtypes = [I, I, I, P, P]
        lib.ip_probe_int8_mix.restype = ctypes.c_longlong
        _lib = lib
        return lib


def strerror(code: int) -> str:
    return load().ip_strerror(code).decode()


def _check(fn: str, code: int):
    if code != 0:
        raise IpError(fn, code, strerror(code))


# ---------------------------------------------------------------- constants

@dataclass(frozen=True)
class LayerConstants:
    multipliers: tuple[int, int, int]   # m_c, m_p, m_o
    shifts: tuple[int, int]             # s_s, s_o (right shift 31 + s)
    softmax: tuple[int, int, int]       # q_ln2, q_b, q_c


def dyadic_multiplier(ratio: float) -> tuple[int, int]:
    m, s = ctypes.c_int32(), ctypes.c_int32()
    _check("ip_dyadic_multiplier", load().ip_dyadic_multiplier(ratio, ctypes.byref(m), ctypes.byref(s)))
    return m.value, s.value


def dyadic_pair(r_c: float, r_p: float) -> tuple[int, int, int]:
    a, b, s = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
    _check("ip_dyadic_pair", load().ip_dyadic_pair(r_c, r_p, ctypes.byref(a), ctypes.byref(b), ctypes.byref(s)))
    return a.value, b.value, s.value


def isoftmax_params_from_scale(S_s: float) -> tuple[int, int, int]:
    prm = SoftmaxParams()
    _check("ip_isoftmax_params_from_scale", load().ip_isoftmax_params_from_scale(S_s, ctypes.byref(prm)))
    return prm.q_ln2, prm.q_b, prm.q_c


def layer_constants(scales: dict, dh: int = IP_DH) -> LayerConstants:
    """Integer constants of one layer from its real scales S_Q, S_K, S_P,
    S_V, S_s, S_O (offline, Eq. 7 and Eq. 11), by ip_relpos_layer_constants."""
    mult = (ctypes.c_int32 * 3)()
    sh = (ctypes.c_int32 * 2)()
    sm = SoftmaxParams()
    _check("ip_relpos_layer_constants", load().ip_relpos_layer_constants(
        float(scales["S_Q"]), float(scales["S_K"]), float(scales["S_P"]), float(scales["S_V"]),
        float(scales["S_s"]), float(scales["S_O"]), int(dh), mult, sh, ctypes.byref(sm)))
    return LayerConstants(tuple(mult), tuple(sh), (sm.q_ln2, sm.q_b, sm.q_c))


# ---------------------------------------------------------------- device path

def workspace_bytes(B: int, H: int, T: int, dh: int = IP_DH) -> int:
    n = load().ip_relpos_mhsa_workspace_bytes(B, H, T, dh)
    if n == 0:
        raise IpError("ip_relpos_mhsa_workspace_bytes", -2, "invalid shape")
    return n


def host_arena_bytes(B: int, H: int, T: int, dh: int = IP_DH) -> int:
    n = load().ip_relpos_mhsa_host_arena_bytes(B, H, T, dh)
    if n == 0:
        raise IpError("ip_relpos_mhsa_host_arena_bytes", -2, "invalid shape")
    return n


def set_timeout_cycles(cycles: int) -> None:
    """Bound of every kernel barrier wait (clock cycles; negative: default)."""
    load().ip_debug_set_timeout_cycles(int(cycles))


def set_stall_injection(on: bool) -> None:
    """Test hook: make the kernels wait on a barrier nothing arrives on."""
    load().ip_debug_set_stall_injection(1 if on else 0)


def set_split_mode(mode: int) -> None:
    """Test hook: -1 planned tail split (default), 0 never split, 1 split
    every 64-row tile into two key-split halves, 2 into four key-split
    quarters."""
    load().ip_debug_set_split_mode(int(mode))


def set_wide_sums(on: bool) -> None:
    """Test hook: always take the general softmax arithmetic (64-bit partial
    row sums, probabilities from the full 64-bit product); False: the fast
    paths where the host has shown they give the same integers."""
    load().ip_debug_set_wide_sums(1 if on else 0)


def _arr(vals, ctype):
    return (ctype * len(vals))(*vals)


def _stream_handle(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dev_ptr(t, name, dtype, shape):
    import torch
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def relpos_mhsa_i8(q, k, v, p, u, v_bias, consts: LayerConstants, lengths=None, out=None,
                   workspace=None, stream=None, out_layout: int = HEADS):
    """Whole layer on the GPU.  q, k, v: int8 [B, H, T, 128] CUDA tensors;
    p: int8 [H, 2T-1, 128]; u, v_bias: int8 [H, 128]; lengths: int32 [B]
    CUDA tensor or None.  Returns out: int8 [B, H, T, 128] (HEADS) or
    [B, T, H, 128] (ROWS, the frames' rows of the output projection).
    Asynchronous on `stream` (default: torch's current stream)."""
    import torch
    B, H, T, dh = q.shape
    shp = (B, H, T, dh)
    oshp = shp if out_layout == HEADS else (B, T, H, dh)
    args = [_dev_ptr(q, "q", torch.int8, shp), _dev_ptr(k, "k", torch.int8, shp),
            _dev_ptr(v, "v", torch.int8, shp), _dev_ptr(p, "p", torch.int8, (H, 2 * T - 1, dh)),
            _dev_ptr(u, "u", torch.int8, (H, dh)), _dev_ptr(v_bias, "v_bias", torch.int8, (H, dh))]
    if out is None:
        out = torch.empty(oshp, dtype=torch.int8, device=q.device)
    lens = None if lengths is None else _dev_ptr(lengths, "lengths", torch.int32, (B,))
    if workspace is None and _default_workspace is None:
        workspace = torch.zeros(workspace_bytes(B, H, T, dh), dtype=torch.uint8, device=q.device)
    # workspace None here: the library uses the registered default workspace
    ws_ptr = None if workspace is None else ctypes.c_void_p(workspace.data_ptr())
    ws_len = 0 if workspace is None else workspace.numel()
    sm = SoftmaxParams(*consts.softmax)
    rc = load().ip_relpos_mhsa_i8_ex(
        *args, _arr(consts.multipliers, ctypes.c_int32), _arr(consts.shifts, ctypes.c_int32),
        ctypes.byref(sm), lens, B, H, T, dh, _dev_ptr(out, "out", torch.int8, oshp), out_layout,
        ws_ptr, ws_len, _stream_handle(stream))
    _check("ip_relpos_mhsa_i8_ex", rc)
    return out


def int8_mma_peak_tops(iters: int = 4096, repeats: int = 3) -> float:
    """Measured integer warp-MMA throughput of the current GPU in TOPS
    (best of `repeats` timed launches, CUDA events on the launching stream)."""
    import torch
    props = torch.cuda.get_device_properties(torch.cuda.current_device())
    blocks = props.multi_processor_count * 8
    sink = torch.empty(blocks * 256, dtype=torch.int32, device="cuda")
    st = torch.cuda.current_stream()
    lib = load()
    h = ctypes.c_void_p(st.cuda_stream)
    lib.ip_probe_int8_mma(blocks, iters, ctypes.c_void_p(sink.data_ptr()), h)   # warm-up
    best = 0.0
    for _ in range(repeats):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(st)
        ops = lib.ip_probe_int8_mma(blocks, iters, ctypes.c_void_p(sink.data_ptr()), h)
        e1.record(st)
        e1.synchronize()
        if ops < 0:
            raise IpError("ip_probe_int8_mma", -5, "launch failed")
        best = max(best, ops / (e0.elapsed_time(e1) * 1e-3) / 1e12)
    return best


def int8_pipe_rates(iters: int = 2048, repeats: int = 3) -> dict:
    """Measured integer throughput (TOPS, best of `repeats` launches, CUDA
    events) of the integer MMA pipe alone, the dp4a pipe alone, and both at
    once (half the warps on each)."""
    import torch
    props = torch.cuda.get_device_properties(torch.cuda.current_device())
    blocks = props.multi_processor_count * 2
    sink = torch.empty(blocks * 256, dtype=torch.int32, device="cuda")
    st = torch.cuda.current_stream()
    lib = load()
    h = ctypes.c_void_p(st.cuda_stream)
    out = {}
    for name, mw in (("imma", 8), ("dp4a", 0), ("imma_plus_dp4a", 4)):
        lib.ip_probe_int8_mix(blocks, iters, mw, ctypes.c_void_p(sink.data_ptr()), h)   # warm-up
        best = 0.0
        for _ in range(repeats):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(st)
            ops = lib.ip_probe_int8_mix(blocks, iters, mw, ctypes.c_void_p(sink.data_ptr()), h)
            e1.record(st)
            e1.synchronize()
            if ops < 0:
                raise IpError("ip_probe_int8_mix", -5, "launch failed")
            best = max(best, ops / (e0.elapsed_time(e1) * 1e-3) / 1e12)
        out[name] = best
    return out


def status(workspace=None, stream=None) -> int:
    """Synchronises the stream and returns the device-side status code of
    the last call that used `workspace` (0 = ok); None: the default
    workspace registered by set_workspace."""
    ptr = None if workspace is None else ctypes.c_void_p(workspace.data_ptr())
    return load().ip_relpos_mhsa_status(ptr, _stream_handle(stream))


def noalloc_status(stream=None) -> int:
    """Synchronises the stream and returns the device-side status code of
    the ip_relpos_mhsa_i8_noalloc calls on the current device since the
    last read (0 = ok), clearing it."""
    return load().ip_relpos_mhsa_noalloc_status(_stream_handle(stream))


_default_workspace = None


def set_workspace(workspace) -> None:
    """Registers `workspace` (a zero-filled uint8 CUDA tensor of at least
    workspace_bytes(...) bytes) as the default of the attention calls that
    pass none; None releases it.  The binding keeps the tensor alive while
    it is registered.  Calls that share it must run on one stream."""
    global _default_workspace
    if workspace is None:
        _check("ip_set_workspace", load().ip_set_workspace(None, 0))
        _default_workspace = None
        return
    import torch
    if not (isinstance(workspace, torch.Tensor) and workspace.is_cuda and
            workspace.dtype == torch.uint8 and workspace.is_contiguous()):
        raise TypeError("workspace: a contiguous uint8 CUDA tensor")
    _check("ip_set_workspace", load().ip_set_workspace(ctypes.c_void_p(workspace.data_ptr()),
                                                       workspace.numel()))
    _default_workspace = workspace


def linear_constants(s_x: float, s_w, s_y):
    """Per-output-channel constants of Eq. 7 (offline), by
    ip_linear_constants: int32 arrays m, s of the length of s_w (s_y: one
    grid per channel, or one for all)."""
    import numpy as np
    s_w = np.ascontiguousarray(s_w, dtype=np.float64).reshape(-1)
    s_y = np.ascontiguousarray(np.broadcast_to(np.asarray(s_y, dtype=np.float64).reshape(-1)
                                               if np.ndim(s_y) else np.float64(s_y), s_w.shape))
    m = np.empty(s_w.shape, dtype=np.int32)
    s = np.empty(s_w.shape, dtype=np.int32)
    dp = ctypes.POINTER(ctypes.c_double)
    ip32 = ctypes.POINTER(ctypes.c_int32)
    _check("ip_linear_constants", load().ip_linear_constants(
        float(s_x), s_w.ctypes.data_as(dp), s_y.ctypes.data_as(dp), int(s_w.size),
        m.ctypes.data_as(ip32), s.ctypes.data_as(ip32)))
    return m, s


def linear_i8(x, w, bias, m, s, *, x_layout: int = ROWS, y_layout: int = ROWS, groups: int = 1,
              out=None, workspace=None, stream=None):
    """Integer linear layer (Eqs. 6-7) on the GPU.  x: int8 [B, T, K] (ROWS)
    or [B, K/128, T, 128] (HEADS); w: int8 [N, K]; bias: int32 [N] or None;
    m, s: int32 [N] (per output channel); all CUDA tensors.  Returns out:
    int8 [B, T, N] (ROWS) or [G, B, N/G/128, T, 128] (HEADS).  Asynchronous
    on `stream` (default: torch's current stream)."""
    import torch
    N, K = w.shape
    if x_layout == ROWS:
        B, T, _ = x.shape
        xs = (B, T, K)
    else:
        B, _, T, _ = x.shape
        xs = (B, K // 128, T, 128)
    ys = (B, T, N) if y_layout == ROWS else (groups, B, N // max(groups, 1) // 128, T, 128)
    if out is None:
        out = torch.empty(ys, dtype=torch.int8, device=w.device)
    if workspace is None:
        workspace = torch.zeros(256, dtype=torch.uint8, device=w.device)
    bp = None if bias is None else _dev_ptr(bias, "bias", torch.int32, (N,))
    rc = load().ip_linear_i8(
        _dev_ptr(x, "x", torch.int8, xs), x_layout, _dev_ptr(w, "w", torch.int8, (N, K)), bp,
        _dev_ptr(m, "m", torch.int32, (N,)), _dev_ptr(s, "s", torch.int32, (N,)), B, T, K, N,
        groups, _dev_ptr(out, "out", torch.int8, ys), y_layout,
        ctypes.c_void_p(workspace.data_ptr()), workspace.numel(), _stream_handle(stream))
    _check("ip_linear_i8", rc)
    return out


def linear_residual_i8(x, w, bias, m, s, res, m_x: int, m_y: int, s_r: int, *, out=None,
                       workspace=None, stream=None):
    """Integer linear layer with the residual addition of its output fused:
    out = residual(res, linear(x)) with (m_x, m_y, s_r) from residual_params.
    x: int8 [B, T, K]; w: int8 [N, K]; bias, m, s as linear_i8; res: int8
    [B, T, N] (not aliasing out); all CUDA tensors, row-major."""
    import torch
    N, K = w.shape
    B, T, _ = x.shape
    if out is None:
        out = torch.empty((B, T, N), dtype=torch.int8, device=w.device)
    if workspace is None:
        workspace = torch.zeros(256, dtype=torch.uint8, device=w.device)
    bp = None if bias is None else _dev_ptr(bias, "bias", torch.int32, (N,))
    rc = load().ip_linear_residual_i8(
        _dev_ptr(x, "x", torch.int8, (B, T, K)), _dev_ptr(w, "w", torch.int8, (N, K)), bp,
        _dev_ptr(m, "m", torch.int32, (N,)), _dev_ptr(s, "s", torch.int32, (N,)),
        _dev_ptr(res, "res", torch.int8, (B, T, N)), int(m_x), int(m_y), int(s_r), B, T, K, N,
        _dev_ptr(out, "out", torch.int8, (B, T, N)), ctypes.c_void_p(workspace.data_ptr()),
        workspace.numel(), _stream_handle(stream))
    _check("ip_linear_residual_i8", rc)
    return out


def swish_params_from_scales(S_z: float, S_y: float) -> tuple[int, int, int, int]:
    """Integer constants (q_c, q_one, m, s) of the minimax Swish for an int8
    input on grid S_z and an int8 output on grid S_y (Eqs. 12-13)."""
    prm = SwishParams()
    _check("ip_swish_params_from_scales",
           load().ip_swish_params_from_scales(S_z, S_y, ctypes.byref(prm)))
    return prm.q_c, prm.q_one, prm.m, prm.s


def linear_swish_i8(x, w, bias, m, s, swish: tuple[int, int, int, int], *, out=None,
                    workspace=None, stream=None):
    """Feed-forward projection with the fused minimax Swish: x int8 [B, T, K],
    w int8 [N, K], bias int32 [N] or None, m, s int32 [N] (onto the Swish
    input grid), swish = (q_c, q_one, m, s).  Returns int8 [B, T, N]."""
    import torch
    N, K = w.shape
    B, T, _ = x.shape
    if out is None:
        out = torch.empty((B, T, N), dtype=torch.int8, device=w.device)
    if workspace is None:
        workspace = torch.zeros(256, dtype=torch.uint8, device=w.device)
    bp = None if bias is None else _dev_ptr(bias, "bias", torch.int32, (N,))
    sw = SwishParams(*swish)
    rc = load().ip_linear_swish_i8(
        _dev_ptr(x, "x", torch.int8, (B, T, K)), _dev_ptr(w, "w", torch.int8, (N, K)), bp,
        _dev_ptr(m, "m", torch.int32, (N,)), _dev_ptr(s, "s", torch.int32, (N,)), ctypes.byref(sw),
        B, T, K, N, _dev_ptr(out, "out", torch.int8, (B, T, N)),
        ctypes.c_void_p(workspace.data_ptr()), workspace.numel(), _stream_handle(stream))
    _check("ip_linear_swish_i8", rc)
    return out


@dataclass(frozen=True)
class NormConstants:
    eps_c: int
    M: "np.ndarray"     # int32 [d]
    B: "np.ndarray"     # int64 [d]
    E: "np.ndarray"     # int32 [d]


def layernorm_constants(s_x: float, gamma, beta, s_y: float, eps: float = 1e-5) -> NormConstants:
    """Offline constants of the integer LayerNorm (host, float64)."""
    import numpy as np
    g = np.ascontiguousarray(gamma, dtype=np.float64)
    b = np.ascontiguousarray(beta, dtype=np.float64)
    d = g.size
    M = np.empty(d, np.int32)
    B = np.empty(d, np.int64)
    E = np.empty(d, np.int32)
    ec = ctypes.c_longlong()
    _check("ip_layernorm_constants", load().ip_layernorm_constants(
        s_x, g.ctypes.data, b.ctypes.data, d, s_y, eps, ctypes.byref(ec), M.ctypes.data,
        B.ctypes.data, E.ctypes.data))
    return NormConstants(ec.value, M, B, E)


def layernorm_i8(x, M, B, E, eps_c: int, *, out=None, workspace=None, stream=None):
    """Integer LayerNorm over the last axis of int8 x (CUDA, d in {512, 1024,
    1536, 2048}); M int32, B int64, E int32 [d] CUDA tensors.  Returns int8
    like x.  Asynchronous on `stream`."""
    import torch
    d = x.shape[-1]
    rows = x.numel() // d if d else 0
    if out is None:
        out = torch.empty_like(x)
    if workspace is None:
        workspace = torch.zeros(256, dtype=torch.uint8, device=x.device)
    rc = load().ip_layernorm_i8(
        _dev_ptr(x, "x", torch.int8, tuple(x.shape)), rows, d, int(eps_c),
        _dev_ptr(M, "M", torch.int32, (d,)), _dev_ptr(B, "B", torch.int64, (d,)),
        _dev_ptr(E, "E", torch.int32, (d,)), _dev_ptr(out, "out", torch.int8, tuple(x.shape)),
        ctypes.c_void_p(workspace.data_ptr()), workspace.numel(), _stream_handle(stream))
    _check("ip_layernorm_i8", rc)
    return out


def residual_params(s_x: float, s_y: float, s_z: float, alpha: float = 1.0):
    """(m_x, m_y, s) of z = x + alpha y onto S_z (Eqs. 1-4)."""
    a, b, s = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
    _check("ip_residual_params", load().ip_residual_params(s_x, s_y, s_z, alpha, ctypes.byref(a),
                                                          ctypes.byref(b), ctypes.byref(s)))
    return a.value, b.value, s.value


def residual_i8(x, y, m_x: int, m_y: int, s: int, *, out=None, stream=None):
    """Residual addition of two int8 CUDA tensors of one shape."""
    import torch
    if out is None:
        out = torch.empty_like(x)
    n = x.numel()
    rc = load().ip_residual_i8(_dev_ptr(x, "x", torch.int8, tuple(x.shape)),
                               _dev_ptr(y, "y", torch.int8, tuple(x.shape)), n, m_x, m_y, s,
                               _dev_ptr(out, "out", torch.int8, tuple(x.shape)),
                               _stream_handle(stream))
    _check("ip_residual_i8", rc)
    return out


def glu_params(s_a: float, s_b: float, s_y: float) -> tuple[int, int, int, int]:
    """(q_c, q_one, m, s) of GLU(a, b) = a sigma(b) (Eq. 5, minimax tanh)."""
    prm = SwishParams()
    _check("ip_glu_params", load().ip_glu_params(s_a, s_b, s_y, ctypes.byref(prm)))
    return prm.q_c, prm.q_one, prm.m, prm.s


def linear_glu_i8(x, w_interleaved, bias, m, s, glu: tuple[int, int, int, int], *, out=None,
                  workspace=None, stream=None):
    """Pointwise convolution with the GLU fused: x int8 [B, T, K]; w int8 [N, K]
    with rows (a_c, b_c) interleaved; bias, m, s int32 [N]; returns int8
    [B, T, N/2]."""
    import torch
    N, K = w_interleaved.shape
    B, T, _ = x.shape
    if out is None:
        out = torch.empty((B, T, N // 2), dtype=torch.int8, device=x.device)
    if workspace is None:
        workspace = torch.zeros(256, dtype=torch.uint8, device=x.device)
    bp = None if bias is None else _dev_ptr(bias, "bias", torch.int32, (N,))
    g = SwishParams(*glu)
    rc = load().ip_linear_glu_i8(
        _dev_ptr(x, "x", torch.int8, (B, T, K)), _dev_ptr(w_interleaved, "w", torch.int8, (N, K)), bp,
        _dev_ptr(m, "m", torch.int32, (N,)), _dev_ptr(s, "s", torch.int32, (N,)), ctypes.byref(g),
        B, T, K, N, _dev_ptr(out, "out", torch.int8, (B, T, N // 2)),
        ctypes.c_void_p(workspace.data_ptr()), workspace.numel(), _stream_handle(stream))
    _check("ip_linear_glu_i8", rc)
    return out


def swish16_params(s_z: float, s_y: float) -> tuple[int, int, int, int]:
    """(q_c, q_one, m, s) of the Swish of an INT16 input grid."""
    prm = Swish16Params()
    _check("ip_swish16_params_from_scales",
           load().ip_swish16_params_from_scales(s_z, s_y, ctypes.byref(prm)))
    return prm.q_c, prm.q_one, prm.m, prm.s


def dwconv_swish_i8(x, w, bias, m, s, sw16: tuple[int, int, int, int], *, out=None,
                    workspace=None, stream=None):
    """Depthwise convolution over time (folded BatchNorm, INT16) + Swish:
    x int8 [B, T, C]; w int8 [C, K]; bias, m, s int32 [C]; returns int8
    [B, T, C]."""
    import torch
    B, T, C = x.shape
    K = w.shape[1]
    if out is None:
        out = torch.empty_like(x)
    if workspace is None:
        workspace = torch.zeros(256, dtype=torch.uint8, device=x.device)
    p = Swish16Params(*sw16)
    rc = load().ip_dwconv_swish_i8(
        _dev_ptr(x, "x", torch.int8, (B, T, C)), B, T, C, _dev_ptr(w, "w", torch.int8, (C, K)), K,
        _dev_ptr(bias, "bias", torch.int32, (C,)), _dev_ptr(m, "m", torch.int32, (C,)),
        _dev_ptr(s, "s", torch.int32, (C,)), ctypes.byref(p),
        _dev_ptr(out, "out", torch.int8, (B, T, C)), ctypes.c_void_p(workspace.data_ptr()),
        workspace.numel(), _stream_handle(stream))
    _check("ip_dwconv_swish_i8", rc)
    return out


def relpos_mhsa_i8_host(q, k, v, p, u, v_bias, consts: LayerConstants, lengths, out, arena,
                        stream=None, wait: bool = True):
    """Whole layer from host buffers (torch CPU tensors, ideally pinned):
    copies in, runs, copies the result into `out` and synchronises.  With
    wait=False the call only enqueues (ip_relpos_mhsa_i8_host_async): `out`
    is valid after the stream synchronises, and host_status() reports
    errors."""
    import torch
    B, H, T, dh = q.shape
    for name, t in (("q", q), ("k", k), ("v", v), ("p", p), ("u", u), ("v_bias", v_bias), ("out", out)):
        if t.is_cuda or t.dtype != torch.int8 or not t.is_contiguous():
            raise TypeError(f"{name} must be a contiguous int8 CPU tensor")
    lens = None
    if lengths is not None:
        if lengths.is_cuda or lengths.dtype != torch.int32 or tuple(lengths.shape) != (B,):
            raise TypeError("lengths must be an int32 [B] CPU tensor")
        lens = ctypes.c_void_p(lengths.data_ptr())
    sm = SoftmaxParams(*consts.softmax)
    ptr = lambda t: ctypes.c_void_p(t.data_ptr())
    fn = load().ip_relpos_mhsa_i8_host if wait else load().ip_relpos_mhsa_i8_host_async
    rc = fn(ptr(q), ptr(k), ptr(v), ptr(p), ptr(u), ptr(v_bias),
            _arr(consts.multipliers, ctypes.c_int32), _arr(consts.shifts, ctypes.c_int32),
            ctypes.byref(sm), lens, B, H, T, dh, ptr(out), ctypes.c_void_p(arena.data_ptr()),
            arena.numel(), _stream_handle(stream))
    _check("ip_relpos_mhsa_i8_host" if wait else "ip_relpos_mhsa_i8_host_async", rc)
    return out


def host_status(arena, B: int, H: int, T: int, dh: int = IP_DH, stream=None) -> int:
    """Synchronises `stream` and returns the status of the last asynchronous
    host-buffer call that used `arena` (0 = ok)."""
    return load().ip_relpos_mhsa_host_status(ctypes.c_void_p(arena.data_ptr()), B, H, T, dh,
                                             _stream_handle(stream))


__all__ = ["build", "load", "relpos_mhsa_i8", "relpos_mhsa_i8_host", "status", "workspace_bytes",
           "host_arena_bytes", "layer_constants", "LayerConstants", "dyadic_multiplier",
           "dyadic_pair", "isoftmax_params_from_scale", "set_timeout_cycles", "strerror",
           "int8_mma_peak_tops", "set_stall_injection", "set_split_mode", "linear_i8",
           "linear_constants", "ROWS", "HEADS", "linear_swish_i8", "swish_params_from_scales",
           "layernorm_i8", "layernorm_constants", "NormConstants", "residual_i8",
           "residual_params", "linear_glu_i8", "glu_params", "dwconv_swish_i8", "swish16_params",
           "host_status", "set_workspace", "int8_pipe_rates", "linear_residual_i8",
           "IpError", "LibraryError", "EXPORTS"]
