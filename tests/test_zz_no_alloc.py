"""The entry point that allocates nothing (ip_relpos_mhsa_i8_noalloc).

It serves callers that cannot allocate device memory - a plugin whose host
framework owns the device pool and passes only inputs and outputs, or a
latency-critical path where an allocation may not happen.  Its scratch (the
device status word) is a file-scope device array inside the library.  This
test calls it through the C ABI twice in a row and checks that both calls
give exactly the output of ip_relpos_mhsa_i8, the entry point that takes a
caller-owned workspace (integer path: the tolerance is bit-exactness), and
issues two calls back to back on one stream with no synchronisation between
them, which is where the shared scratch is reused.  A barrier wait that runs
out inside such a call (the stall-injection hook with a short bound) is read
back by ip_relpos_mhsa_noalloc_status.  It lives in a file of its own that
pytest collects last.
"""
import ctypes

import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr())


@pytest.mark.parametrize("masked", [False, True])
def test_noalloc_matches_workspace_entry_point(masked):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30846_gb300 as ip
    lib = ip.load()
    B, H, T, dh = 3, 8, 150, 128
    lens = np.array([150, 97, 1], np.int32) if masked else None
    cases = [synth.draw(B, H, T, dh, seed=8100 + i + 10 * masked, p_mode="sinusoid",
                        lengths=lens) for i in range(2)]
    stream = torch.cuda.current_stream()
    for lay in cases:      # two calls in a row, each against the workspace path
        c = ip.layer_constants(lay.scales)
        dev = {n: torch.from_numpy(np.ascontiguousarray(getattr(lay, n))).cuda()
               for n in ("q", "k", "v", "p", "u", "vb")}
        dlen = None if lens is None else torch.from_numpy(lens).cuda()
        ws = torch.zeros(ip.workspace_bytes(B, H, T), dtype=torch.uint8, device="cuda")
        want = ip.relpos_mhsa_i8(dev["q"], dev["k"], dev["v"], dev["p"], dev["u"], dev["vb"], c,
                                 lengths=dlen, workspace=ws)
        assert ip.status(ws) == 0
        got = torch.full((B, H, T, dh), 99, dtype=torch.int8, device="cuda")
        sm = ip.SoftmaxParams(*c.softmax)
        rc = lib.ip_relpos_mhsa_i8_noalloc(
            _ptr(dev["q"]), _ptr(dev["k"]), _ptr(dev["v"]), _ptr(dev["p"]), _ptr(dev["u"]),
            _ptr(dev["vb"]), (ctypes.c_int32 * 3)(*c.multipliers),
            (ctypes.c_int32 * 2)(*c.shifts), ctypes.byref(sm),
            None if dlen is None else _ptr(dlen), B, H, T, dh, _ptr(got),
            ctypes.c_void_p(stream.cuda_stream))
        assert rc == 0, ip.strerror(rc)
        assert ip.noalloc_status() == 0
        np.testing.assert_array_equal(got.cpu().numpy(), want.cpu().numpy())


def _noalloc_call(lib, ip, dev, c, dlen, shape, out, stream):
    B, H, T, dh = shape
    sm = ip.SoftmaxParams(*c.softmax)
    rc = lib.ip_relpos_mhsa_i8_noalloc(
        _ptr(dev["q"]), _ptr(dev["k"]), _ptr(dev["v"]), _ptr(dev["p"]), _ptr(dev["u"]),
        _ptr(dev["vb"]), (ctypes.c_int32 * 3)(*c.multipliers), (ctypes.c_int32 * 2)(*c.shifts),
        ctypes.byref(sm), None if dlen is None else _ptr(dlen), B, H, T, dh, _ptr(out),
        ctypes.c_void_p(stream.cuda_stream))
    assert rc == 0, ip.strerror(rc)


def test_noalloc_calls_back_to_back_in_stream_order():
    # Two calls on one stream with no synchronisation between them: the
    # second call clears the shared scratch (the kernel's status word and work
    # counters) in stream order after the first call's kernel, on another
    # shape and with a key-padding mask.  One synchronisation at the end;
    # both outputs equal the workspace entry point's.
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30846_gb300 as ip
    lib = ip.load()
    shapes = [(3, 8, 150, 128), (2, 8, 97, 128)]
    lens = [None, np.array([97, 40], np.int32)]
    stream = torch.cuda.current_stream()
    todo = []
    for i, ((B, H, T, dh), ln) in enumerate(zip(shapes, lens)):
        lay = synth.draw(B, H, T, dh, seed=8200 + i, p_mode="sinusoid", lengths=ln)
        c = ip.layer_constants(lay.scales)
        dev = {n: torch.from_numpy(np.ascontiguousarray(getattr(lay, n))).cuda()
               for n in ("q", "k", "v", "p", "u", "vb")}
        dlen = None if ln is None else torch.from_numpy(ln).cuda()
        ws = torch.zeros(ip.workspace_bytes(B, H, T), dtype=torch.uint8, device="cuda")
        want = ip.relpos_mhsa_i8(dev["q"], dev["k"], dev["v"], dev["p"], dev["u"], dev["vb"], c,
                                 lengths=dlen, workspace=ws)
        assert ip.status(ws) == 0
        got = torch.full((B, H, T, dh), 99, dtype=torch.int8, device="cuda")
        todo.append((dev, c, dlen, (B, H, T, dh), got, want))
    torch.cuda.synchronize()
    for dev, c, dlen, shape, got, _ in todo:      # back to back, no sync between
        _noalloc_call(lib, ip, dev, c, dlen, shape, got, stream)
    assert ip.noalloc_status() == 0
    for _, _, _, _, got, want in todo:
        np.testing.assert_array_equal(got.cpu().numpy(), want.cpu().numpy())


def test_noalloc_reports_barrier_timeout():
    # every consumer warp first waits on a barrier nobody arrives on, with a
    # bound of about a millisecond: the wait runs out, the kernel records
    # IP_ERR_TIMEOUT in the library's scratch word and returns; the status
    # reader reports it once and clears it, and the next call is exact
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import oracle
    import paper_2609_30846_gb300 as ip
    lib = ip.load()
    B, H, T, dh = 2, 8, 200, 128
    lay = synth.draw(B, H, T, dh, seed=8301, p_mode="sinusoid")
    c = ip.layer_constants(lay.scales)
    dev = {n: torch.from_numpy(np.ascontiguousarray(getattr(lay, n))).cuda()
           for n in ("q", "k", "v", "p", "u", "vb")}
    out = torch.zeros((B, H, T, dh), dtype=torch.int8, device="cuda")
    stream = torch.cuda.current_stream()
    assert ip.noalloc_status() == 0
    try:
        ip.set_timeout_cycles(2_000_000)
        ip.set_stall_injection(True)
        _noalloc_call(lib, ip, dev, c, None, (B, H, T, dh), out, stream)
        assert ip.noalloc_status() == -6     # IP_ERR_TIMEOUT, read and cleared
        assert ip.noalloc_status() == 0
    finally:
        ip.set_stall_injection(False)
        ip.set_timeout_cycles(-1)
    _noalloc_call(lib, ip, dev, c, None, (B, H, T, dh), out, stream)
    assert ip.noalloc_status() == 0
    want = oracle.relpos_mhsa(lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb,
                              oracle.layer_constants(lay.scales, 128))
    np.testing.assert_array_equal(out.cpu().numpy(), want)


def test_noalloc_rejects_bad_shapes():
    import paper_2609_30846_gb300 as ip
    lib = ip.load()
    args = [None] * 6 + [None, None, None, None]
    assert lib.ip_relpos_mhsa_i8_noalloc(*args, 1, 8, ip.IP_MAX_T + 1, 128, None, None) == -2
    assert lib.ip_relpos_mhsa_i8_noalloc(*args, 1, 8, 10, 64, None, None) == -4
