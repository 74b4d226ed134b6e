"""Parity of the CUDA path (through the C ABI) with the CPU oracle.

Integer work: the bar is bit-exactness on every output.  Inputs come from
the seeded generator; the oracle's expected values come from the oracle
only.
"""
import numpy as np
import pytest

import synth
from guard import Guarded

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def ip():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30846_gb300 as mod
    mod.load()
    return mod


@pytest.fixture(scope="module")
def orc():
    import oracle
    oracle.build()
    return oracle


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def run_gpu(ip, lay, consts, lengths=None):
    B, H, T, dh = lay.q.shape
    ws = torch.zeros(ip.workspace_bytes(B, H, T, dh), dtype=torch.uint8, device="cuda")
    lens = None if lengths is None else _dev(lengths.astype(np.int32))
    g = Guarded((B, H, T, dh), torch.int8)
    out = ip.relpos_mhsa_i8(_dev(lay.q), _dev(lay.k), _dev(lay.v), _dev(lay.p), _dev(lay.u),
                            _dev(lay.vb), consts, lengths=lens, out=g.view, workspace=ws)
    assert ip.status(ws) == 0
    g.check()
    return out.cpu().numpy()


def oracle_out(orc, lay, consts, lengths=None):
    c = orc.LayerConstants(consts.multipliers, consts.shifts, consts.softmax)
    return orc.relpos_mhsa(lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb, c, lengths)


def assert_same(got, want):
    bad = got != want
    if bad.any():
        idx = np.argwhere(bad)[:5]
        raise AssertionError(f"{int(bad.sum())} of {got.size} outputs differ; first at {idx.tolist()}: "
                             f"gpu {got[tuple(idx[0])]} oracle {want[tuple(idx[0])]}")


@pytest.mark.parametrize("w", [0, 1, 2, 4])
def test_workload_full_size(ip, orc, w):
    lay = synth.layer(w, 0)
    c = ip.layer_constants(lay.scales)
    assert_same(run_gpu(ip, lay, c, lay.lengths), oracle_out(orc, lay, c, lay.lengths))


def test_encoder_layer_full_size(ip, orc):
    # one layer of the 24-layer encoder sweep (B=32, T=375), every output
    lay = synth.layer(3, 5)
    c = ip.layer_constants(lay.scales)
    assert_same(run_gpu(ip, lay, c), oracle_out(orc, lay, c))


@pytest.mark.parametrize("T", [1, 2, 3, 17, 63, 64, 65, 100, 127, 128, 129, 191, 200])
def test_ragged_lengths_of_T(ip, orc, T):
    lay = synth.draw(2, 3, T, 128, seed=500 + T, p_mode="sinusoid")
    c = ip.layer_constants(lay.scales)
    assert_same(run_gpu(ip, lay, c), oracle_out(orc, lay, c))


@pytest.mark.parametrize("seed", range(3))
def test_key_padding_masks(ip, orc, seed):
    T = 150
    rng = np.random.default_rng(seed)
    lens = np.array([0, 1, 2, 63, 64, 65, 149, 150, 999, -4] + list(rng.integers(0, T + 1, 6)), np.int32)
    lay = synth.draw(len(lens), 2, T, 128, seed=900 + seed, lengths=lens)
    c = ip.layer_constants(lay.scales)
    assert_same(run_gpu(ip, lay, c, lens), oracle_out(orc, lay, c, lens))


def test_extreme_values_and_constants(ip, orc):
    B, H, T = 2, 2, 96
    rng = np.random.default_rng(7)
    base = synth.draw(B, H, T, 128, seed=31)
    for lo, hi in ((-128, 127), (-128, -127), (126, 127)):
        q = rng.integers(lo, hi + 1, size=base.q.shape).astype(np.int8)
        k = rng.integers(lo, hi + 1, size=base.q.shape).astype(np.int8)
        v = rng.integers(-128, 128, size=base.q.shape).astype(np.int8)
        p = rng.integers(lo, hi + 1, size=base.p.shape).astype(np.int8)
        u = rng.integers(lo, hi + 1, size=base.u.shape).astype(np.int8)
        vb = rng.integers(lo, hi + 1, size=base.vb.shape).astype(np.int8)
        lay = synth.Layer(q, k, v, p, u, vb, None, base.scales)
        for mult, shifts, sm in (((2 ** 31 - 1, 2 ** 31 - 1, 2 ** 31 - 1), (0, 0), (3, 6, 10)),
                                 ((2 ** 31 - 1, 12345, 2 ** 30), (31, 31), (100, 195, 20000)),
                                 ((0, 2 ** 30, 1), (20, 8), (12, 24, 327)),
                                 ((2 ** 30, 0, 2 ** 31 - 1), (12, 0), (1, 2, 0))):
            c = ip.LayerConstants(mult, shifts, sm)
            assert_same(run_gpu(ip, lay, c), oracle_out(orc, lay, c))


def test_uniform_scores(ip, orc):
    # all keys equal: every probability is the same closed-form value
    B, H, T = 1, 2, 300
    lay = synth.draw(B, H, T, 128, seed=3)
    lay.k[:] = 0
    lay.p[:] = 0
    c = ip.layer_constants(lay.scales)
    assert_same(run_gpu(ip, lay, c), oracle_out(orc, lay, c))


def test_longest_sequence(ip, orc):
    T = ip.IP_MAX_T
    lay = synth.draw(1, 2, T, 128, seed=77, dist="t3", p_mode="random")
    c = ip.layer_constants(lay.scales)
    assert_same(run_gpu(ip, lay, c), oracle_out(orc, lay, c))


@pytest.mark.parametrize("T,masked", [(450, False), (520, True), (1100, False)])
def test_long_sequences_in_both_score_modes(ip, orc, T, masked):
    # Beyond 384 frames the int8 scores move to the workspace when it holds
    # their region (ip_relpos_mhsa_workspace_bytes counts it): two CTAs per
    # SM instead of one.  With only the 256-byte status workspace the kernel
    # keeps them in shared memory.  Both equal the oracle.
    B, H = 2, 3
    lens = np.array([T, T // 2 + 7], np.int32) if masked else None
    lay = synth.draw(B, H, T, 128, seed=1300 + T, p_mode="sinusoid", lengths=lens)
    c = ip.layer_constants(lay.scales)
    want = oracle_out(orc, lay, c, lens)
    assert ip.workspace_bytes(B, H, T) > 256
    for ws_bytes in (ip.workspace_bytes(B, H, T), 256):
        ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
        dl = None if lens is None else _dev(lens)
        g = Guarded((B, H, T, 128), torch.int8)
        out = ip.relpos_mhsa_i8(_dev(lay.q), _dev(lay.k), _dev(lay.v), _dev(lay.p), _dev(lay.u),
                                _dev(lay.vb), c, lengths=dl, out=g.view, workspace=ws)
        assert ip.status(ws) == 0
        g.check()
        assert_same(out.cpu().numpy(), want)


def test_empty_batch(ip):
    lay = synth.draw(0, 8, 10, 128, seed=1)
    c = ip.layer_constants(synth.draw(1, 8, 10, 128, seed=1).scales)
    out = torch.full((0, 8, 10, 128), 5, dtype=torch.int8, device="cuda")
    ws = torch.zeros(ip.workspace_bytes(0, 8, 10), dtype=torch.uint8, device="cuda")
    ip.relpos_mhsa_i8(_dev(lay.q), _dev(lay.k), _dev(lay.v), _dev(lay.p), _dev(lay.u),
                      _dev(lay.vb), c, out=out, workspace=ws)
    torch.cuda.synchronize()
    assert out.numel() == 0


def test_host_entry_point_matches_device(ip, orc):
    lay = synth.layer(2, 1)
    c = ip.layer_constants(lay.scales)
    B, H, T, dh = lay.q.shape
    arena = torch.empty(ip.host_arena_bytes(B, H, T), dtype=torch.uint8, device="cuda")
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a)).pin_memory()
    out = torch.empty((B, H, T, dh), dtype=torch.int8).pin_memory()
    ip.relpos_mhsa_i8_host(pin(lay.q), pin(lay.k), pin(lay.v), pin(lay.p), pin(lay.u),
                           pin(lay.vb), c, pin(lay.lengths), out, arena)
    assert_same(out.numpy(), oracle_out(orc, lay, c, lay.lengths))


def test_repeated_calls_share_workspace(ip, orc):
    # back-to-back calls on one stream reuse one workspace: results stay exact
    ws = None
    for i in range(3):
        lay = synth.draw(3, 8, 130, 128, seed=60 + i, p_mode="sinusoid")
        c = ip.layer_constants(lay.scales)
        if ws is None:
            ws = torch.zeros(ip.workspace_bytes(3, 8, 130), dtype=torch.uint8, device="cuda")
        out = ip.relpos_mhsa_i8(_dev(lay.q), _dev(lay.k), _dev(lay.v), _dev(lay.p), _dev(lay.u),
                                _dev(lay.vb), c, workspace=ws)
        assert ip.status(ws) == 0
        assert_same(out.cpu().numpy(), oracle_out(orc, lay, c))


def test_async_host_calls_overlap_on_two_streams(ip, orc):
    # three layers from host buffers, issued without waiting on alternating
    # streams and arenas, each output checked against the oracle
    B, H, T = 2, 8, 100
    lays = [synth.draw(B, H, T, 128, seed=990 + i, p_mode="sinusoid") for i in range(3)]
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a)).pin_memory()
    arenas = [torch.empty(ip.host_arena_bytes(B, H, T), dtype=torch.uint8, device="cuda")
              for _ in range(2)]
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    outs = []
    for i, lay in enumerate(lays):
        c = ip.layer_constants(lay.scales)
        out = torch.empty((B, H, T, 128), dtype=torch.int8).pin_memory()
        ip.relpos_mhsa_i8_host(pin(lay.q), pin(lay.k), pin(lay.v), pin(lay.p), pin(lay.u),
                               pin(lay.vb), c, None, out, arenas[i & 1], stream=streams[i & 1],
                               wait=False)
        outs.append((out, c))
    for j in range(2):
        assert ip.host_status(arenas[j], B, H, T, stream=streams[j]) == 0
    for (out, c), lay in zip(outs, lays):
        assert_same(out.numpy(), oracle_out(orc, lay, c))


def test_work_counters_return_to_zero(ip, orc):
    # The kernel's CTAs claim query tiles from counters in the workspace
    # (bytes 64 and 128); the last CTA of every call sets them back to zero,
    # so calls in a row on one workspace each see all the work.
    lay = synth.layer(3, 2)
    c = ip.layer_constants(lay.scales)
    B, H, T, dh = lay.q.shape
    ws = torch.zeros(ip.workspace_bytes(B, H, T, dh), dtype=torch.uint8, device="cuda")
    want = oracle_out(orc, lay, c)
    args = [_dev(a) for a in (lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb)]
    for _ in range(3):
        out = ip.relpos_mhsa_i8(*args, c, workspace=ws)
        torch.cuda.synchronize()
        counters = ws[64:256].cpu().numpy()
        assert not counters.any(), counters.nonzero()
        assert_same(out.cpu().numpy(), want)
    assert ip.status(ws) == 0


def test_default_workspace(ip, orc):
    # A workspace registered with ip_set_workspace serves the calls that
    # pass none, its status reads back through a NULL workspace, and its
    # item counters return to zero like an explicit workspace's.
    lay = synth.layer(3, 4)
    c = ip.layer_constants(lay.scales)
    B, H, T, dh = lay.q.shape
    ws = torch.zeros(ip.workspace_bytes(B, H, T, dh), dtype=torch.uint8, device="cuda")
    args = [_dev(a) for a in (lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb)]
    want = oracle_out(orc, lay, c)
    ip.set_workspace(ws)
    try:
        for _ in range(2):
            out = ip.relpos_mhsa_i8(*args, c)
            assert ip.status() == 0
            # the status word and the work counters (the first 256 bytes)
            # are back to zero; a score region after them is scratch
            assert not ws[:256].cpu().numpy().any()
            assert_same(out.cpu().numpy(), want)
    finally:
        ip.set_workspace(None)
    assert ip.status() == -1   # IP_ERR_NULL: nothing registered


def test_descriptor_cache_across_buffers(ip, orc):
    # The library keeps the TMA descriptors of recent (pointer, shape)
    # pairs.  Ten layers on their own buffers (two shapes, 40 descriptors,
    # more than the table holds), called in an interleaved order twice over,
    # must each produce their own oracle output.
    lays = [synth.draw(1 + (i & 1), 2, 70 + 30 * (i & 1), 128, seed=1300 + i, p_mode="sinusoid")
            for i in range(10)]
    consts = [ip.layer_constants(l.scales) for l in lays]
    want = [oracle_out(orc, l, c) for l, c in zip(lays, consts)]
    dev = [[_dev(a) for a in (l.q, l.k, l.v, l.p, l.u, l.vb)] for l in lays]
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    for rnd in range(2):
        for i in (list(range(10)) if rnd == 0 else [9, 2, 7, 0, 5, 4, 3, 6, 1, 8]):
            out = ip.relpos_mhsa_i8(*dev[i], consts[i], workspace=ws)
            assert ip.status(ws) == 0
            assert_same(out.cpu().numpy(), want[i])


def test_descriptor_cache_same_pointer_other_shape(ip, orc):
    # One allocation seen as two problem shapes at the same base address:
    # the cached TMA descriptors are keyed by pointer and shape, so each
    # call must still see its own shape.
    shapes = [(2, 2, 100), (1, 2, 200), (2, 2, 100)]
    n = max(b * h * t * 128 for b, h, t in shapes)
    np_ = max(h * (2 * t - 1) * 128 for b, h, t in shapes)
    bufs = {k: torch.empty(n, dtype=torch.int8, device="cuda") for k in "qkv"}
    pbuf = torch.empty(np_, dtype=torch.int8, device="cuda")
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    for i, (B, H, T) in enumerate(shapes):
        lay = synth.draw(B, H, T, 128, seed=1400 + i, p_mode="sinusoid")
        c = ip.layer_constants(lay.scales)
        views = {}
        for k, a in (("q", lay.q), ("k", lay.k), ("v", lay.v)):
            views[k] = bufs[k][:a.size].view(a.shape)
            views[k].copy_(torch.from_numpy(np.ascontiguousarray(a)))
        pv = pbuf[:lay.p.size].view(lay.p.shape)
        pv.copy_(torch.from_numpy(np.ascontiguousarray(lay.p)))
        out = ip.relpos_mhsa_i8(views["q"], views["k"], views["v"], pv, _dev(lay.u), _dev(lay.vb),
                                c, workspace=ws)
        assert ip.status(ws) == 0
        assert_same(out.cpu().numpy(), oracle_out(orc, lay, c))


def test_back_to_back_launches_see_the_previous_output(ip, orc):
    # Each launch may be scheduled while the one before it on the stream
    # finishes (programmatic dependent launch) and must wait for it before
    # reading memory: a second call that takes the first call's output as
    # its Q, K and V, issued right behind it, must see that output complete.
    lay = synth.layer(3, 9)
    c = ip.layer_constants(lay.scales)
    B, H, T, dh = lay.q.shape
    ws = torch.zeros(ip.workspace_bytes(B, H, T, dh), dtype=torch.uint8, device="cuda")
    first = ip.relpos_mhsa_i8(_dev(lay.q), _dev(lay.k), _dev(lay.v), _dev(lay.p), _dev(lay.u),
                              _dev(lay.vb), c, workspace=ws)
    second = ip.relpos_mhsa_i8(first, first, first, _dev(lay.p), _dev(lay.u), _dev(lay.vb), c,
                               workspace=ws)
    assert ip.status(ws) == 0
    want1 = oracle_out(orc, lay, c)
    assert_same(first.cpu().numpy(), want1)
    lay2 = synth.Layer(want1, want1, want1, lay.p, lay.u, lay.vb, None, lay.scales)
    assert_same(second.cpu().numpy(), oracle_out(orc, lay2, c))
