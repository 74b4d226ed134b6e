"""Seeded random sweep of the attention layer (Sec. 3.1, Eqs. 8-11 with the
integer softmax and Eq. 7) through the C ABI against the oracle, bit for
bit: each case draws its shape (B, H, T), its value distribution and
position table, a key-padding mask (lengths 0 .. T), a score grid S_s
scaled by 2^U(-2, 2) around the calibrated one (so that q_ln2 runs from
coarse to fine grids), the output grid, the tile split of the kernel, the
output layout and, for T > 384, whether the workspace holds the score
region (scores in L2) or only its first 256 bytes (scores in shared
memory).  Guard bytes around the output catch a write outside it.
"""
import numpy as np
import pytest

import synth
from guard import Guarded

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

HEADS, ROWS = 1, 0


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


def _case(i):
    rng = np.random.default_rng(50_000 + i)
    H = int(rng.choice([1, 2, 3, 5, 8, 16]))
    # a mix of short, tile-edge and long sequences, B H T^2 bounded so that
    # the oracle takes well under a second per case
    T = int(rng.choice([int(rng.integers(1, 130)), int(rng.choice([63, 64, 65, 127, 128, 129,
                                                                    383, 384, 385])),
                        int(rng.integers(130, 900))]))
    B = int(max(1, min(int(rng.integers(1, 5)), 6_000_000 // (H * T * T + 1))))
    masked = bool(rng.integers(0, 2))
    lengths = None
    if masked:
        lengths = rng.integers(0, T + 1, size=B).astype(np.int32)
        if B > 1 and rng.integers(0, 2):
            lengths[int(rng.integers(0, B))] = 0
    lay = synth.draw(B, H, T, 128, seed=60_000 + i, p_mode=str(rng.choice(["random", "sinusoid"])),
                     dist=str(rng.choice(["normal", "t3"])), lengths=lengths)
    scales = dict(lay.scales)
    scales["S_s"] *= float(2.0 ** rng.uniform(-2.0, 2.0))
    scales["S_O"] *= float(2.0 ** rng.uniform(-1.0, 1.0))
    split = int(rng.choice([-1, 0, 1, 2]))
    layout = int(rng.choice([HEADS, ROWS]))
    small_ws = bool(T > 384 and rng.integers(0, 2))
    return lay, scales, lengths, split, layout, small_ws


@pytest.mark.parametrize("i", range(32))
def test_random_layers(ip, orc, i):
    lay, scales, lengths, split, layout, small_ws = _case(i)
    B, H, T, dh = lay.q.shape
    c = ip.layer_constants(scales)
    want = orc.relpos_mhsa(lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb,
                           orc.LayerConstants(c.multipliers, c.shifts, c.softmax), lengths)
    if layout == ROWS:
        want = np.ascontiguousarray(want.transpose(0, 2, 1, 3))
    nbytes = 256 if small_ws else ip.workspace_bytes(B, H, T, dh)
    ws = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
    g = Guarded(want.shape, torch.int8)
    lens = None if lengths is None else _dev(lengths)
    try:
        ip.set_split_mode(split)
        ip.relpos_mhsa_i8(_dev(lay.q), _dev(lay.k), _dev(lay.v), _dev(lay.p), _dev(lay.u),
                          _dev(lay.vb), c, lengths=lens, out=g.view, workspace=ws,
                          out_layout=layout)
        assert ip.status(ws) == 0
    finally:
        ip.set_split_mode(-1)
    g.check()
    got = g.view.cpu().numpy()
    bad = got != want
    if bad.any():
        idx = np.argwhere(bad)[0].tolist()
        raise AssertionError(f"case {i} (B={B} H={H} T={T} split={split} layout={layout} "
                             f"small_ws={small_ws}): {int(bad.sum())} of {got.size} outputs "
                             f"differ; first at {idx}")
