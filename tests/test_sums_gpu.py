"""Parity of the softmax arithmetic on its general and its fast paths.

The kernel adds the integer exponentials of a row in 32-bit partial sums
when exp(0) times the terms one thread adds per row stays below 2^32, else
in 64 bits; and it takes each probability min(floor(e f / 2^24), 255) as
one multiply-high of e and f 2^8 when exp(0) > 2^8 (every row sum then
exceeds 2^8, so f < 2^24), else from the full 64-bit product.  The host
checks both bounds per call.  The paths compute the same integers, so each
case here runs with the general paths forced and must match the oracle bit
for bit; the other parity tests take the planned (mostly fast) paths.
"""
import numpy as np
import pytest

import synth
from test_parity_gpu import assert_same, oracle_out, run_gpu

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def ip():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30846_gb300 as mod
    mod.load()
    mod.set_wide_sums(True)
    yield mod
    mod.set_wide_sums(False)


@pytest.fixture(scope="module")
def orc():
    import oracle
    oracle.build()
    return oracle


@pytest.mark.parametrize("w", [0, 1, 2])
def test_workloads_with_wide_sums(ip, orc, w):
    lay = synth.layer(w, 0)
    c = ip.layer_constants(lay.scales)
    assert_same(run_gpu(ip, lay, c, lay.lengths), oracle_out(orc, lay, c, lay.lengths))


def test_small_exponentials_take_the_general_path(ip, orc):
    # exp(0) = q_b^2 + q_c <= 2^8: a row sum can be as small as exp(0), so
    # the planned probabilities take the full 64-bit product as well
    lay = synth.draw(3, 2, 130, 128, seed=1760, p_mode="sinusoid")
    base = ip.layer_constants(lay.scales)
    ip.set_wide_sums(False)
    try:
        for sm in ((3, 6, 10), (1, 2, 0), (5, 16, 0), (2, 10, 156)):
            c = ip.LayerConstants(base.multipliers, base.shifts, sm)
            assert_same(run_gpu(ip, lay, c), oracle_out(orc, lay, c))
    finally:
        ip.set_wide_sums(True)


def test_encoder_layer_with_wide_sums(ip, orc):
    lay = synth.layer(3, 7)
    c = ip.layer_constants(lay.scales)
    assert_same(run_gpu(ip, lay, c), oracle_out(orc, lay, c))


@pytest.mark.parametrize("split", [0, 1, 2])
def test_masks_and_halves_with_wide_sums(ip, orc, split):
    T = 150
    lens = np.array([0, 1, 33, 64, 97, 150, 7, 120], np.int32)
    lay = synth.draw(len(lens), 2, T, 128, seed=1700 + split, p_mode="sinusoid", lengths=lens)
    c = ip.layer_constants(lay.scales)
    ip.set_split_mode(split)
    try:
        assert_same(run_gpu(ip, lay, c, lens), oracle_out(orc, lay, c, lens))
    finally:
        ip.set_split_mode(-1)


def test_large_exponentials_take_the_wide_path(ip, orc):
    # exp(0) = q_b^2 + q_c near 2^27: 16 terms per thread and chunk would
    # wrap 32 bits, so the planned sums are the 64-bit ones as well (and the
    # probabilities take the one multiply-high path)
    lay = synth.draw(2, 2, 96, 128, seed=1750, p_mode="sinusoid")
    base = ip.layer_constants(lay.scales)
    c = ip.LayerConstants(base.multipliers, base.shifts, (20, 100, 1 << 27))
    ip.set_wide_sums(False)
    try:
        assert_same(run_gpu(ip, lay, c), oracle_out(orc, lay, c))
    finally:
        ip.set_wide_sums(True)
