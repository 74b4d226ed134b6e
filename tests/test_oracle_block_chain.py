"""The oracle's whole integer Conformer block (Sec. 2.1 Eqs. 1-5) against the
real-valued block it quantises: the dequantised int8 output of the
calibration utterances tracks the float64 forward (the integer chain adds
rounding at every grid, the final LayerNorm rescales), and the parts that
the chain reuses are pinned in their own tests."""
import numpy as np

import synth.block as sb
from oracle.block import conformer_block


def test_every_stage_tracks_the_real_valued_block():
    # each dequantised intermediate against the float64 forward of the same
    # stage: a wrong grid, coefficient or wiring shows as a slope away from 1
    # or a drop in correlation at the stage where it happens
    case = sb.conformer_block(2, 48, seed=3)
    tr = {}
    conformer_block(case, trace=tr)
    n = case.calib
    for name, ref in case.ref.items():
        if name not in tr:
            continue                       # the block input itself
        got = tr[name][:n]
        y = got.astype(np.float64) * case.s[name]
        y, r = y.ravel(), np.asarray(ref, dtype=np.float64).ravel()
        slope = float(np.dot(y, r) / np.dot(r, r))
        corr = float(np.corrcoef(y, r)[0, 1])
        assert 0.9 < slope < 1.1, (name, slope)
        assert corr > 0.97, (name, corr)
    y = tr["out"][:n].astype(np.float64) * case.s["out"]
    assert np.mean(np.abs(y - case.ref_out)) / case.s["out"] < 4.0


def test_block_is_per_utterance():
    # each utterance of a batch is processed independently
    case = sb.conformer_block(3, 40, seed=4)
    full = conformer_block(case)
    sub = sb.BlockCase(**{**case.__dict__, "x": case.x[1:2]})
    np.testing.assert_array_equal(conformer_block(sub)[0], full[1])
