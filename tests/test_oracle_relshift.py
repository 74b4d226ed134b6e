"""Pins of the oracle's relative shift Phi (Sec. 3.1, Eq. 8 and the remark
after Eq. 11 that Phi only moves values and inserts zeros, applied as a
static index map on the integer tensor).

The pin is the literal Transformer-XL route for the shift (Dai et al., 2019,
appendix B): prepend one zero column to BD [T, 2T-1], reinterpret the
[T, 2T] buffer as [2T, T], drop the first row, reinterpret the remainder as
[T, 2T-1] and keep the first T columns.  That route is written here from
that description and compared, brute force, with the oracle's gather.
"""
import numpy as np
import pytest

import synth


def literal_relshift(bd: np.ndarray, pad_value=0) -> np.ndarray:
    """Transformer-XL shift of bd [..., T, 2T-1] -> [..., T, T]."""
    *lead, T, R = bd.shape
    assert R == 2 * T - 1
    padded = np.concatenate([np.full((*lead, T, 1), pad_value, dtype=bd.dtype), bd], axis=-1)
    flat = padded.reshape(*lead, T * 2 * T)
    rows = flat.reshape(*lead, 2 * T, T)[..., 1:, :]          # drop the first row
    back = rows.reshape(*lead, T * (2 * T - 1))
    return back.reshape(*lead, T, 2 * T - 1)[..., :T]


def _bd(lay):
    """(Q + 1v^T) P^T by integer matrix products, int64 [B, H, T, 2T-1]."""
    q = lay.q.astype(np.int64) + lay.vb.astype(np.int64)[None, :, None, :]
    return np.einsum("bhid,hrd->bhir", q, lay.p.astype(np.int64))


@pytest.mark.parametrize("T", list(range(1, 17)))
def test_phi_equals_transformer_xl_route(oracle_lib, T):
    lay = synth.draw(1, 2, T, 8, seed=700 + T)
    want = literal_relshift(_bd(lay))
    got = oracle_lib.position_scores(lay.q, lay.p, lay.vb)
    np.testing.assert_array_equal(got, want)


@pytest.mark.parametrize("T", [1, 2, 3, 5, 9, 16])
def test_phi_inserted_zeros_never_reach_kept_scores(T):
    # Run the literal route with a sentinel in place of the inserted zeros:
    # with 2T-1 relative rows no sentinel survives in the T kept columns.
    bd = np.arange(T * (2 * T - 1), dtype=np.int64).reshape(T, 2 * T - 1)
    out = literal_relshift(bd, pad_value=-1)
    assert (out >= 0).all()
    i = np.arange(T)[:, None]
    j = np.arange(T)[None, :]
    np.testing.assert_array_equal(out, bd[i, j - i + T - 1])


def test_phi_direction_relative_distance(oracle_lib):
    # Row r of P carries relative distance T-1-r: with Q = e_0 and v = 0,
    # qp[i][j] reads P[j-i+T-1][0]; encode r itself in that column.
    T, dh = 6, 4
    q = np.zeros((1, 1, T, dh), np.int8)
    q[..., 0] = 1
    p = np.zeros((1, 2 * T - 1, dh), np.int8)
    p[0, :, 0] = np.arange(2 * T - 1)
    vb = np.zeros((1, dh), np.int8)
    got = oracle_lib.position_scores(q, p, vb)[0, 0]
    i = np.arange(T)[:, None]
    j = np.arange(T)[None, :]
    np.testing.assert_array_equal(got, j - i + T - 1)
    # the diagonal (i == j, distance 0) reads the middle row T-1
    assert (np.diag(got) == T - 1).all()


def test_phi_commutes_with_scaling(oracle_lib):
    # Phi(S q) = S Phi(q): the position branch is linear in P.
    lay = synth.draw(1, 2, 9, 16, seed=11)
    p_small = (lay.p // 4).astype(np.int8)
    one = oracle_lib.position_scores(lay.q, p_small, lay.vb).astype(np.int64)
    three = oracle_lib.position_scores(lay.q, (3 * p_small).astype(np.int8), lay.vb).astype(np.int64)
    np.testing.assert_array_equal(three, 3 * one)
