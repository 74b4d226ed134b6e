"""The guard-byte helper of the GPU parity tests, on the CPU: a write past
either end of a guarded output is reported, writes inside it are not."""
import numpy as np
import pytest

from guard import GUARD, Guarded

torch = pytest.importorskip("torch")


def test_inside_writes_pass():
    g = Guarded((3, 7, 5), torch.int8, device="cpu")
    g.view.fill_(-3)
    g.check()
    assert g.view.shape == (3, 7, 5) and g.view.dtype == torch.int8


@pytest.mark.parametrize("where", [GUARD - 1, 0, -1, -GUARD])
def test_stray_write_is_caught(where):
    g = Guarded((4, 16), torch.int8, device="cpu")
    idx = where if where >= 0 else g.buf.numel() + where
    g.buf[idx] ^= 0x5A
    with pytest.raises(AssertionError):
        g.check()


def test_view_keeps_alignment():
    g = Guarded((2, 8, 128), torch.int8, device="cpu")
    assert (g.view.data_ptr() - g.buf.data_ptr()) == GUARD and GUARD % 256 == 0


def test_valid_ops_of_masked_workload():
    import bench
    import synth
    w = synth.WORKLOADS[2]
    lens = np.array([w.T] * w.B)
    assert bench.valid_ops(w, lens) == bench.useful_ops(w.B, w.H, w.T, w.dh, 1)
    assert bench.valid_ops(w, np.array([0, w.T + 5] + [0] * (w.B - 2))) == 6 * w.dh * w.H * w.T ** 2
