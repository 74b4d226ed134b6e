"""The throughput probes behind the roofline denominators: argument checks,
the op counts they return, and rates that are positive and finite."""
import ctypes
import math

import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def ip():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30846_gb300 as mod
    mod.load()
    return mod


def test_probe_op_counts(ip):
    lib = ip.load()
    sink = torch.zeros(4 * 256, dtype=torch.int32, device="cuda")
    ptr = ctypes.c_void_p(sink.data_ptr())
    # per MMA warp and round: 8 chains (4 in the mixed probe) x 16 x 8 x 32 multiply-adds
    assert lib.ip_probe_int8_mma(4, 3, ptr, None) == 4 * 8 * 3 * 8 * 8192
    # mixed: per block 2 MMA warps x 4 chains, 6 dp4a warps x 4 x 4 rounds x 8 chains
    # x 32 lanes x 4 multiply-adds
    assert lib.ip_probe_int8_mix(4, 3, 2, ptr, None) == 4 * (2 * 3 * 4 * 8192 + 6 * 12 * 32 * 256)
    torch.cuda.synchronize()
    assert bool(sink.ne(0).any())
    for bad in ((0, 3, 2), (4, 0, 2), (4, 3, -1), (4, 3, 9)):
        assert lib.ip_probe_int8_mix(*bad, ptr, None) == -1
    assert lib.ip_probe_int8_mix(4, 3, 2, None, None) == -1


def test_pipe_rates_are_finite(ip):
    r = ip.int8_pipe_rates(iters=256, repeats=1)
    assert set(r) == {"imma", "dp4a", "imma_plus_dp4a"}
    for v in r.values():
        assert math.isfinite(v) and v > 0
