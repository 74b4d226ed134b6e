"""Failure detection on the GPU without a fault: every barrier wait inside
the kernel is bounded.  The stall-injection hook makes every consumer warp
wait on a barrier that nothing arrives on (with a short budget of about a
millisecond); the wait runs out, the kernel records IP_ERR_TIMEOUT in its
status word, lets its own copies in flight land and returns.  The host reads
the status, and the context stays usable: the next call is exact again."""
import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def test_barrier_timeout_is_reported_and_context_survives():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import oracle
    import paper_2609_30846_gb300 as ip
    lay = synth.draw(2, 8, 200, 128, seed=4401, p_mode="sinusoid")
    c = ip.layer_constants(lay.scales)
    dev = [torch.from_numpy(np.ascontiguousarray(a)).cuda()
           for a in (lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb)]
    ws = torch.zeros(ip.workspace_bytes(2, 8, 200), dtype=torch.uint8, device="cuda")
    try:
        ip.set_timeout_cycles(2_000_000)
        ip.set_stall_injection(True)
        ip.relpos_mhsa_i8(*dev, c, workspace=ws)
        assert ip.status(ws) == -6          # IP_ERR_TIMEOUT, read and cleared
        assert ip.status(ws) == 0
    finally:
        ip.set_stall_injection(False)
        ip.set_timeout_cycles(-1)
    out = ip.relpos_mhsa_i8(*dev, c, workspace=ws)
    assert ip.status(ws) == 0
    want = oracle.relpos_mhsa(lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb,
                              oracle.layer_constants(lay.scales, 128))
    np.testing.assert_array_equal(out.cpu().numpy(), want)
