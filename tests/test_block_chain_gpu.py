"""The whole integer Conformer block (Sec. 2.1 Eqs. 1-5) on the GPU, nineteen
kernel launches, against the oracle's composition of the same block:
bit-exact on every output."""
import numpy as np
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


@pytest.mark.parametrize("B,T,seed", [(2, 64, 1), (3, 150, 2)])
def test_block_matches_oracle(ip, B, T, seed):
    import synth.block as sb
    from oracle.block import conformer_block as oracle_block
    from paper_2609_30846_gb300.block import ConformerBlock
    case = sb.conformer_block(B, T, seed=seed)
    want = oracle_block(case)
    blk = ConformerBlock(case, B, T, torch.device("cuda"))
    got = blk(torch.from_numpy(case.x).cuda())
    assert ip.status(blk.ws) == 0
    got = got.cpu().numpy()
    bad = got != want
    assert not bad.any(), f"{int(bad.sum())} of {got.size} outputs differ"
