"""The whole integer Conformer block (Sec. 2.1 Eqs. 1-5) on the GPU, fifteen
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


# (32, 375): the benchmark's block shape (30 s utterances, 12000 frames);
# (3, 301): 903 frames, not a multiple of the 128-frame tiles of the
# projections, and T not a multiple of the attention's 64-row tiles.
@pytest.mark.parametrize("B,T,seed", [(2, 64, 1), (3, 150, 2), (3, 301, 4), (4, 375, 3),
                                      (32, 375, 5)])
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
    if bad.any():
        idx = np.argwhere(bad)[0].tolist()
        raise AssertionError(f"{int(bad.sum())} of {got.size} outputs differ; first at {idx}")


def test_block_graph_replay_matches_oracle(ip):
    # the fifteen launches captured once into a CUDA graph; each replay on a
    # new input equals the oracle's block on that input
    import synth.block as sb
    from oracle.block import conformer_block as oracle_block
    from paper_2609_30846_gb300.block import ConformerBlock
    B, T = 2, 100
    cases = [sb.conformer_block(B, T, seed=s) for s in (11, 12)]
    blk = ConformerBlock(cases[0], B, T, torch.device("cuda"))
    x = torch.from_numpy(cases[0].x).cuda()
    g = blk.graph(x)
    for case in cases:
        # same weights and grids, new frames
        x.copy_(torch.from_numpy(case.x).cuda())
        g.replay()
        torch.cuda.synchronize()
        want = oracle_block(sb.BlockCase(**{**cases[0].__dict__, "x": case.x}))
        got = blk.out.cpu().numpy()
        bad = got != want
        assert not bad.any(), f"{int(bad.sum())} of {got.size} outputs differ"
    assert ip.status(blk.ws) == 0
