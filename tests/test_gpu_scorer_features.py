"""The scorer's feature block (sdd_scorer_features) against its definition
written out with torch ops: App. A.7's column order, bf16 rounding, zeros in
the columns without a counterpart here."""
import pytest
import torch

from paper_2608_14787_gb300 import synth
from paper_2608_14787_gb300.binding import MLP_HIDDEN

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("B,gamma,round_", [(3, 5, 0), (16, 32, 7), (1, 1, 1000)])
def test_feature_block_columns(sdd, B, gamma, round_):
    blk = synth.make_block("c3", device="cuda", B=B, gamma=gamma, V=4096)
    conf = sdd.confidence(blk.z_d, blk.x, features=True)
    f = sdd.scorer_features(conf, round_)
    torch.cuda.synchronize()
    want = torch.zeros(B, gamma, MLP_HIDDEN, dtype=torch.bfloat16, device="cuda")
    pos = torch.arange(gamma, device="cuda", dtype=torch.float32).view(1, gamma) / gamma
    cols = {4: conf.maxprob, 5: torch.log(conf.maxprob), 6: conf.entropy, 7: -conf.entropy, 8: conf.margin,
            9: conf.top5, 14: pos.expand(B, gamma), 15: torch.full((B, gamma), round_ / 256.0, device="cuda")}
    for c, v in cols.items():
        want[:, :, c] = v.to(torch.bfloat16)
    got = f.view(B, gamma, -1)
    other = [c for c in range(MLP_HIDDEN) if c not in cols]
    assert (got[:, :, other] == 0).all()
    for c in cols:
        if c == 5:   # log: one bf16 unit of rounding either way
            torch.testing.assert_close(got[:, :, c].float(), want[:, :, c].float(), rtol=2 ** -7, atol=0)
        else:
            assert torch.equal(got[:, :, c], want[:, :, c]), c


def test_feature_block_needs_features(sdd):
    blk = synth.make_block("c3", device="cuda", B=2, gamma=3, V=1024)
    conf = sdd.confidence(blk.z_d, blk.x)
    with pytest.raises(ValueError):
        sdd.scorer_features(conf, 0)
