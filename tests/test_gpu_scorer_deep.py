"""GPU parity of the deep scorer (sdd_scorer_deep: the learned scorer's shape of
App. A.7, (3584 + 19) -> 256 -> 256 -> 256 -> 1 with stand-in weights) against
the fp64 oracle, whose activations are exact.

Tolerance (derived).  The tensor-core path rounds the first two layers'
activations to bf16 operands (unit roundoff u = 2^-8, errors independent with
variance <= u^2 |a|^2 / 3) and accumulates exact bf16 products in fp32 (~1e-6).
With the stand-in scales (W2, W3, w4 ~ U(+-1/16), |a1| ~ 0.3, |a2| ~ 0.3 rms)
the first-order propagation gives a layer-2 pre-activation error of
sqrt(256 * 1.3e-3 * 0.1 * u^2 / 3) ~ 4e-4 rms, a layer-3 error ~ 3.4e-4, a head
error ~ 1.3e-4 and, through the sigmoid's slope <= 1/4, an output error
sigma_s ~ 3e-5; measured in fp64 on the decode-loop batch: 1e-5 rms, 4e-5
maximum over 4096 rows.  The tests allow 3e-4 absolute (about 10 sigma_s); a
wrong operand layout or index errs by ~1e-1."""
import numpy as np
import pytest
import torch

from paper_2608_14787_gb300 import synth

pytestmark = pytest.mark.gpu
ATOL = 3e-4


def _oracle(orc, h, f, w, rows):
    W1, b1, W2, b2, W3, b3, w4, b4 = w
    x = torch.cat([h[rows], f[rows]], dim=-1)
    bits = synth.bf16_bits
    return orc.scorer_deep(bits(x), bits(W1), b1.cpu().numpy(), bits(W2), b2.cpu().numpy(), bits(W3),
                           b3.cpu().numpy(), bits(w4), b4)


@pytest.mark.parametrize("M,Kh", [(1, 64), (130, 256), (300, 1024), (128, 3584)])
def test_scorer_deep_matches_oracle(sdd, orc, M, Kh):
    w = synth.make_scorer_deep(device="cuda", hidden=Kh)
    h = synth.make_hidden(M, device="cuda", seed=8, hidden=Kh)
    f = synth.make_features(M, device="cuda")
    status = sdd.new_status(h.device)
    s = sdd.scorer_deep(h, f, *w, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    want = _oracle(orc, h, f, w, slice(None))
    np.testing.assert_allclose(s.cpu().numpy(), want, rtol=0, atol=ATOL)


def test_scorer_deep_decode_loop_batch_sampled(sdd, orc):
    """The decode-loop batch (128 blocks x 32 positions, hidden 3584), 192
    sampled rows across all 32 tiles; the two launches reuse the same act."""
    M, Kh = 4096, synth.HIDDEN
    w = synth.make_scorer_deep(device="cuda", hidden=Kh)
    h = synth.make_hidden(M, device="cuda", seed=9, hidden=Kh)
    f = synth.make_features(M, device="cuda", round_=1)
    act = torch.empty(M, 256, dtype=torch.bfloat16, device="cuda")
    status = sdd.new_status(h.device)
    s1 = sdd.scorer_deep(h, f, *w, act=act, status=status)
    s2 = sdd.scorer_deep(h, f, *w, act=act, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert torch.equal(s1, s2)                          # deterministic
    rows = np.random.default_rng(0).choice(M, 192, replace=False)
    want = _oracle(orc, h, f, w, torch.from_numpy(rows).to("cuda"))
    np.testing.assert_allclose(s1.cpu().numpy()[rows], want, rtol=0, atol=ATOL)
    # the first layer's activations are the bf16 operands of the second layer
    assert act.dtype == torch.bfloat16 and torch.isfinite(act.float()).all()


def test_scorer_deep_feature_columns_matter(sdd, orc):
    """Only the feature block changes between the two calls: the scores move,
    and both match the oracle (the second A operand is indexed correctly)."""
    M, Kh = 256, 512
    w = synth.make_scorer_deep(device="cuda", hidden=Kh)
    h = synth.make_hidden(M, device="cuda", seed=10, hidden=Kh)
    f0 = synth.make_features(M, device="cuda", round_=0)
    f1 = synth.make_features(M, device="cuda", round_=1)
    s0 = sdd.scorer_deep(h, f0, *w)
    s1 = sdd.scorer_deep(h, f1, *w)
    torch.cuda.synchronize()
    assert (s0 - s1).abs().max().item() > 1e-3
    np.testing.assert_allclose(s1.cpu().numpy(), _oracle(orc, h, f1, w, slice(None)), rtol=0, atol=ATOL)
