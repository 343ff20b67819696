"""The seeded synthetic inputs (paper_2608_14787_gb300/synth.py) against the
recipes they state: the workloads' shapes, value distributions and structure
(planted peaks, peaked / flat runs, temperatures, target noise), drafted
tokens drawn from the drafter softmax, and seeding.  Reduced vocabularies keep
this on the CPU in seconds; the recipes do not depend on V beyond the planted
value ln(V - 1) + 1/2 + 8."""
import math

import numpy as np
import pytest
import torch

from paper_2608_14787_gb300 import synth
from paper_2608_14787_gb300.synth import _gumbel_draft


def test_workload_shapes_match_their_configs():
    want = {"tiny": (1, 8, 32_000, torch.float32), "c2": (1, 32, 151_936, torch.bfloat16),
            "c3": (16, 32, 151_936, torch.bfloat16), "c4": (64, 64, 151_936, torch.bfloat16),
            "c5": (128, 32, 151_936, torch.bfloat16)}
    for name, (B, gamma, V, dt) in want.items():
        wl = synth.WORKLOADS[name]
        assert (wl.B, wl.gamma, wl.V, wl.dtype) == (B, gamma, V, dt), name
    assert synth.WORKLOADS["c5"].rounds == 256
    assert len(synth.WORKLOADS["c4"].taus) == 16
    assert synth.WORKLOADS["c3"].ells == (1.5, 2.0, 4.0) and synth.WORKLOADS["c3"].topks == (2, 5, 10)
    blk = synth.make_block("tiny")
    assert blk.z_d.shape == (1, 8, 32_000) and blk.z_t.shape == (1, 9, 32_000) and blk.x.shape == (1, 8)
    assert blk.z_d.dtype == torch.float32 and blk.x.dtype == torch.int32


def test_tiny_recipe():
    """N(0, 2) rows (one entry per row raised by 6, which moves neither
    statistic measurably); target = drafter + N(0, 0.5)."""
    blk = synth.make_block("tiny", B=4, gamma=8, V=32_000)
    zd = blk.z_d.double()
    zt = blk.z_t[:, :8].double()
    assert abs(zd.std().item() - 2.0) < 0.02
    assert abs(zd.mean().item()) < 0.02
    assert abs((zt - zd).std().item() - 0.5) < 0.01


def test_c2_recipe_temperatures_and_planted_margin():
    """n ~ N(0, 1) with a top token 2 above the next entry; drafter = n / T,
    T ~ U[0.3, 1.5]; target = 0.9 drafter + N(0, 0.7)."""
    blk = synth.make_block("c2", B=3, gamma=32, V=20_000)
    zd = blk.z_d.double()                      # bf16 values, widened
    srt = zd.sort(dim=-1, descending=True).values
    gap = srt[..., 0] - srt[..., 1]
    spread = zd.std(dim=-1)                    # ~ 1 / T (the planted entry barely moves it)
    T = 1.0 / spread
    assert (T > 0.28).all() and (T < 1.55).all()
    assert T.max() - T.min() > 0.5               # temperatures differ by position
    np.testing.assert_allclose((gap * T).numpy(), 2.0, atol=0.12)   # bf16 rounding of the two entries
    resid = blk.z_t[:, :32].double() - 0.9 * zd
    assert abs(resid.std().item() - 0.7) < 0.01


@pytest.mark.parametrize("wl_name,sigma", [("c3", 0.5), ("c4", None)])
def test_runs_recipe(wl_name, sigma):
    """Half of each block's positions peaked, in at most two contiguous runs;
    a peaked row plants one token at ln(V - 1) + 1/2 + 8 (8 nats above the
    expected log-sum-exp of the other entries) over N(0, 1), a flat row is
    N(0, 0.5); target = drafter + N(0, sigma) (c4: sigma per block row from
    U[0.2, 1.2]); the bonus row is flat."""
    gamma = 32 if wl_name == "c3" else 64
    B, V = 6, 4096
    blk = synth.make_block(wl_name, B=B, gamma=gamma, V=V)
    pk = blk.peaked.numpy()
    assert not pk[:, gamma].any()
    for b in range(B):
        row = pk[b, :gamma]
        assert row.sum() == gamma // 2
        runs = np.sum(np.diff(np.concatenate([[0], row.astype(int)])) == 1)
        assert 1 <= runs <= 2
    zd = blk.z_d.double()
    plant = math.log(V - 1) + 0.5 + 8.0
    plant_bf16 = torch.tensor(plant).to(torch.bfloat16).double().item()
    mx = zd.max(dim=-1).values.numpy()
    pkd = pk[:, :gamma]
    np.testing.assert_allclose(mx[pkd], plant_bf16)
    p_top = torch.softmax(zd, dim=-1).max(dim=-1).values.numpy()
    assert (p_top[pkd] > 0.999).all()                       # close to sigmoid(8)
    assert (p_top[~pkd] < 0.01).all()
    flat = zd[torch.from_numpy(~pkd)]
    assert abs(flat.std().item() - 0.5) < 0.01
    resid = (blk.z_t[:, :gamma].double() - zd).std(dim=(1, 2)).numpy()
    if sigma is not None:
        np.testing.assert_allclose(resid, sigma, atol=0.01)
    else:
        assert (resid > 0.19).all() and (resid < 1.21).all() and resid.max() - resid.min() > 0.1


def test_drafted_tokens_follow_the_drafter_softmax():
    """Gumbel-max drafting samples exactly the softmax: a chi-square test over
    a 4-entry row drawn 40,000 times; greedy drafting takes the argmax."""
    z = torch.tensor([1.0, 0.0, -1.0, 0.5])
    N = 40_000
    zd = z.expand(1, N, 4).contiguous()
    x = _gumbel_draft(zd, torch.Generator().manual_seed(3), greedy=False)
    counts = np.bincount(x.numpy().ravel(), minlength=4)
    p = torch.softmax(z.double(), dim=0).numpy()
    chi2 = float(((counts - N * p) ** 2 / (N * p)).sum())
    assert chi2 < 16.27     # chi-square, 3 degrees of freedom, p = 0.001
    xg = _gumbel_draft(zd[:, :10], torch.Generator().manual_seed(3), greedy=True)
    assert (xg == 0).all()
    blk = synth.make_block("c3", B=2, gamma=32, V=4096, greedy_drafts=True)
    np.testing.assert_array_equal(blk.x.numpy(), blk.z_d.float().argmax(dim=-1).numpy())


def test_inputs_are_seeded():
    a = synth.make_block("c3", B=2, gamma=8, V=2048, round_=5)
    b = synth.make_block("c3", B=2, gamma=8, V=2048, round_=5)
    c = synth.make_block("c3", B=2, gamma=8, V=2048, round_=6)
    assert torch.equal(a.z_d, b.z_d) and torch.equal(a.z_t, b.z_t) and torch.equal(a.x, b.x)
    assert not torch.equal(a.z_d, c.z_d)
