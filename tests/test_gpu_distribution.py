"""GPU Monte-Carlo check of the sampling rule's output law.

Many blocks share the same tiny target/drafter distributions (V = 4, gamma = 2)
and differ only in their drafts (drawn from the drafter law) and in their
Philox streams (the block index b).  The committed sequences the GPU produces
must follow the exact law that the oracle's decisions induce (computed by
exact enumeration, as in the oracle's own pin), by a chi-square test."""
import itertools

import numpy as np
import pytest
import torch

import oracle as orc
import paper_2608_14787_gb300 as sdd

pytestmark = pytest.mark.gpu

scipy_stats = pytest.importorskip("scipy.stats")


def _exact_law(pt, pd):
    from test_oracle_verify import _exact_output_law
    return _exact_output_law(orc, pt, pd)


@pytest.mark.parametrize("seed", [11, 12])
def test_sampling_law_chi_square(seed):
    rng = np.random.default_rng(seed)
    V, gamma, N = 4, 2, 131072
    zd = (rng.normal(size=(gamma, V)) * 1.2).astype(np.float32)
    zt = (rng.normal(size=(gamma + 1, V)) * 1.2).astype(np.float32)
    pd = np.stack([orc.row_probs(zd[j]) for j in range(gamma)])
    pt = np.stack([orc.row_probs(zt[j]) for j in range(gamma + 1)])
    x = np.stack([rng.choice(V, size=N, p=pd[j]) for j in range(gamma)], axis=1).astype(np.int32)
    z_d = torch.from_numpy(np.broadcast_to(zd, (N, gamma, V)).copy()).cuda()
    z_t = torch.from_numpy(np.broadcast_to(zt, (N, gamma + 1, V)).copy()).cuda()
    xd = torch.from_numpy(x).cuda()
    draft = sdd.confidence(z_d, xd)
    L, tok, n = sdd.verify_strict(z_t, xd, z_d=z_d, draft=draft, seed=seed, round_=3)
    torch.cuda.synchronize()
    Lh, th = L.cpu().numpy(), tok.cpu().numpy()
    counts = {}
    for b in range(N):
        key = tuple(th[b, :Lh[b] + 1].tolist())
        counts[key] = counts.get(key, 0) + 1
    law = _exact_law(pt, pd)
    assert set(counts) <= set(law), f"outputs outside the support: {set(counts) - set(law)}"
    keys = sorted(law)
    exp = np.array([law[k] * N for k in keys])
    obs = np.array([counts.get(k, 0) for k in keys], dtype=np.float64)
    # merge categories with small expectations
    small = exp < 5
    if small.any():
        exp = np.append(exp[~small], exp[small].sum())
        obs = np.append(obs[~small], obs[small].sum())
    res = scipy_stats.chisquare(obs, exp)
    print(f"chi-square over {len(exp)} outcomes: stat {res.statistic:.1f}, p {res.pvalue:.3g}")
    assert res.pvalue > 1e-4
    # the first committed token follows the target law exactly
    first = np.bincount(th[:, 0], minlength=V) / N
    assert np.max(np.abs(first - pt[0])) < 5 * np.sqrt(0.25 / N)
