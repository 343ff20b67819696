"""Pins for the oracle's offline diagnostics: the permutation test of Sec. 5
(H1 mechanism, Table 1) and the positionwise BCE / AUROC."""
import math

import numpy as np
import pytest


def test_identical_blocks_are_permutation_invariant(orc):
    rng = np.random.default_rng(0)
    row = rng.uniform(0.6, 1.0, 16)
    q = np.tile(row, (40, 1))
    L = rng.integers(0, 17, 40)
    for signal in (0, 1, 2):
        s = orc.permutation_diagnostic(q, L, signal, 0.8, 0.85, 12, 3)
        assert (s == s[-1]).all()


@pytest.mark.parametrize("rho", [0.25, 0.5, 0.8])
def test_shared_factor_construction_of_proposition_1(orc, rho):
    """Prop. 1's construction: a block has all-high scores with probability rho,
    else all-low.  Logged order: the feasible prefix is gamma for high blocks, 0
    otherwise.  Every permutation draws each position's score independently,
    high with probability m / B (m high blocks), so the expected feasible
    prefix is sum_{k=1..gamma} (m / B)^k."""
    B, gamma, n_rep = 400, 12, 60
    m = int(rho * B)
    q = np.full((B, gamma), 0.3)
    q[:m] = 0.97
    L = np.full(B, gamma)
    s = orc.permutation_diagnostic(q, L, 0, 0.9, 0.9, n_rep, 11)
    assert s[-1] == m * gamma
    p = m / B
    mean = sum(p ** k for k in range(1, gamma + 1))
    # variance of one block's prefix K: E[K^2] - E[K]^2 with P(K >= k) = p^k
    ek2 = sum((2 * k - 1) * p ** k for k in range(1, gamma + 1))
    sd = math.sqrt((ek2 - mean ** 2) / (B * n_rep))
    assert abs(s[:-1].mean() / B - mean) < 6 * sd + 1e-12
    assert s[:-1].mean() / B < s[-1] / B or p == 1.0   # the collapse of Table 1


def test_conditional_permutes_only_blocks_still_at_risk(orc):
    """Blocks with L < j - 1 keep their score at j: with L = 0 everywhere only
    position 1 is permuted, and with position-1 scores all equal nothing moves."""
    rng = np.random.default_rng(2)
    q = rng.uniform(0.5, 1.0, (30, 10))
    q[:, 0] = 0.99
    L = np.zeros(30, np.int64)
    s = orc.permutation_diagnostic(q, L, 2, 0.6, 0.6, 8, 5)
    assert (s == s[-1]).all()
    s_raw = orc.permutation_diagnostic(q, L, 0, 0.6, 0.6, 8, 5)   # raw: every block at every position
    assert not (s_raw[:-1] == s_raw[-1]).all()


def test_position_metrics_vs_library(orc):
    sk = pytest.importorskip("sklearn.metrics")
    rng = np.random.default_rng(4)
    B, gamma = 300, 6
    L = rng.integers(0, gamma + 1, B)
    q = np.clip(0.5 + 0.1 * (L[:, None] - np.arange(1, gamma + 1)[None, :]) + rng.normal(0, 0.2, (B, gamma)),
                0.0, 1.0)
    q[::7, 2] = 1.0                    # exact ones: the clamp keeps the loss finite
    q[::5, 1] = np.round(q[::5, 1], 1)  # ties for the AUROC
    for cond in (False, True):
        bce, base, auc, npos, nneg = orc.position_metrics(q, L, cond)
        for j in range(gamma):
            idx = np.arange(B) if not cond else np.where(L >= j)[0]
            y = (L[idx] >= j + 1).astype(int)
            qc = np.clip(q[idx, j], 1e-7, 1 - 1e-7)
            assert bce[j] == pytest.approx(sk.log_loss(y, qc, labels=[0, 1]), rel=1e-12)
            p = y.mean()
            want = 0.0 if p in (0.0, 1.0) else -(p * math.log(p) + (1 - p) * math.log(1 - p))
            assert base[j] == pytest.approx(want, rel=1e-12, abs=1e-15)
            if 0 < y.sum() < len(y):
                assert auc[j] == pytest.approx(sk.roc_auc_score(y, q[idx, j]), rel=1e-12)
            assert npos[j] == y.sum() and nneg[j] == len(y) - y.sum()
