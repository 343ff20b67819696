"""Pins of the oracle's softmax normaliser, its -2^23 logit floor and the
permutation diagnostic's shuffle (checks in tests/oracle_pins.py).  The same
checks are run against oracle builds with planted mistakes in
tests/test_oracle_mutants.py, where each must fail."""
import numpy as np

from oracle_pins import check_fisher_yates, check_floor, check_row_probs


def test_row_probs_is_the_library_softmax(orc):
    check_row_probs(orc)


def test_logit_floor(orc):
    check_floor(orc)


def test_features_share_the_floor(orc):
    """The extended features follow the same floor: rows at or below it have no
    features; entries far below it change nothing."""
    z = np.array([[-2.0 ** 23, -1e30, -np.inf, -3e38]], np.float32)
    mg, t5 = orc.row_features(z)
    assert np.isnan(mg[0]) and np.isnan(t5[0])


def test_fisher_yates_is_uniform(orc):
    check_fisher_yates(orc)


def test_diagnostic_applies_the_shuffle(orc):
    """One repetition of the permutation diagnostic on a column with distinct
    scores equals re-scheduling the scores permuted by orc.shuffle (the t-th
    valid block takes the score of valid block perm[t])."""
    rng = np.random.default_rng(3)
    B, gamma, seed = 9, 3, 77
    q = rng.uniform(0.5, 1.0, (B, gamma))
    L = rng.integers(0, gamma + 1, B).astype(np.int32)
    for signal in (0, 2):
        sums = orc.permutation_diagnostic(q, L, signal, 0.7, 0.75, 1, seed)
        qp = q.copy()
        for j in range(gamma):
            valid = [b for b in range(B) if signal != 2 or L[b] >= j]
            perm = orc.shuffle(len(valid), seed, j, 0)
            for t, b in enumerate(valid):
                qp[b, j] = q[valid[perm[t]], j]
        Kh, _, _, _ = orc.schedule(qp, signal, 0.7, 0.75, 0, 1 << 30)
        assert sums[0] == Kh.sum()
        Kh0, _, _, _ = orc.schedule(q, signal, 0.7, 0.75, 0, 1 << 30)
        assert sums[1] == Kh0.sum()
