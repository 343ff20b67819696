"""Pin checks of the oracle that are shared by the ordinary pin tests and by
the planted-mistake tests (tests/test_oracle_mutants.py).  Each check takes
the oracle module, raises AssertionError when the oracle disagrees with what
the mathematics fixes, and returns None otherwise.

* check_row_probs    -- the normalised softmax behind the strict rule's
                        residual max(0, p_t - p_d) and its bonus draw (Sec. 3.1)
                        against fp64 library softmax on random, peaked and
                        masked rows, fp32 and bf16.
* check_floor        -- logits are floored at -2^23: a row whose entries all lie
                        at or below the floor has no distribution, and entries far
                        below it act as masked.
* check_fisher_yates -- the permutation diagnostic's shuffle (Sec. 5, Table 1)
                        is uniform over all n! orders (chi-square, n = 3 and 4).
"""
import math

import numpy as np
import torch
from scipy import stats


def _bf16_bits(x: np.ndarray) -> np.ndarray:
    return torch.from_numpy(np.asarray(x, np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def _bf16_vals(bits: np.ndarray) -> np.ndarray:
    return torch.from_numpy(np.asarray(bits, np.uint16).view(np.int16)).view(torch.bfloat16).double().numpy()


def _library_softmax(vals: np.ndarray) -> np.ndarray:
    return torch.softmax(torch.from_numpy(vals), dim=-1).numpy()


def _row_probs_cases():
    rng = np.random.default_rng(20)
    cases = []
    for V in (1, 5, 1003, 32000):
        cases.append(rng.normal(0.0, 2.0, V).astype(np.float32))              # random
    peaked = rng.normal(0.0, 1.0, 4001).astype(np.float32)
    peaked[1234] = 30.0                                                       # one dominant token
    cases.append(peaked)
    masked = rng.normal(0.0, 1.5, 2000).astype(np.float32)
    masked[rng.choice(2000, 700, replace=False)] = -np.inf                   # masked entries
    cases.append(masked)
    return cases


def check_row_probs(orc):
    for z in _row_probs_cases():
        for bits in (False, True):
            arg = _bf16_bits(z) if bits else z
            vals = _bf16_vals(arg) if bits else z.astype(np.float64)
            p = orc.row_probs(arg)
            want = _library_softmax(vals)
            assert p.shape == want.shape
            np.testing.assert_allclose(p, want, rtol=1e-12, atol=1e-300)
            assert abs(p.sum() - 1.0) < 1e-12
            assert np.all(p[np.isneginf(vals)] == 0.0)


def check_floor(orc):
    floor = -2.0 ** 23
    # every entry at or below the floor: no distribution
    below = np.array([[floor, -1e30, floor * 4, -np.inf],
                      [-3e38, -3e38, -3e38, -3e38],
                      [floor, floor, floor, floor]], np.float32)
    st = orc.row_stats(below, tokens=[0, 1, 2])
    for name in ("lse", "q", "logq", "maxprob", "entropy"):
        assert np.all(np.isnan(getattr(st, name))), name
    assert np.all(st.argmax == -1)
    # finite entries far below the floor act as masked entries
    rng = np.random.default_rng(21)
    z = rng.normal(0.0, 2.0, (3, 600)).astype(np.float32)
    far = z.copy()
    masked = z.copy()
    for r in range(3):
        idx = rng.choice(600, 150, replace=False)
        idx = idx[idx != 7]
        far[r, idx] = -3e38
        masked[r, idx] = -np.inf
    a = orc.row_stats(far, tokens=[7, 7, 7])
    b = orc.row_stats(masked, tokens=[7, 7, 7])
    for name in ("lse", "q", "logq", "maxprob", "entropy"):
        np.testing.assert_array_equal(getattr(a, name), getattr(b, name), err_msg=name)
    np.testing.assert_array_equal(a.argmax, b.argmax)
    # a row above the floor keeps its distribution (one entry 1024 above it: the
    # floored others weigh exp(-1024) = 0, so LSE is that logit)
    one = np.full((1, 8), -np.inf, np.float32)
    one[0, 5] = floor + 1024.0
    st = orc.row_stats(one, tokens=[5])
    assert st.lse[0] == floor + 1024.0 and st.maxprob[0] == 1.0 and st.q[0] == 1.0 and st.argmax[0] == 5
    assert st.entropy[0] == 0.0


def check_fisher_yates(orc, n_draws: int = 24000, seed: int = 0x5EED):
    """The n! orders of n = 3 and n = 4 items are equally likely over
    n_draws repetitions (counter r), at a fixed position; the chi-square
    statistic must be plausible at the 1e-4 level.  A shuffle that cannot
    produce some order (Sattolo's cyclic variant never yields the identity)
    fails outright."""
    for n in (3, 4):
        counts = {}
        for r in range(n_draws):
            p = tuple(int(v) for v in orc.shuffle(n, seed, 2, r))
            assert sorted(p) == list(range(n))
            counts[p] = counts.get(p, 0) + 1
        cells = math.factorial(n)
        assert len(counts) == cells, f"only {len(counts)} of {cells} orders drawn for n = {n}"
        expected = n_draws / cells
        chi2 = sum((c - expected) ** 2 / expected for c in counts.values())
        pval = stats.chi2.sf(chi2, cells - 1)
        assert pval > 1e-4, f"n = {n}: chi2 = {chi2:.1f} on {cells - 1} dof (p = {pval:.2e})"
    # degenerate sizes
    assert list(orc.shuffle(0, seed, 0, 0)) == []
    assert list(orc.shuffle(1, seed, 0, 0)) == [0]
