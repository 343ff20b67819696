"""Pins for the oracle's acceptance rules: Strict SDD (Sec. 3.1, the
speculative-sampling rule it cites), lenience (App. A.6 Eq. 9), top-k (App. A.6),
the inverse-CDF draw and the agreement metrics (Sec. 3.2 Eq. 1-2)."""
import itertools
import math

import numpy as np
import pytest
import torch


def _softmax(z):
    return torch.softmax(torch.from_numpy(np.asarray(z, np.float64)), dim=-1).numpy()


def _measure_monotone(f, outcomes):
    """Lebesgue measure of {u in (0,1): f(u) = o} for a step function f that is
    monotone in u (each outcome occupies one interval).  Boundaries by bisection."""
    grid = np.linspace(0, 1, 257)[1:-1]
    vals = [f(u) for u in grid]
    pts = [0.0]
    for i in range(len(grid) - 1):
        if vals[i] != vals[i + 1]:
            lo, hi = grid[i], grid[i + 1]
            vlo = vals[i]
            # there may be several boundaries inside; walk them one by one
            while True:
                a, b = lo, hi
                for _ in range(60):
                    mid = 0.5 * (a + b)
                    if f(mid) == vlo:
                        a = mid
                    else:
                        b = mid
                pts.append(b)
                nxt = f(b)
                if nxt == vals[i + 1]:
                    break
                lo, vlo = b, nxt
    pts.append(1.0)
    seq = [vals[0]]
    for p in pts[1:-1]:
        seq.append(f(min(p + 1e-15, 1 - 1e-16)))
    m = {o: 0.0 for o in outcomes}
    for k in range(len(pts) - 1):
        m[seq[k]] = m.get(seq[k], 0.0) + (pts[k + 1] - pts[k])
    return m


def _exact_output_law(orc, pt, pd):
    """Law of (committed tokens) of the oracle's strict sampling rule, with the
    drafts drawn from pd (independently per position) and the acceptance/residual/
    bonus uniforms integrated out exactly through the oracle's own decisions."""
    gamma, V = pd.shape
    law = {}
    HI = 1.0 - 2.0 ** -24
    for x in itertools.product(range(V), repeat=gamma):
        px = float(np.prod([pd[j, x[j]] for j in range(gamma)]))
        if px == 0.0:
            continue

        # acceptance probability at each position from the oracle's accept decision
        def L_of(u_vec):
            L, _, _ = orc.strict_sample_probs(pt, pd, x, u_vec, 0.5, 0.5)
            return L

        acc = []
        for j in range(gamma):
            def f(u, j=j):
                uv = [1e-9] * gamma
                uv[j] = u
                for k in range(j + 1, gamma):
                    uv[k] = HI
                return L_of(uv) > j
            acc.append(_measure_monotone(f, [True, False])[True])
        # reach position L exactly and draw the final token
        for L in range(gamma + 1):
            p_reach = px * np.prod(acc[:L]) * ((1 - acc[L]) if L < gamma else 1.0)
            if p_reach == 0.0:
                continue
            u_vec = [1e-9] * L + ([HI] if L < gamma else []) + [HI] * max(0, gamma - L - 1)
            if L < gamma and acc[L] >= 1.0:
                continue

            def g(u, L=L, u_vec=u_vec):
                if L < gamma:
                    Lr, tok, _ = orc.strict_sample_probs(pt, pd, x, u_vec, u, 0.5)
                else:
                    Lr, tok, _ = orc.strict_sample_probs(pt, pd, x, u_vec, 0.5, u)
                assert Lr == L
                return int(tok[L])

            draw = _measure_monotone(g, list(range(V)))
            for y, pm in draw.items():
                if pm == 0.0:
                    continue
                key = tuple(x[:L]) + (y,)
                law[key] = law.get(key, 0.0) + p_reach * pm
    return law


@pytest.mark.parametrize("V,gamma,seed", [(3, 1, 0), (4, 2, 1), (3, 3, 2), (5, 2, 3), (8, 1, 4)])
def test_strict_sampling_reproduces_target_law(orc, V, gamma, seed):
    rng = np.random.default_rng(seed)
    zd = rng.normal(size=(gamma, V)) * 1.5
    zt = rng.normal(size=(gamma + 1, V)) * 1.5
    pd, pt = _softmax(zd), _softmax(zt)
    law = _exact_output_law(orc, pt, pd)
    assert abs(sum(law.values()) - 1.0) < 1e-9
    # Target rows here do not depend on the prefix, so the committed sequence must
    # follow pt position by position: P(c_1..c_m = y, n >= m) = P(c_1..c_{m-1} = y', n >= m) pt_m(y_m),
    # where P(n >= m | prefix) is whatever the rule produces.
    def prefix_mass(prefix):
        return sum(p for k, p in law.items() if k[:len(prefix)] == tuple(prefix))

    for y in range(V):
        assert prefix_mass([y]) == pytest.approx(pt[0, y], abs=1e-9)
    for m in range(2, gamma + 2):
        for prefix in itertools.product(range(V), repeat=m - 1):
            reach = sum(p for k, p in law.items() if len(k) >= m and k[:m - 1] == prefix)
            for y in range(V):
                got = sum(p for k, p in law.items() if len(k) >= m and k[:m] == prefix + (y,))
                assert got == pytest.approx(reach * pt[m - 1, y], abs=1e-9)


def test_identical_rows_always_accept(orc):
    rng = np.random.default_rng(5)
    for trial in range(50):
        gamma, V = 6, 40
        z = (rng.normal(size=(gamma + 1, V)) * 2).astype(np.float32)
        x = rng.integers(0, V, size=gamma).astype(np.int32)
        L, tok, _ = orc.verify_strict(z, z[:gamma], x, seed=trial, b=trial % 7, round_=trial)
        assert L == gamma
        np.testing.assert_array_equal(tok[:gamma], x)


def test_residual_has_zero_mass_on_overrepresented_tokens(orc):
    rng = np.random.default_rng(6)
    V = 50
    for trial in range(200):
        pd = _softmax(rng.normal(size=(1, V)) * 2)
        pt = _softmax(rng.normal(size=(2, V)) * 2)
        x = [int(np.argmax(pd[0] - pt[0]))]         # a token the target underweights
        L, tok, _ = orc.strict_sample_probs(pt, pd, x, [1 - 2 ** -24], rng.random(), 0.5)
        assert L == 0
        assert pt[0, tok[0]] > pd[0, tok[0]]


def test_inverse_cdf_matches_searchsorted(orc):
    rng = np.random.default_rng(7)
    for trial in range(200):
        V = int(rng.integers(1, 60))
        w = rng.random(V) * (rng.random(V) < 0.7)
        if w.sum() == 0:
            w[rng.integers(V)] = 1.0
        u = rng.random()
        v, _ = orc.inverse_cdf(w, u)
        want = int(np.searchsorted(np.cumsum(w), u * w.sum(), side="right"))
        assert v == want
        assert w[v] > 0


def test_inverse_cdf_frequencies(orc):
    w = np.array([0.1, 0.0, 0.25, 0.15, 0.5])
    us = (np.arange(100000) + 0.5) / 100000
    counts = np.bincount([orc.inverse_cdf(w, u)[0] for u in us], minlength=5)
    np.testing.assert_allclose(counts / us.size, w / w.sum(), atol=2e-5)


def _bf16_bits(x):
    return torch.from_numpy(np.asarray(x, np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def _random_block(rng, gamma, V, scale=0.4):
    zt = _bf16_bits(rng.normal(size=(gamma + 1, V)) * scale)
    zd = _bf16_bits(rng.normal(size=(gamma, V)) * scale)
    vals = torch.from_numpy(zt.view(np.int16)).view(torch.bfloat16).float().numpy()
    x = np.array([int(np.argmax(vals[j])) if rng.random() < 0.8 else int(rng.integers(V))
                  for j in range(gamma)], np.int32)
    return zt, zd, x


def test_lenience_one_and_top1_are_strict_greedy(orc):
    rng = np.random.default_rng(8)
    for trial in range(40):
        zt, _, x = _random_block(rng, 8, 64, scale=0.2)   # coarse bf16 rows: many ties
        facts = orc.target_facts(zt, x)
        Lg, tg, _ = orc.verify_greedy(facts, x)
        Ll, tl, _ = orc.verify_lenient(facts, x, 1.0)
        Lk, tk, _ = orc.verify_topk(facts, x, 1)
        assert Lg == Ll == Lk
        np.testing.assert_array_equal(tg, tl)
        np.testing.assert_array_equal(tg, tk)


def test_greedy_accepts_iff_target_argmax(orc):
    rng = np.random.default_rng(9)
    for trial in range(40):
        zt, _, x = _random_block(rng, 6, 100)
        vals = torch.from_numpy(zt.view(np.int16)).view(torch.bfloat16).double()
        am = torch.argmax(vals, dim=-1).numpy()
        facts = orc.target_facts(zt, x)
        L, tok, _ = orc.verify_greedy(facts, x)
        want = next((j for j in range(6) if x[j] != am[j]), 6)
        assert L == want
        assert tok[L] == am[L]
        assert np.all(tok[L + 1:] == -1)


def test_monotone_in_ell_and_k(orc):
    rng = np.random.default_rng(10)
    ells = [1.0, 0.99, 0.975, 0.95, 0.90, 0.80, 0.70, 0.50, 0.30]   # App. A.6 grid
    for trial in range(40):
        zt, _, x = _random_block(rng, 8, 80, scale=0.3)
        facts = orc.target_facts(zt, x)
        Ls = [orc.verify_lenient(facts, x, e)[0] for e in ells]
        assert all(a <= b for a, b in zip(Ls, Ls[1:]))
        Ks = [orc.verify_topk(facts, x, k)[0] for k in (1, 2, 3, 5, 10)]
        assert all(a <= b for a, b in zip(Ks, Ks[1:]))
        assert orc.verify_greedy(facts, x)[0] <= Ks[1]


def test_lenience_threshold_closed_form(orc):
    # a drafted token 0.5 below the row max is accepted iff log(ell) <= -0.5
    V, gamma = 16, 1
    zt = np.zeros((gamma + 1, V), np.float32)
    zt[0, 3] = 2.0
    zt[0, 7] = 1.5
    x = np.array([7], np.int32)
    facts = orc.target_facts(zt, x)
    assert orc.verify_lenient(facts, x, math.exp(-0.5) - 1e-9)[0] == 1
    assert orc.verify_lenient(facts, x, math.exp(-0.5) + 1e-9)[0] == 0
    L, tok, _ = orc.verify_lenient(facts, x, 0.9)
    assert L == 0 and tok[0] == 3
    L, tok, _ = orc.verify_lenient(facts, x, 0.5)
    assert L == 1 and tok[1] == 0     # bonus = argmax of the all-zero bonus row (lowest index)


def test_agreement_metrics(orc):
    # Eq. 1-2: rounds with K=0 are excluded; K <= L counts as a full-prefix success.
    K = [0, 4, 6, 3, 0, 5]
    L = [2, 4, 2, 7, 0, 0]
    acc = orc.agreement(K, L)
    assert list(acc) == [4 + 2 + 3 + 0, 4 + 6 + 3 + 5, 1 + 0 + 1 + 0, 4]
    # Strict SDD (every committed prefix is verified, K_b = L_b): both metrics are 1
    acc = orc.agreement([3, 5, 1], [3, 5, 1])
    assert acc[0] == acc[1] and acc[2] == acc[3]


def test_acceptance_tie_accepts(orc):
    # The rule accepts iff u <= p_t/p_d; at equality the draft is kept.
    pd = np.array([[0.5, 0.5]])
    pt = np.array([[0.25, 0.75], [0.5, 0.5]])
    L, tok, mg = orc.strict_sample_probs(pt, pd, [0], [0.5], 0.5, 0.5)
    assert L == 1 and tok[0] == 0 and mg == 0.0
    L, _, _ = orc.strict_sample_probs(pt, pd, [0], [0.5 + 2 ** -24], 0.5, 0.5)
    assert L == 0
