"""Pins for the oracle's prefix skip policy (Sec. 4.1 Eq. 3 and commit rule;
Sec. 4.2 signals and Eq. 4; Sec. 4.3 Eq. 5, the constant-hazard example and
Proposition 1)."""
import math

import numpy as np
import pytest

RAW, MARG, COND = 0, 1, 2


def _rand_q(rng, B, gamma, lo=0.5):
    # scores concentrated near 1 so that prefixes of every length occur
    return 1.0 - (1.0 - lo) * rng.random((B, gamma)) ** 3


def _first_below(q, eta):
    idx = np.nonzero(q < eta)[0]
    return int(idx[0]) + 1 if idx.size else q.size + 1


@pytest.mark.parametrize("sig", [RAW, MARG, COND])
def test_prefix_never_passes_first_local_failure(orc, sig):
    rng = np.random.default_rng(10)
    q = _rand_q(rng, 400, 16)
    for eb, ec in [(0.9, 0.93), (0.95, 0.8), (0.7, 0.99)]:
        Kh, K, _, _ = orc.schedule(q, sig, eb, ec, 0, 10**9)
        eta_loc = max(eb, ec) if sig == MARG else eb
        for b in range(q.shape[0]):
            assert Kh[b] <= _first_below(q[b], eta_loc) - 1


def test_raw_prefix_gate_implied_when_eta_c_le_eta_b(orc):
    # Eq. 4: min q <= geometric mean, so B_k >= eta_b >= eta_c gives C_k >= eta_c:
    # K_hat is then the first local failure minus one.
    rng = np.random.default_rng(11)
    q = _rand_q(rng, 500, 32)
    for eb, ec in [(0.9, 0.9), (0.95, 0.5), (0.8, 0.7)]:
        Kh, _, _, _ = orc.schedule(q, RAW, eb, ec, 0, 10**9)
        for b in range(q.shape[0]):
            assert Kh[b] == _first_below(q[b], eb) - 1


def test_conditional_local_gate_redundant_when_eta_c_ge_eta_b(orc):
    # Eq. 4: prod q <= min q, so the product gate implies the local gate whenever
    # eta_c >= eta_b (Sec. 4.2; App. A.3 "Product only" equals "Full").
    rng = np.random.default_rng(12)
    q = _rand_q(rng, 500, 32, lo=0.8)
    for eb, ec in [(0.9, 0.9), (0.5, 0.9), (0.85, 0.95)]:
        full, _, _, _ = orc.schedule(q, COND, eb, ec, 0, 10**9)
        prod_only, _, _, _ = orc.schedule(q, COND, 0.0, ec, 0, 10**9)
        np.testing.assert_array_equal(full, prod_only)


def test_conditional_local_gate_binds_when_eta_b_gt_eta_c(orc):
    rng = np.random.default_rng(13)
    q = _rand_q(rng, 2000, 32, lo=0.6)
    full, _, _, _ = orc.schedule(q, COND, 0.95, 0.5, 0, 10**9)
    prod_only, _, _, _ = orc.schedule(q, COND, 0.0, 0.5, 0, 10**9)
    assert np.all(full <= prod_only) and np.any(full < prod_only)


def test_marginal_collapses_to_max_threshold(orc):
    # Sec. 4.2: B_k = C_k = running min, so both gates reduce to eta_m = max(eta_b, eta_c)
    rng = np.random.default_rng(14)
    q = _rand_q(rng, 500, 32)
    for eb, ec in [(0.9, 0.95), (0.97, 0.85), (0.9, 0.9)]:
        Kh, _, _, _ = orc.schedule(q, MARG, eb, ec, 0, 10**9)
        em = max(eb, ec)
        for b in range(q.shape[0]):
            assert Kh[b] == _first_below(q[b], em) - 1
        Kh2, _, _, _ = orc.schedule(q, MARG, em, em, 0, 10**9)
        np.testing.assert_array_equal(Kh, Kh2)


@pytest.mark.parametrize("h,eta", [(0.01, 0.9), (0.003, 0.95), (0.05, 0.5), (0.02, 0.99)])
def test_constant_hazard_worked_example(orc, h, eta):
    # Sec. 4.3: constant conditional failure probability h gives a_K = (1-h)^K, while
    # multiplying the marginals a_j = (1-h)^j gives (1-h)^(K(K+1)/2).
    gamma = 64
    s = np.full((1, gamma), 1.0 - h)
    a = (1.0 - h) ** np.arange(1, gamma + 1)[None, :]
    # conditional signal on s_j: largest K with (1-h)^K >= eta
    K_cond = min(gamma, math.floor(math.log(eta) / math.log(1.0 - h)))
    Kh, _, _, _ = orc.schedule(s, COND, 0.0, eta, 0, 10**9)
    assert Kh[0] == K_cond
    # Eq. 5: the marginal signal on a_j selects the same prefix (a_K = prod s_j)
    Kh_m, _, _, _ = orc.schedule(a, MARG, 0.0, eta, 0, 10**9)
    assert Kh_m[0] == K_cond
    # multiplying marginals counts earlier survival repeatedly: K(K+1)/2 exponent
    x = math.log(eta) / math.log(1.0 - h)
    K_wrong = min(gamma, max(k for k in range(0, gamma + 1) if k * (k + 1) / 2 <= x))
    Kh_w, _, _, _ = orc.schedule(a, COND, 0.0, eta, 0, 10**9)
    assert Kh_w[0] == K_wrong
    assert K_wrong < K_cond or K_cond <= 1


def test_proposition_1_prefix_frequency(orc):
    # Prop. 1 / App. A.1: same positionwise laws, P(min_{j<=K} q >= tau) is
    # P(L>=K) rho for a shared Z and P(L>=K) rho^K for independent Z_j.
    rng = np.random.default_rng(15)
    N, gamma, rho, tau, qlo, qhi = 40000, 8, 0.6, 0.8, 0.3, 0.95
    L = np.minimum(rng.geometric(0.15, size=N) - 1, gamma)
    Y = (np.arange(1, gamma + 1)[None, :] <= L[:, None]).astype(float)
    Z = rng.random(N) < rho
    Zj = rng.random((N, gamma)) < rho
    q1 = qlo + (qhi - qlo) * Y * Z[:, None]
    q2 = qlo + (qhi - qlo) * Y * Zj
    # positionwise laws agree
    for j in range(gamma):
        assert abs(q1[:, j].mean() - q2[:, j].mean()) < 0.02
    # the local gate alone (marginal signal, eta_m = tau) gives K_hat >= K iff min_{j<=K} q >= tau
    K1, _, _, _ = orc.schedule(q1, MARG, tau, tau, 0, 10**9)
    K2, _, _, _ = orc.schedule(q2, MARG, tau, tau, 0, 10**9)
    for K in (1, 2, 4, 6):
        pL = np.mean(L >= K)
        for Kh, want in ((K1, pL * rho), (K2, pL * rho ** K)):
            got = np.mean(Kh >= K)
            sd = math.sqrt(max(want * (1 - want), 1e-12) / N)
            assert abs(got - want) < 5 * sd + 1e-3


def test_staleness_overshoot_and_reset(orc):
    # Sec. 4.1: staleness is checked before a skip, so D exceeds S_max by at most
    # gamma-1 and the next round is strict; every verifier call resets D to 0.
    rng = np.random.default_rng(16)
    B, gamma, S_max = 64, 16, 20
    D = np.zeros(B, np.int32)
    for r in range(300):
        q = _rand_q(rng, B, gamma, lo=0.85)
        Kh, K, Dn, _ = orc.schedule(q, RAW, 0.9, 0.9, 3, S_max, D_in=D)
        assert np.all(Dn <= S_max + gamma - 1)
        assert np.all(K[D >= S_max] == 0)
        assert np.all(Dn[K == 0] == 0)
        np.testing.assert_array_equal(Dn[K > 0], D[K > 0] + K[K > 0])
        D = Dn


def test_kmin_zero_still_requires_positive_khat(orc):
    q = np.array([[0.5, 0.99, 0.99], [0.99, 0.99, 0.2]])
    Kh, K, Dn, _ = orc.schedule(q, RAW, 0.9, 0.9, 0, 64, D_in=[5, 5])
    np.testing.assert_array_equal(Kh, [0, 2])
    np.testing.assert_array_equal(K, [0, 2])
    np.testing.assert_array_equal(Dn, [0, 7])
    Kh, K, Dn, _ = orc.schedule(q, RAW, 0.9, 0.9, 3, 64, D_in=[5, 5])
    np.testing.assert_array_equal(K, [0, 0])      # K_hat = 2 < K_min = 3
    np.testing.assert_array_equal(Dn, [0, 0])


def test_threshold_one_disables_skipping(orc):
    q = np.ones((8, 12))
    for sig in (RAW, MARG, COND):
        for eb, ec in [(1.0, 0.5), (0.5, 1.0), (1.0, 1.0)]:
            Kh, K, Dn, _ = orc.schedule(q, sig, eb, ec, 0, 64)
            assert np.all(K == 0) and np.all(Kh == 0) and np.all(Dn == 0)


def test_guards_and_invalid_scores(orc):
    q = np.full((3, 10), 0.99)
    q[1, 6] = np.nan
    guard = np.zeros((3, 10), np.uint8)
    guard[0, 4] = 1
    Kh, K, _, _ = orc.schedule(q, RAW, 0.9, 0.9, 0, 64, guard=guard, force_strict=[0, 0, 1])
    np.testing.assert_array_equal(Kh, [4, 6, 0])
    np.testing.assert_array_equal(K, [4, 6, 0])


def test_raw_geometric_gate_is_not_monotone(orc):
    # C_k^raw can fail at k and pass again later (Eq. 3 takes the max over all k)
    q = np.array([[0.99, 0.80, 0.999, 0.999, 0.999, 0.999]])
    Kh, _, _, _ = orc.schedule(q, RAW, 0.7, 0.95, 0, 64)
    # geometric means: k=1 .99, k=2 .889, k=3 .925, k=4 .943, k=5 .954, k=6 .962
    assert Kh[0] == 6
    Kh, _, _, _ = orc.schedule(q, RAW, 0.7, 0.96, 0, 64)
    assert Kh[0] == 6
    Kh, _, _, _ = orc.schedule(q, RAW, 0.7, 0.97, 0, 64)
    assert Kh[0] == 1


def test_margin_reports_distance_to_threshold(orc):
    q = np.array([[0.9000004, 0.95, 0.95]])
    _, _, _, mg = orc.schedule(q, MARG, 0.9, 0.9, 0, 64)
    assert mg[0] == pytest.approx(4e-7, rel=1e-3)


# ---------------------------------------------------------------------------
# Periodic skipping baseline (appendix): K_skip tokens once every P rounds
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("P", [1, 3, 4, 8])
def test_periodic_attempts_once_per_period(orc, P):
    """Over any P consecutive rounds exactly one attempt; without guards and with
    staleness far away every attempt skips K_skip tokens and the others are strict."""
    B, gamma, K_skip = 5, 32, 6
    for start in range(0, 3 * P):
        skips = 0
        for r in range(start, start + P):
            Kh, K, Do = orc.schedule_periodic(B, gamma, P, K_skip, r, 6, 10**6)
            assert (Kh == K).all() and len(set(K.tolist())) == 1
            if K[0] > 0:
                skips += 1
                assert K[0] == K_skip and r % P == P - 1
                assert (Do == K_skip).all()
            else:
                assert (Do == 0).all()
        assert skips == 1


def test_periodic_staleness_run_matches_closed_form(orc):
    """A simulated sequence: D grows by K_skip at every attempt and resets on
    every strict round, so with S_max >= K_skip every attempt skips and the
    fraction of verifier calls saved is exactly 1/P."""
    for P in (3, 4, 8):
        D = np.zeros(1, np.int32)
        calls = 0
        R = 24 * P
        for r in range(R):
            Kh, K, Do = orc.schedule_periodic(1, 32, P, 6, r, 6, 64, D_in=D)
            calls += int(K[0] == 0)
            D = Do
        assert calls == R - R // P


def test_periodic_guards_kmin_force_and_staleness(orc):
    B, gamma, P, K_skip = 4, 16, 2, 6
    guard = np.zeros((B, gamma), np.uint8)
    guard[1, 2] = 1            # guarded third position: prefix of 2
    guard[2, 7] = 1            # beyond K_skip: no effect
    force = np.array([0, 0, 0, 1], np.uint8)
    D = np.array([0, 0, 0, 0], np.int32)
    Kh, K, Do = orc.schedule_periodic(B, gamma, P, K_skip, 1, 6, 64, guard=guard, force_strict=force, D_in=D)
    assert Kh.tolist() == [6, 2, 6, 0] and K.tolist() == [6, 0, 6, 0]     # K_min = 6 cancels the short prefix
    Kh, K, Do = orc.schedule_periodic(B, gamma, P, K_skip, 1, 0, 64, guard=guard, force_strict=force, D_in=D)
    assert K.tolist() == [6, 2, 6, 0] and Do.tolist() == [6, 2, 6, 0]
    Kh, K, Do = orc.schedule_periodic(B, gamma, P, K_skip, 1, 0, 64, D_in=np.array([63, 64, 70, 0], np.int32))
    assert K.tolist() == [6, 0, 0, 6] and Do.tolist() == [69, 0, 0, 6]   # staleness: D >= S_max forces strict
    Kh, K, Do = orc.schedule_periodic(B, 4, P, K_skip, 1, 0, 64)            # gamma below K_skip
    assert K.tolist() == [4] * B
