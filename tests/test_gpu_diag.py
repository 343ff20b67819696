"""GPU parity of the offline diagnostics (sdd_permutation_diagnostic, the
Sec. 5 permutation test of Table 1, and sdd_position_metrics) against the
oracle, on synthetic score logs and on logs of the fused round itself."""
import numpy as np
import pytest
import torch

from paper_2608_14787_gb300 import synth

pytestmark = pytest.mark.gpu
LEVELS = np.array([0.5, 0.75, 0.875, 0.9375, 0.96875, 1.0], np.float32)


def _synthetic_log(B, gamma, seed):
    """Scores on a few exact levels with a block-shared factor (so positions
    within a block are dependent) and strict lengths that follow them."""
    rng = np.random.default_rng(seed)
    z = rng.normal(size=(B, 1)) + 0.6 * rng.normal(size=(B, gamma))
    q = LEVELS[np.clip(np.digitize(z, [-1.2, -0.6, 0.0, 0.6, 1.2]), 0, 5)]
    L = np.array([next((j for j in range(gamma) if q[b, j] < 0.9), gamma) for b in range(B)], np.int32)
    return q, L


@pytest.mark.parametrize("signal,eta_b,eta_c", [(0, 0.90, 0.93), (1, 0.90, 0.90), (2, 0.90, 0.90)])
def test_permutation_diagnostic_vs_oracle(sdd, orc, signal, eta_b, eta_c):
    q, L = _synthetic_log(257, 20, signal)
    sums = sdd.permutation_diagnostic(torch.from_numpy(q).cuda(), torch.from_numpy(L).cuda(), signal=signal,
                                      eta_b=eta_b, eta_c=eta_c, n_rep=24, seed=9)
    torch.cuda.synchronize()
    want = orc.permutation_diagnostic(q.astype(np.float64), L, signal, eta_b, eta_c, 24, 9)
    np.testing.assert_array_equal(sums.cpu().numpy(), want)
    assert want[:-1].mean() < want[-1]           # the dependence the permutation breaks


@pytest.mark.parametrize("signal", [0, 2])
def test_permutation_diagnostic_long_log_vs_oracle(sdd, orc, signal):
    """A log longer than the parallel shuffle's limit (4096 blocks): the serial
    swap loop, also when few blocks remain valid (conditional signal, late
    positions)."""
    q, L = _synthetic_log(4500, 12, 5 + signal)
    sums = sdd.permutation_diagnostic(torch.from_numpy(q).cuda(), torch.from_numpy(L).cuda(), signal=signal,
                                      eta_b=0.90, eta_c=0.90, n_rep=3, seed=4)
    torch.cuda.synchronize()
    want = orc.permutation_diagnostic(q.astype(np.float64), L, signal, 0.90, 0.90, 3, 4)
    np.testing.assert_array_equal(sums.cpu().numpy(), want)


def test_position_metrics_vs_oracle(sdd, orc):
    q, L = _synthetic_log(300, 16, 5)
    qd, Ld = torch.from_numpy(q).cuda(), torch.from_numpy(L).cuda()
    for cond in (False, True):
        bce, base, auc, npos, nneg = sdd.position_metrics(qd, Ld, conditional=cond)
        torch.cuda.synchronize()
        wb, wbase, wauc, wp, wn = orc.position_metrics(q.astype(np.float64), L, cond)
        np.testing.assert_allclose(bce.cpu().numpy(), wb, rtol=1e-10, equal_nan=True)
        np.testing.assert_allclose(base.cpu().numpy(), wbase, rtol=1e-10, atol=1e-15, equal_nan=True)
        np.testing.assert_allclose(auc.cpu().numpy(), wauc, rtol=1e-12, equal_nan=True)
        np.testing.assert_array_equal(npos.cpu().numpy(), wp)
        np.testing.assert_array_equal(nneg.cpu().numpy(), wn)


def test_diagnostics_on_logged_rounds(sdd, orc):
    """Logs of the fused round (raw confidence and shadow-verified strict L)
    over several rounds of a small workload: the diagnostic's sums and the
    metrics' counts match the oracle on the same log."""
    B, gamma, V = 16, 16, 4096
    rnd = sdd.BlockRound(B, gamma, V, taus=(0.9,), K_min=6, S_max=64)
    qs, Ls = [], []
    for r in range(6):
        blk = synth.make_block("c3", device="cuda", B=B, gamma=gamma, V=V, round_=r)
        rnd.set_inputs(blk.z_d, blk.z_t, blk.x, seed=3, round_=r)
        rnd.run()
        qs.append(rnd.q.clone())
        Ls.append(rnd.L_strict.clone())
    q, L = torch.cat(qs), torch.cat(Ls)
    torch.cuda.synchronize()
    sums = sdd.permutation_diagnostic(q, L, signal=0, eta_b=0.9, eta_c=0.93, n_rep=16, seed=1)
    _, _, _, npos, nneg = sdd.position_metrics(q, L)
    torch.cuda.synchronize()
    want = orc.permutation_diagnostic(q.double().cpu().numpy(), L.cpu().numpy(), 0, 0.9, 0.93, 16, 1)
    np.testing.assert_array_equal(sums.cpu().numpy(), want)
    _, _, _, wp, wn = orc.position_metrics(q.double().cpu().numpy(), L.cpu().numpy(), False)
    np.testing.assert_array_equal(npos.cpu().numpy(), wp)
    np.testing.assert_array_equal(nneg.cpu().numpy(), wn)
