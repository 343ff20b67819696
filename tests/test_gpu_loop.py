"""The decode loop (raw-confidence policy driving strict verification of the
blocks it does not skip, a survival-score policy in shadow, D carried across
rounds, committed tokens) against an oracle replay of the same rounds:
row statistics -> Eq. 3 schedule with D -> strict sampling on the blocks
with K = 0 -> commit."""
import numpy as np
import pytest
import torch

from paper_2608_14787_gb300 import synth
from paper_2608_14787_gb300.binding import MLP_HIDDEN
from paper_2608_14787_gb300.loop import DecodeLoop

pytestmark = pytest.mark.gpu
NEAR = 1e-6


def _bits(t):
    return synth.bf16_bits(t)


def _oracle_features(orc, st, zd, gamma, round_):
    """The scorer's scalar-feature block (App. A.7's column order; the drafter
    quantities without a counterpart here stay 0) from the oracle's row
    statistics and features, rounded to bf16 bits: [B * gamma, 256]."""
    B = st.q.shape[0]
    margin, top5 = orc.row_features(zd)
    cols = {4: st.maxprob, 5: np.log(st.maxprob), 6: st.entropy, 7: -st.entropy, 8: margin, 9: top5,
            14: np.broadcast_to(np.arange(gamma) / gamma, (B, gamma)), 15: np.full((B, gamma), round_ / 256.0)}
    f = np.zeros((B * gamma, MLP_HIDDEN), np.float32)
    for c, v in cols.items():
        f[:, c] = np.asarray(v, np.float64).reshape(-1)
    return _bits(torch.from_numpy(f).to(torch.bfloat16))


@pytest.mark.parametrize("scorer", ["deep", "mlp"])
@pytest.mark.parametrize("B,gamma,V,hidden,rounds", [(6, 8, 3008, 128, 4), (3, 32, 20016, 256, 3)])
def test_loop_matches_oracle_replay(sdd, orc, B, gamma, V, hidden, rounds, scorer):
    wl = synth.WORKLOADS["c5"]
    loop = DecodeLoop(B, gamma, V, tau=0.5, tau_mlp=0.3, K_min=2, S_max=6, seed=wl.seed, hidden=hidden, period=2,
                      scorer=scorer)
    D_raw = np.zeros(B, np.int32)
    D_mlp = np.zeros(B, np.int32)
    D_per = np.zeros(B, np.int32)
    seen_skip = seen_verify = 0
    for r in range(rounds):
        blk = synth.make_block(wl, device="cuda", round_=r, B=B, gamma=gamma, V=V)
        h = synth.make_hidden(B * gamma, device="cuda", seed=wl.seed, round_=r, hidden=hidden)
        out = loop.step(blk.z_d, blk.z_t, blk.x, h, round_=r)
        torch.cuda.synchronize()
        assert int(loop.status.item()) == 0
        zd, zt, x = _bits(blk.z_d), _bits(blk.z_t), blk.x.cpu().numpy()
        # oracle replay of the round
        st = orc.row_stats(zd, tokens=x)
        _, K_raw, D_raw, mg_raw = orc.schedule(st.q, orc.SIG_RAW, 0.5, 0.5, 2, 6, D_in=D_raw)
        if scorer == "deep":
            # the scorer on a feature block built from the oracle's own row statistics
            W1, b1, W2, b2, W3, b3, w4, b4 = loop.deep
            feat = _oracle_features(orc, st, zd, gamma, r)
            x_in = np.concatenate([_bits(h).reshape(B * gamma, -1), feat], axis=-1)
            s = orc.scorer_deep(x_in, _bits(W1), b1.cpu().numpy(), _bits(W2), b2.cpu().numpy(), _bits(W3),
                                b3.cpu().numpy(), _bits(w4), b4).reshape(B, gamma)
        else:
            s = orc.survival_mlp(_bits(h), _bits(loop.W1), loop.b1.cpu().numpy(), _bits(loop.w2),
                                 loop.b2).reshape(B, gamma)
        _, K_mlp, D_mlp, mg_mlp = orc.schedule(s, orc.SIG_CONDITIONAL, 0.3, 0.3, 2, 6, D_in=D_mlp)
        assert (mg_raw >= NEAR).all(), "near-threshold row: pick another seed"
        np.testing.assert_array_equal(out.K_raw.cpu().numpy(), K_raw)
        np.testing.assert_array_equal(loop.D_raw.cpu().numpy(), D_raw)
        # the scorer's schedule: rows whose decision lies within the scores'
        # tolerance of a threshold (a product of up to gamma scores, each within
        # 3e-4 for the deep scorer, 5e-5 for the one-layer one) are exempt, and
        # the oracle continues from the device's staleness counters
        tol = gamma * (3e-4 if scorer == "deep" else 5e-5)
        sure = mg_mlp >= tol
        np.testing.assert_array_equal(out.K_mlp.cpu().numpy()[sure], K_mlp[sure])
        np.testing.assert_array_equal(loop.D_mlp.cpu().numpy()[sure], D_mlp[sure])
        D_mlp = loop.D_mlp.cpu().numpy().astype(np.int32)
        _, K_per, D_per = orc.schedule_periodic(B, gamma, 2, 2, r, 2, 6, D_in=D_per)   # P = 2, K_skip = K_min
        np.testing.assert_array_equal(out.K_per.cpu().numpy(), K_per)
        np.testing.assert_array_equal(loop.D_per.cpu().numpy(), D_per)
        L_dev, tok_dev, n_dev = out.L.cpu().numpy(), out.tokens.cpu().numpy(), out.n.cpu().numpy()
        assert int(out.n_verified.item()) == int((K_raw == 0).sum())
        for b in range(B):
            if K_raw[b] > 0:
                seen_skip += 1
                want = np.full(gamma + 1, -1, np.int32)
                want[:K_raw[b]] = x[b, :K_raw[b]]
                np.testing.assert_array_equal(tok_dev[b], want)
                assert n_dev[b] == K_raw[b] and L_dev[b] == -2     # the verifier never saw this block
            else:
                seen_verify += 1
                L, tokens, margin = orc.verify_strict(zt[b], zd[b], x[b], seed=wl.seed, b=b, round_=r)
                assert margin >= NEAR, "near-threshold acceptance: pick another seed"
                assert L_dev[b] == L
                np.testing.assert_array_equal(tok_dev[b], tokens)
                assert n_dev[b] == L + 1
    assert seen_skip > 0 and seen_verify > 0     # both branches of the loop were exercised


def test_loop_full_size_decode_workload(sdd, orc):
    """The decode-loop workload at its stated size (B = 128, gamma = 32,
    V = 151,936 bf16, hidden 3584, the deep scorer) over three rounds with D
    carried (Sec. 4.1 loop): every block's K and D under raw confidence
    against the oracle (rows within 1e-6 of a threshold are flagged and the
    oracle continues from the device's D there), the strict verification of
    at least eight verified blocks per round (L and committed tokens), the
    periodic shadow schedule, and the deep scorer on 64 sampled positions per
    round."""
    from parity_util import row_stats_threads
    wl = synth.WORKLOADS["c5"]
    B, gamma, V = wl.B, wl.gamma, wl.V
    loop = DecodeLoop(B, gamma, V, tau=0.9, tau_mlp=0.9, K_min=6, S_max=64, seed=wl.seed, period=4, scorer="deep")
    D_raw = np.zeros(B, np.int32)
    D_per = np.zeros(B, np.int32)
    rng = np.random.default_rng(55)
    flagged = verified_checked = 0
    for r in range(3):
        blk = synth.make_block(wl, device="cuda", round_=r)
        h = synth.make_hidden(B * gamma, device="cuda", seed=wl.seed, round_=r)
        out = loop.step(blk.z_d, blk.z_t, blk.x, h, round_=r)
        torch.cuda.synchronize()
        assert int(loop.status.item()) == 0
        zd, x = _bits(blk.z_d), blk.x.cpu().numpy()
        st = row_stats_threads(zd, x)
        _, K_raw, D_next, mg = orc.schedule(st.q, orc.SIG_RAW, 0.9, 0.9, 6, 64, D_in=D_raw)
        K_dev, D_dev = out.K_raw.cpu().numpy(), loop.D_raw.cpu().numpy()
        sure = mg >= NEAR
        flagged += int((~sure).sum())
        np.testing.assert_array_equal(K_dev[sure], K_raw[sure])
        np.testing.assert_array_equal(D_dev[sure], D_next[sure])
        D_raw = D_dev.astype(np.int32)
        _, K_per, D_per = orc.schedule_periodic(B, gamma, 4, 6, r, 6, 64, D_in=D_per)
        np.testing.assert_array_equal(out.K_per.cpu().numpy(), K_per)
        np.testing.assert_array_equal(loop.D_per.cpu().numpy(), D_per)
        # strict verification of verified blocks (K = 0): the first, the last and random ones
        ver = np.flatnonzero(K_dev == 0)
        assert int(out.n_verified.item()) == ver.size
        pick = sorted(set(ver[:2].tolist() + ver[-2:].tolist() +
                          rng.choice(ver, size=min(6, ver.size), replace=False).tolist())) if ver.size else []
        assert len(pick) >= min(8, ver.size)
        zt = _bits(blk.z_t)
        L_dev, tok_dev, n_dev = out.L.cpu().numpy(), out.tokens.cpu().numpy(), out.n.cpu().numpy()
        for b in pick:
            L, tokens, margin = orc.verify_strict(zt[b], zd[b], x[b], seed=wl.seed, b=b, round_=r)
            if margin < NEAR:
                flagged += 1
                continue
            assert L_dev[b] == L and n_dev[b] == L + 1
            np.testing.assert_array_equal(tok_dev[b], tokens)
            verified_checked += 1
        for b in np.flatnonzero(K_dev > 0)[:8]:
            want = np.full(gamma + 1, -1, np.int32)
            want[:K_dev[b]] = x[b, :K_dev[b]]
            np.testing.assert_array_equal(tok_dev[b], want)
        # the deep scorer on sampled positions, its features from the oracle's statistics
        rows = rng.choice(B * gamma, size=64, replace=False)
        blk_idx, pos = rows // gamma, rows % gamma
        margin_f, top5 = orc.row_features(zd[blk_idx, pos])
        cols = {4: st.maxprob[blk_idx, pos], 5: np.log(st.maxprob[blk_idx, pos]), 6: st.entropy[blk_idx, pos],
                7: -st.entropy[blk_idx, pos], 8: margin_f, 9: top5, 14: pos / gamma, 15: np.full(64, r / 256.0)}
        f = np.zeros((64, MLP_HIDDEN), np.float32)
        for c, v in cols.items():
            f[:, c] = v
        feat = _bits(torch.from_numpy(f).to(torch.bfloat16))
        x_in = np.concatenate([_bits(h)[rows], feat], axis=-1)
        W1, b1, W2, b2, W3, b3, w4, b4 = loop.deep
        s = orc.scorer_deep(x_in, _bits(W1), b1.cpu().numpy(), _bits(W2), b2.cpu().numpy(), _bits(W3),
                            b3.cpu().numpy(), _bits(w4), b4)
        np.testing.assert_allclose(out.score.cpu().numpy().reshape(-1)[rows], s, rtol=0, atol=3e-4)
        del blk, h
    assert verified_checked >= 8
    print(f"decode workload: flagged near-threshold decisions {flagged}, verified blocks compared {verified_checked}")
