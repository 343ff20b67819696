"""GPU parity: every entry point of the C ABI against the fp64 oracle on the
same seeded inputs, at sizes the oracle finishes in seconds (several tiles per
row, ragged tails), plus the edge cases of the method."""
import math

import numpy as np
import pytest
import torch

import oracle as orc
from paper_2608_14787_gb300 import synth
from parity_util import Tally, assert_close_logratio, assert_close_stats, compare_rule, host, oracle_block

pytestmark = pytest.mark.gpu

DEV = "cuda"


def _to_dev(blk):
    return blk.z_d.to(DEV), blk.z_t.to(DEV), blk.x.to(DEV)


def _padded(z: torch.Tensor, stride: int) -> torch.Tensor:
    """Same logits with each row padded to `stride` elements (padding = +inf,
    which the library must never read into a result)."""
    B, P, V = z.shape
    buf = torch.full((B, P, stride), float("inf"), dtype=z.dtype, device=z.device)
    buf[..., :V] = z
    return buf[..., :V]


# ---------------------------------------------------------------------------
# confidence (Sec. 4.2)
# ---------------------------------------------------------------------------

def _check_confidence(sdd, z_d, x, dtype):
    out = sdd.confidence(z_d, x)
    torch.cuda.synchronize()
    st = orc.row_stats(host(z_d.contiguous() if z_d.is_contiguous() else z_d), tokens=x.cpu().numpy())
    errs = {}
    errs["q"] = assert_close_stats("q", out.q, st.q, dtype)
    errs["logq"] = assert_close_logratio("logq", out.logq, st.logq, dtype)
    errs["maxprob"] = assert_close_stats("maxprob", out.maxprob, st.maxprob, dtype)
    errs["lse"] = assert_close_stats("lse", out.lse, st.lse, dtype)
    errs["entropy"] = assert_close_stats("entropy", out.entropy, st.entropy, dtype)
    np.testing.assert_array_equal(out.argmax.cpu().numpy(), st.argmax)
    return errs


def test_confidence_tiny_fp32(sdd):
    blk = synth.make_block("tiny", device="cpu")
    z_d, z_t, x = _to_dev(blk)
    errs = _check_confidence(sdd, z_d, x, torch.float32)
    print("tiny fp32 max rel errors:", errs)


@pytest.mark.parametrize("B,gamma,V", [(3, 5, 1003), (2, 7, 8), (1, 3, 1), (4, 33, 20011), (2, 64, 4096)])
def test_confidence_bf16_shapes(sdd, B, gamma, V):
    blk = synth.make_block("c3", device="cpu", B=B, gamma=gamma, V=V)
    z_d, z_t, x = _to_dev(blk)
    stride = ((V + 7) // 8) * 8
    zp = _padded(z_d, stride) if stride != V else z_d
    errs = _check_confidence(sdd, zp, x, torch.bfloat16)
    print(f"bf16 B={B} gamma={gamma} V={V} max rel errors:", errs)


def test_confidence_fp32_ragged(sdd):
    blk = synth.make_block("tiny", device="cpu", B=3, gamma=4, V=1001)
    z_d, _, x = _to_dev(blk)
    _check_confidence(sdd, _padded(z_d, 1004), x, torch.float32)


def test_confidence_nonfinite_and_bad_tokens(sdd):
    blk = synth.make_block("c3", device="cpu", B=2, gamma=4, V=3000)
    z_d, _, x = _to_dev(blk)
    z_d = z_d.clone()
    z_d[0, 1, 17] = float("nan")
    z_d[1, 2, 5] = float("inf")
    z_d[1, 3, :] = float("-inf")
    x = x.clone()
    x[0, 3] = 3000          # out of range
    status = sdd.new_status()
    out = sdd.confidence(z_d, x, status=status)
    torch.cuda.synchronize()
    s = int(status.item())
    assert s & sdd.DEV_NONFINITE and s & sdd.DEV_BAD_TOKEN
    q = out.q.cpu()
    assert math.isnan(q[0, 1]) and math.isnan(q[1, 2]) and math.isnan(q[1, 3]) and math.isnan(q[0, 3])
    assert out.argmax[0, 1].item() == -1 and out.argmax[1, 3].item() == -1
    # untouched rows still agree with the oracle
    st = orc.row_stats(host(z_d), tokens=np.clip(x.cpu().numpy(), 0, 2999))
    assert q[0, 0].item() == pytest.approx(st.q[0, 0], rel=2e-3)
    # masked (-inf) entries in an otherwise finite row are fine
    z2 = z_d.clone()
    z2[0, 0, :100] = float("-inf")
    x2 = x.clone()
    x2[0, 0] = 500
    out2 = sdd.confidence(z2, x2)
    st2 = orc.row_stats(host(z2[:1, :1]), tokens=x2[:1, :1].cpu().numpy())
    assert out2.entropy[0, 0].item() == pytest.approx(st2.entropy[0, 0], rel=2e-3)
    assert out2.q[0, 0].item() == pytest.approx(st2.q[0, 0], rel=2e-3)


def test_confidence_deterministic(sdd):
    blk = synth.make_block("c3", device="cpu", B=4, gamma=16, V=50000)
    z_d, _, x = _to_dev(blk)
    a = sdd.confidence(z_d, x)
    b = sdd.confidence(z_d, x)
    for f in ("q", "logq", "maxprob", "lse", "entropy", "argmax"):
        assert torch.equal(getattr(a, f), getattr(b, f)), f


# ---------------------------------------------------------------------------
# schedule (Sec. 4.1 Eq. 3)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("signal", [0, 1, 2])
def test_schedule_vs_oracle(sdd, signal):
    rng = np.random.default_rng(100 + signal)
    B, gamma = 257, 40
    q = (1.0 - 0.35 * rng.random((B, gamma)) ** 4).astype(np.float32)
    q[rng.random((B, gamma)) < 0.01] = np.nan
    guard = (rng.random((B, gamma)) < 0.02).astype(np.uint8)
    force = (rng.random(B) < 0.05).astype(np.uint8)
    D = rng.integers(0, 80, size=B).astype(np.int32)
    pairs = [(0.9, 0.93), (0.95, 0.9), (0.8, 0.85), (0.7, 0.7), (0.9, 1.0), (0.99, 0.995), (0.6, 0.5),
             (0.0, 0.9), (0.9, 0.0)]
    K_min, S_max = 3, 64
    dq = torch.from_numpy(q).to(DEV)
    Kh, K, Do = sdd.schedule_prefix(dq, [p[0] for p in pairs], [p[1] for p in pairs], signal=signal, K_min=K_min,
                                    S_max=S_max, guard=torch.from_numpy(guard).to(DEV),
                                    force_strict=torch.from_numpy(force).to(DEV), D_in=torch.from_numpy(D).to(DEV))
    torch.cuda.synchronize()
    tally = Tally()
    for t, (eb, ec) in enumerate(pairs):
        oKh, oK, oD, mg = orc.schedule(q.astype(np.float64), signal, eb, ec, K_min, S_max, guard=guard,
                                       force_strict=force, D_in=D)
        for b in range(B):
            ok = (Kh[t, b].item() == oKh[b]) and (K[t, b].item() == oK[b]) and (Do[t, b].item() == oD[b])
            tally.check(f"signal {signal} pair {(eb, ec)} block {b}", ok, mg[b])
    print("schedule", signal, tally)


# ---------------------------------------------------------------------------
# verification rules (Sec. 3.1, App. A.6)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("wl,B,gamma,V,greedy_drafts", [
    ("c3", 6, 12, 5003, False), ("c3", 5, 9, 30000, True), ("c2", 2, 16, 20000, False), ("tiny", 3, 8, 4001, False),
])
def test_verify_rules_vs_oracle(sdd, wl, B, gamma, V, greedy_drafts):
    blk = synth.make_block(wl, device="cpu", B=B, gamma=gamma, V=V, greedy_drafts=greedy_drafts,
                           dtype=torch.float32 if wl == "tiny" else torch.bfloat16)
    z_d, z_t, x = _to_dev(blk)
    stride = ((V + 7) // 8) * 8
    if stride != V:
        z_d, z_t = _padded(z_d, stride), _padded(z_t, stride)
    ells = (1.0, 0.9, 0.5, 0.25)
    ks = (1, 2, 5, 10)
    seed, rnd = 1234, 7
    draft = sdd.confidence(z_d, x)
    Ls, tks, _ = sdd.verify_strict(z_t, x, z_d=z_d, draft=draft, greedy=False, seed=seed, round_=rnd)
    Lg, tkg, _ = sdd.verify_strict(z_t, x, greedy=True)
    Ll, tkl, _ = sdd.verify_lenient(z_t, x, ells)
    Lk, tkk, _ = sdd.verify_topk(z_t, x, ks)
    torch.cuda.synchronize()
    ob = oracle_block(z_d, z_t, x, seed=seed, round_=rnd, ells=ells, ks=ks)
    blocks = list(range(B))
    tally = Tally()
    compare_rule(tally, "strict-sampling", Ls, tks, ob.strict, blocks)
    compare_rule(tally, "strict-greedy", Lg, tkg, ob.greedy, blocks)
    for r, e in enumerate(ells):
        compare_rule(tally, f"lenient {e}", Ll[r], tkl[r], ob.lenient[e], blocks)
    for r, k in enumerate(ks):
        compare_rule(tally, f"top-{k}", Lk[r], tkk[r], ob.topk[k], blocks)
    print(wl, tally)
    assert tally.compared == B * (2 + len(ells) + len(ks))


def test_verify_row_subset(sdd):
    blk = synth.make_block("c3", device="cpu", B=8, gamma=10, V=4096)
    z_d, z_t, x = _to_dev(blk)
    rows = torch.tensor([6, 1, 3], dtype=torch.int32, device=DEV)
    draft = sdd.confidence(z_d, x)
    L, tok, n = sdd.verify_strict(z_t, x, z_d=z_d, draft=draft, seed=5, round_=2, rows=rows)
    torch.cuda.synchronize()
    ob = oracle_block(z_d, z_t, x, seed=5, round_=2, blocks=[6, 1, 3])
    tally = Tally()
    compare_rule(tally, "subset", L, tok, ob.strict, [6, 1, 3])
    untouched = [b for b in range(8) if b not in (6, 1, 3)]
    assert torch.all(L[untouched] == -2) and torch.all(tok[untouched] == -2) and torch.all(n[untouched] == -2)


def test_workspace_reused_across_shapes(sdd):
    """One workspace serves stream-ordered calls of different shapes in any
    order: sampling verifications (which use the draw's arrival counters) at
    (B, gamma) = (24, 12), (5, 3), (24, 12), (9, 7) on the same workspace, each
    against the oracle.  The smaller calls' counters fall on bytes that the
    larger calls used for other scratch."""
    ws = sdd.Workspace(24, 12, 4096, DEV)
    tally = Tally()
    for B, gamma, r in [(24, 12, 1), (5, 3, 2), (24, 12, 3), (9, 7, 4)]:
        blk = synth.make_block("c3", device="cpu", B=B, gamma=gamma, V=4096, round_=r)
        z_d, z_t, x = _to_dev(blk)
        draft = sdd.confidence(z_d, x, ws=ws)
        L, tok, n = sdd.verify_strict(z_t, x, z_d=z_d, draft=draft, seed=11, round_=r, ws=ws)
        torch.cuda.synchronize()
        ob = oracle_block(z_d, z_t, x, seed=11, round_=r)
        compare_rule(tally, f"ws-reuse B={B} gamma={gamma}", L, tok, ob.strict, range(B))
        np.testing.assert_array_equal(n.cpu().numpy(), L.cpu().numpy() + 1)


def test_identical_rows_accept_everything(sdd):
    blk = synth.make_block("c3", device="cpu", B=16, gamma=16, V=8192)
    z_d, _, x = _to_dev(blk)
    z_t = torch.cat([z_d, z_d[:, -1:]], dim=1).contiguous()
    draft = sdd.confidence(z_d, x)
    L, tok, n = sdd.verify_strict(z_t, x, z_d=z_d, draft=draft, seed=9, round_=0)
    Lg, tokg, ng = sdd.verify_strict(z_t, x, greedy=True)
    torch.cuda.synchronize()
    # p_t = p_d always accepts (Sec. 3.1).  The two rows' LSE are computed from
    # the same logits along different warp splits, so log p_t - log p_d is the
    # difference of two double-float roundings (|.| <~ 1e-9), far inside the
    # 6e-8 gap between the largest uniform (1 - 2^-24) and 1: every position
    # accepts and the bonus token comes from row gamma + 1.
    assert torch.all(L == 16), L
    assert torch.all(n == 17)
    np.testing.assert_array_equal(tok[:, :16].cpu().numpy(), x.cpu().numpy())
    ob = oracle_block(z_d, z_t, x, seed=9, round_=0)
    tally = Tally()
    compare_rule(tally, "identical", L, tok, ob.strict, range(16))
    compare_rule(tally, "identical-greedy", Lg, tokg, ob.greedy, range(16))
    np.testing.assert_array_equal(ng.cpu().numpy(), Lg.cpu().numpy() + 1)


def test_philox_device_matches_oracle(sdd):
    n = 1 << 20
    rng = np.random.default_rng(3)
    j = rng.integers(0, 1 << 32, size=n, dtype=np.uint64).astype(np.uint32)
    b = rng.integers(0, 1 << 32, size=n, dtype=np.uint64).astype(np.uint32)
    r = rng.integers(0, 1 << 62, size=n, dtype=np.uint64)
    p = rng.integers(0, 4, size=n).astype(np.uint32)
    seed = 0xDEADBEEF12345678
    u = sdd.uniforms(seed, torch.from_numpy(j.view(np.int32)).to(DEV), torch.from_numpy(b.view(np.int32)).to(DEV),
                     torch.from_numpy(r.view(np.int64)).to(DEV), torch.from_numpy(p.view(np.int32)).to(DEV))
    want = orc.uniform_many(seed, j, b, r, p)
    np.testing.assert_array_equal(u.cpu().numpy().astype(np.float64), want)


# ---------------------------------------------------------------------------
# fused round
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("greedy", [False, True])
def test_block_round_vs_oracle(sdd, greedy):
    B, gamma, V = 12, 16, 12007
    blk = synth.make_block("c3", device="cpu", B=B, gamma=gamma, V=V, greedy_drafts=greedy)
    z_d, z_t, x = _to_dev(blk)
    z_d, z_t = _padded(z_d, 12008), _padded(z_t, 12008)
    taus = (0.5, 0.9, 0.95, 1.0)
    ells, ks = (1.0, 0.5), (2, 5)
    rnd = sdd.BlockRound(B, gamma, V, taus=taus, ells=ells, ks=ks, greedy=greedy, K_min=2, S_max=64)
    D = torch.randint(0, 70, (B,), dtype=torch.int32)
    rnd.D_in.copy_(D)
    rnd.set_inputs(z_d, z_t, x, seed=77, round_=3)
    rnd.run()
    torch.cuda.synchronize()
    assert int(rnd.status.item()) == 0
    ob = oracle_block(z_d, z_t, x, seed=77, round_=3, pairs=[(t, t) for t in taus], K_min=2, S_max=64,
                      D_in=D.numpy(), ells=ells, ks=ks, sampling=not greedy)
    assert_close_stats("q", rnd.q, ob.stats.q, torch.bfloat16)
    assert_close_stats("entropy", rnd.entropy, ob.stats.entropy, torch.bfloat16)
    np.testing.assert_array_equal(rnd.argmax.cpu().numpy(), ob.stats.argmax)
    blocks = list(range(B))
    tally = Tally()
    compare_rule(tally, "strict", rnd.L_strict, rnd.tokens_strict, ob.greedy if greedy else ob.strict, blocks)
    for r, e in enumerate(ells):
        compare_rule(tally, f"lenient {e}", rnd.L_lenient[r], rnd.tokens_lenient[r], ob.lenient[e], blocks)
    for r, k in enumerate(ks):
        compare_rule(tally, f"top-{k}", rnd.L_topk[r], rnd.tokens_topk[r], ob.topk[k], blocks)
    L_or = np.array([(ob.greedy if greedy else ob.strict)[b][0] for b in blocks])
    acc_want = np.zeros((len(taus), 4), np.int64)
    for t, tau in enumerate(taus):
        oKh, oK, oD, mg = ob.sched[(tau, tau)]
        for b in blocks:
            ok = (rnd.K_hat[t, b].item() == oKh[b] and rnd.K[t, b].item() == oK[b] and rnd.D_out[t, b].item() == oD[b])
            tally.check(f"schedule tau {tau} block {b}", ok, mg[b])
        acc_want[t] = orc.agreement(oK, L_or)
    np.testing.assert_array_equal(rnd.agreement.cpu().numpy(), acc_want)
    # committed tokens under pair 0
    oK0 = ob.sched[(taus[0], taus[0])][1]
    ct = rnd.commit_tokens.cpu().numpy()
    cn = rnd.commit_n.cpu().numpy()
    xs = x.cpu().numpy()
    for b in blocks:
        if oK0[b] > 0:
            assert cn[b] == oK0[b] and np.array_equal(ct[b][:oK0[b]], xs[b][:oK0[b]]) and np.all(ct[b][oK0[b]:] == -1)
        else:
            L, tok, _ = (ob.greedy if greedy else ob.strict)[b]
            assert cn[b] == L + 1 and np.array_equal(ct[b], tok)
    print("block round", tally)
    # tau = 1 reproduces Strict SDD with zero skips
    assert torch.all(rnd.K[3] == 0)


@pytest.mark.parametrize("sigma", [0.2, 0.05, 0.01])
def test_strict_sampling_small_residuals(sdd, sigma):
    """Target = drafter + N(0, sigma): p_t is close to p_d, so the residual mass
    R of a rejection is small and made of nearly cancelling terms (on peaked
    positions R is of order 1e-4).  The draws must still match the oracle."""
    B, gamma, V = 24, 12, 30000
    blk = synth.make_block("c3", device="cpu", B=B, gamma=gamma, V=V)
    g = torch.Generator().manual_seed(int(sigma * 10000))
    zt = blk.z_t.float().clone()
    zt[:, :gamma] = blk.z_d.float() + sigma * torch.randn(B, gamma, V, generator=g)
    z_t = zt.to(torch.bfloat16).contiguous().to(DEV)
    z_d, x = blk.z_d.to(DEV), blk.x.to(DEV)
    draft = sdd.confidence(z_d, x)
    tally = Tally()
    for rnd in range(3):
        L, tok, _ = sdd.verify_strict(z_t, x, z_d=z_d, draft=draft, seed=17, round_=rnd)
        torch.cuda.synchronize()
        ob = oracle_block(z_d, z_t, x, seed=17, round_=rnd)
        compare_rule(tally, f"strict sigma={sigma} round {rnd}", L, tok, ob.strict, list(range(B)))
    print("small residuals", sigma, tally)


def test_topk_and_greedy_with_tied_logits(sdd):
    """Ranks with exact ties (App. A.6 top-k, greedy strict): target rows hold a
    few entries above the drafted token's logit and a dozen exactly equal to it,
    on both sides of the token, so the index tie-break decides the rank."""
    B, gamma, V = 4, 6, 6000
    g = torch.Generator().manual_seed(77)
    z_t = torch.full((B, gamma + 1, V), -4.0)
    x = torch.zeros((B, gamma), dtype=torch.int32)
    for b in range(B):
        for j in range(gamma + 1):
            pos = torch.randperm(V, generator=g)[:15]
            z_t[b, j, pos[:3]] = 2.0 + j % 2       # above the tie level (or two maxima ties)
            z_t[b, j, pos[3:]] = 1.0 if j % 3 else 2.0 + j % 2
            if j < gamma:
                x[b, j] = int(pos[3 + (b * 7 + j * 5) % 12])
    z_t = z_t.to(torch.bfloat16)
    z_d = torch.randn((B, gamma, V), generator=g).to(torch.bfloat16)
    z_d, z_t, x = z_d.to(DEV), z_t.to(DEV), x.to(DEV)
    ks = (1, 2, 5, 10)
    Lg, tkg, _ = sdd.verify_strict(z_t, x, greedy=True)
    Lk, tkk, _ = sdd.verify_topk(z_t, x, ks)
    torch.cuda.synchronize()
    ob = oracle_block(z_d, z_t, x, ks=ks, sampling=False)
    tally = Tally()
    compare_rule(tally, "strict-greedy", Lg, tkg, ob.greedy, list(range(B)))
    for r, k in enumerate(ks):
        compare_rule(tally, f"top-{k}", Lk[r], tkk[r], ob.topk[k], list(range(B)))
    assert tally.compared == B * (1 + len(ks)) and tally.flagged == 0


# ---------------------------------------------------------------------------
# periodic skipping baseline (appendix): stand-alone and in the fused round
# ---------------------------------------------------------------------------

def test_schedule_periodic_vs_oracle(sdd):
    B, gamma = 37, 40                     # two warp chunks of positions
    g = torch.Generator().manual_seed(5)
    guard = (torch.rand(B, gamma, generator=g) < 0.03).to(torch.uint8)
    force = (torch.rand(B, generator=g) < 0.1).to(torch.uint8)
    D = torch.randint(0, 80, (B,), generator=g, dtype=torch.int32)
    periods = (1, 3, 4, 8)
    for round_ in range(10):
        for K_min, K_skip in ((6, 6), (0, 6), (2, 45)):
            Kh, K, Do = sdd.schedule_periodic(B, gamma, periods, K_skip=K_skip, round_=round_, K_min=K_min,
                                              S_max=64, guard=guard.to(DEV), force_strict=force.to(DEV),
                                              D_in=D.to(DEV))
            torch.cuda.synchronize()
            for t, P in enumerate(periods):
                oKh, oK, oD = orc.schedule_periodic(B, gamma, P, K_skip, round_, K_min, 64, guard=guard.numpy(),
                                                    force_strict=force.numpy(), D_in=D.numpy())
                np.testing.assert_array_equal(Kh[t].cpu().numpy(), oKh)
                np.testing.assert_array_equal(K[t].cpu().numpy(), oK)
                np.testing.assert_array_equal(Do[t].cpu().numpy(), oD)


@pytest.mark.parametrize("round_", [2, 3])
def test_block_round_periodic_vs_oracle(sdd, round_):
    B, gamma, V = 6, 16, 4096
    blk = synth.make_block("c3", device="cpu", B=B, gamma=gamma, V=V)
    z_d, z_t, x = _to_dev(blk)
    periods = (2, 3, 4)
    rnd = sdd.BlockRound(B, gamma, V, signal=sdd.SIG_PERIODIC, periods=periods, K_skip=6, K_min=6, S_max=64)
    D = torch.tensor([0, 5, 60, 64, 70, 10], dtype=torch.int32)
    rnd.D_in.copy_(D)
    rnd.set_inputs(z_d, z_t, x, seed=11, round_=round_)
    rnd.run()
    torch.cuda.synchronize()
    assert int(rnd.status.item()) == 0
    ob = oracle_block(z_d, z_t, x, seed=11, round_=round_)
    tally = Tally()
    compare_rule(tally, "strict", rnd.L_strict, rnd.tokens_strict, ob.strict, list(range(B)))
    xs = x.cpu().numpy()
    for t, P in enumerate(periods):
        oKh, oK, oD = orc.schedule_periodic(B, gamma, P, 6, round_, 6, 64, D_in=D.numpy())
        np.testing.assert_array_equal(rnd.K_hat[t].cpu().numpy(), oKh)
        np.testing.assert_array_equal(rnd.K[t].cpu().numpy(), oK)
        np.testing.assert_array_equal(rnd.D_out[t].cpu().numpy(), oD)
    oK0 = orc.schedule_periodic(B, gamma, periods[0], 6, round_, 6, 64, D_in=D.numpy())[1]
    ct, cn = rnd.commit_tokens.cpu().numpy(), rnd.commit_n.cpu().numpy()
    for b in range(B):
        if oK0[b] > 0:
            assert cn[b] == 6 and np.array_equal(ct[b][:6], xs[b][:6]) and np.all(ct[b][6:] == -1)
        else:
            L, tok, _ = ob.strict[b]
            assert cn[b] == L + 1 and np.array_equal(ct[b], tok)
    assert tally.flagged_mismatch == 0


# ---------------------------------------------------------------------------
# extended features (App. A.7): probability margin and top-5 mass
# ---------------------------------------------------------------------------

def _check_features(sdd, z_d, x, dtype):
    base = sdd.confidence(z_d, x)
    out = sdd.confidence(z_d, x, features=True)
    torch.cuda.synchronize()
    for f in ("q", "logq", "maxprob", "lse", "entropy", "argmax"):   # the feature pass changes nothing else
        torch.testing.assert_close(getattr(out, f), getattr(base, f), rtol=0, atol=0, equal_nan=True, msg=f)
    mg, t5 = orc.row_features(host(z_d.contiguous() if z_d.is_contiguous() else z_d))
    p1 = orc.row_stats(host(z_d)).maxprob
    # margin = p1 - p2 cancels: hold it to the tolerance of p1
    g = out.margin.cpu().double().numpy()
    both = np.isnan(g) & np.isnan(mg)
    assert (np.isnan(g) == np.isnan(mg)).all()
    err = np.abs(g - mg)[~both]
    assert (err <= (2e-3 if dtype == torch.bfloat16 else 1e-5) * np.abs(p1[~both]) + 1e-7).all(), err.max()
    assert_close_stats("top5", out.top5, t5, dtype)


@pytest.mark.parametrize("B,gamma,V", [(4, 16, 50000), (3, 5, 151936), (2, 33, 4096), (8, 3, 17)])
def test_features_bf16_vs_oracle(sdd, B, gamma, V):
    blk = synth.make_block("c3", device="cpu", B=B, gamma=gamma, V=V)
    z_d, _, x = _to_dev(blk)
    z_d = z_d.clone()
    z_d[0, 0, :] = z_d[0, 0].max()                 # a row of ties: margin 0, top5 = 5 / V
    z_d[0, 1, 5:] = float("-inf")                  # five finite entries
    if gamma > 2:
        z_d[0, 2, 3] = float("nan")                # no distribution
    if V % 8:
        z_d = _padded(z_d, (V + 7) // 8 * 8)       # 16-byte row stride
    _check_features(sdd, z_d, x, torch.bfloat16)


def test_features_fp32_padded_rows(sdd):
    blk = synth.make_block("tiny", device="cpu", B=3, gamma=8, V=4001, dtype=torch.float32)
    z_d, _, x = _to_dev(blk)
    z_d = _padded(z_d, 4004)
    _check_features(sdd, z_d, x, torch.float32)


@pytest.mark.parametrize("V", [151936, 20003])
def test_features_planted_top5_layouts(sdd, V):
    """The five largest entries placed where the selection of lane-tile groups
    (a lane's 8 vectors of one tile) is tested: all five in one 16-byte vector,
    one per 2048-entry tile, in the row's last (partial) vector, four tied
    below the maximum in different groups, and a row whose maximum ties six
    times (one tie outside the five selected groups)."""
    blk = synth.make_block("c3", device="cpu", B=2, gamma=6, V=V)
    z_d, _, x = _to_dev(blk)
    z_d = z_d.clone()
    top = 30.0
    r = z_d[0]
    r[0, 1000:1005] = torch.tensor([top, top - 1, top - 2, top - 3, top - 4])     # one vector (8-aligned start)
    for k in range(5):
        r[1, k * 2048 + 37 * k] = top - k                                              # one per tile
    r[2, V - 5:] = torch.tensor([top - 4, top - 3, top - 2, top - 1, top])        # the row's end
    r[3, 3] = top
    for k, pos in enumerate((9000, 17000, 41000 % V, 77000 % V)):
        r[3, pos] = top - 1                                                          # ties below the max
    for k in range(6):
        r[4, 3000 * k + 5] = top                                                     # the maximum six times
    r[5, :] = r[5].clamp(max=0.0)
    r[5, 123] = 1.0                                                                  # a single positive entry
    if V % 8:
        z_d = _padded(z_d, (V + 7) // 8 * 8)
    _check_features(sdd, z_d, x, torch.bfloat16)


def test_entropy_of_peaked_fp32_rows(sdd):
    """fp32 rows with one token 8 nats above the rest (entropy ~ 6e-3): the
    entropy is a difference of two terms of order one unless it is accumulated
    against the row maximum; it must hold the fp32 tolerance (1e-5 relative)
    in the confidence call and in the fused round."""
    blk = synth.make_block("c3", device="cpu", B=6, gamma=16, V=20_008, dtype=torch.float32, greedy_drafts=True)
    z_d, z_t, x = _to_dev(blk)
    conf = sdd.confidence(z_d, x)
    rnd = sdd.BlockRound(6, 16, 20_008, dtype=torch.float32, taus=(0.9,), K_min=2)
    rnd.set_inputs(z_d, z_t, x, seed=1, round_=0)
    rnd.run()
    torch.cuda.synchronize()
    st = orc.row_stats(blk.z_d.numpy(), tokens=blk.x.numpy())
    assert (st.entropy < 0.05).mean() > 0.25    # the workload's peaked rows
    assert_close_stats("entropy", conf.entropy, st.entropy, torch.float32)
    assert_close_stats("entropy", rnd.entropy, st.entropy, torch.float32)


@pytest.mark.parametrize("frac", [0.0, 0.4, 1.0])
def test_select_rows_and_listed_verify(sdd, frac):
    """The verifier's block list selected on the device (K == 0) and verified
    with its count read there equals sdd_verify_strict on the host list;
    unlisted blocks keep their previous contents."""
    B, gamma, V = 21, 10, 6000
    blk = synth.make_block("c3", device="cpu", B=B, gamma=gamma, V=V)
    z_d, z_t, x = _to_dev(blk)
    g = torch.Generator().manual_seed(int(frac * 10))
    K = torch.where(torch.rand(B, generator=g) < frac, torch.zeros(B, dtype=torch.int32),
                    torch.randint(1, gamma + 1, (B,), generator=g, dtype=torch.int32)).to(DEV)
    rows, n = sdd.select_rows(K)
    draft = sdd.confidence(z_d, x)
    L, tok, nc = sdd.verify_strict_listed(z_t, x, rows, n, z_d=z_d, draft=draft, seed=4, round_=9)
    torch.cuda.synchronize()
    want_rows = torch.nonzero(K == 0).flatten().to(torch.int32)
    assert int(n.item()) == want_rows.numel()
    assert torch.equal(rows[:want_rows.numel()], want_rows)
    if want_rows.numel():
        L2, tok2, nc2 = sdd.verify_strict(z_t, x, z_d=z_d, draft=draft, seed=4, round_=9, rows=want_rows)
        torch.cuda.synchronize()
        assert torch.equal(L, L2) and torch.equal(tok, tok2) and torch.equal(nc, nc2)
        ob = oracle_block(z_d, z_t, x, seed=4, round_=9, blocks=want_rows.cpu().tolist())
        compare_rule(Tally(), "listed", L, tok, ob.strict, want_rows.cpu().tolist())
    skipped = (K != 0).nonzero().flatten()
    assert torch.all(L[skipped] == -2) and torch.all(tok[skipped] == -2)


def test_listed_verify_few_blocks_full_vocabulary(sdd):
    """Two of 24 blocks listed at V = 151,936: the decide grid, cut on the
    device from the count, gives each listed block many draw segments (38),
    the same cut as a host list of those two blocks; the results equal
    sdd_verify_strict's on the host list bit for bit, and the oracle's."""
    B, gamma, V = 24, 8, 151_936
    blk = synth.make_block("c3", device="cpu", B=B, gamma=gamma, V=V)
    z_d, z_t, x = _to_dev(blk)
    K = torch.full((B,), 3, dtype=torch.int32)
    K[5] = 0
    K[17] = 0
    K = K.to(DEV)
    rows, n = sdd.select_rows(K)
    draft = sdd.confidence(z_d, x)
    L, tok, nc = sdd.verify_strict_listed(z_t, x, rows, n, z_d=z_d, draft=draft, seed=11, round_=3)
    want_rows = torch.tensor([5, 17], dtype=torch.int32, device=DEV)
    L2, tok2, nc2 = sdd.verify_strict(z_t, x, z_d=z_d, draft=draft, seed=11, round_=3, rows=want_rows)
    torch.cuda.synchronize()
    assert int(n.item()) == 2
    assert torch.equal(L, L2) and torch.equal(tok, tok2) and torch.equal(nc, nc2)
    ob = oracle_block(z_d, z_t, x, seed=11, round_=3, blocks=[5, 17])
    compare_rule(Tally(), "listed, few blocks", L, tok, ob.strict, [5, 17])
    others = [b for b in range(B) if b not in (5, 17)]
    assert torch.all(L[others] == -2) and torch.all(tok[others] == -2)
