"""GPU parity of the pipelined round (sdd_block_pipelined): rounds over
independent batches, each streamed in one launch and decided in the next
(beside the following round's streaming pass), every round's outputs against
the oracle exactly as for sdd_block: statistics within the dtype's tolerance,
decisions and tokens bit-exact outside the near-threshold band, the agreement
counters and commits of pair 0."""
import numpy as np
import pytest
import torch

import oracle as orc
import paper_2608_14787_gb300 as sdd
from paper_2608_14787_gb300 import synth
from parity_util import Tally, assert_close_stats, compare_rule, oracle_block

pytestmark = pytest.mark.gpu

DEV = "cuda"


def _padded(z: torch.Tensor, stride: int) -> torch.Tensor:
    """Same logits with each row padded to `stride` elements (+inf padding,
    which must never reach a result)."""
    B, P, V = z.shape
    buf = torch.full((B, P, stride), float("inf"), dtype=z.dtype, device=z.device)
    buf[..., :V] = z
    return buf[..., :V]


class _Round:
    """One round of a sequence: its inputs, its BlockRound and its rules."""

    def __init__(self, rnd, blk, seed, round_, taus, ells, ks, greedy, K_min, S_max, D, sample=None):
        self.rnd, self.blk = rnd, blk
        self.seed, self.round_ = seed, round_
        self.taus, self.ells, self.ks, self.greedy = taus, ells, ks, greedy
        self.K_min, self.S_max, self.D = K_min, S_max, D
        self.sample = sample


def _check(r: _Round, tally: Tally):
    """Round r's outputs against the oracle: every block, or the blocks in
    r.sample (then without the batch-wide agreement counters)."""
    rnd, blk = r.rnd, r.blk
    dtype = blk.z_d.dtype
    assert int(rnd.status.item()) == 0
    blocks = list(range(blk.x.shape[0])) if r.sample is None else list(r.sample)
    ob = oracle_block(blk.z_d, blk.z_t, blk.x, seed=r.seed, round_=r.round_, pairs=[(t, t) for t in r.taus],
                      K_min=r.K_min, S_max=r.S_max, D_in=r.D.numpy(), ells=r.ells, ks=r.ks, sampling=not r.greedy,
                      blocks=blocks)
    sub = lambda t: t[blocks]   # noqa: E731
    assert_close_stats("q", sub(rnd.q), ob.stats.q, dtype)
    assert_close_stats("lse", sub(rnd.lse), ob.stats.lse, dtype)
    assert_close_stats("entropy", sub(rnd.entropy), ob.stats.entropy, dtype)
    np.testing.assert_array_equal(sub(rnd.argmax).cpu().numpy(), ob.stats.argmax)
    idx = list(range(len(blocks)))
    strict = ob.greedy if r.greedy else ob.strict
    compare_rule(tally, "strict", sub(rnd.L_strict), sub(rnd.tokens_strict), strict, idx)
    for i, e in enumerate(r.ells):
        compare_rule(tally, f"lenient {e:.4f}", sub(rnd.L_lenient[i]), sub(rnd.tokens_lenient[i]), ob.lenient[e], idx)
    for i, k in enumerate(r.ks):
        compare_rule(tally, f"top-{k}", sub(rnd.L_topk[i]), sub(rnd.tokens_topk[i]), ob.topk[k], idx)
    L_or = np.array([strict[i][0] for i in idx])
    acc_want = np.zeros((len(r.taus), 4), np.int64)
    for t, tau in enumerate(r.taus):
        oKh, oK, oD, mg = ob.sched[(tau, tau)]
        for i, b in enumerate(blocks):
            ok = (rnd.K_hat[t, b].item() == oKh[i] and rnd.K[t, b].item() == oK[i] and rnd.D_out[t, b].item() == oD[i])
            tally.check(f"schedule tau {tau} block {b}", ok, mg[i])
        acc_want[t] = orc.agreement(oK, L_or)
    if r.sample is None:
        np.testing.assert_array_equal(rnd.agreement.cpu().numpy(), acc_want)
    oK0 = ob.sched[(r.taus[0], r.taus[0])][1]
    ct, cn, xs = rnd.commit_tokens.cpu().numpy(), rnd.commit_n.cpu().numpy(), blk.x.cpu().numpy()
    for i, b in enumerate(blocks):
        if oK0[i] > 0:
            assert cn[b] == oK0[i] and np.array_equal(ct[b][:oK0[i]], xs[b][:oK0[i]]) and np.all(ct[b][oK0[i]:] == -1)
        else:
            L, tok, _ = strict[i]
            assert cn[b] == L + 1 and np.array_equal(ct[b], tok)


def _run_sequence(rounds):
    """sdd_block_pipelined over the rounds in order: call n streams round n
    and decides round n-1; round n-1 is compared once that call has completed,
    before its BlockRound is used again."""
    tally = Tally()
    prev = None
    for r in rounds:
        r.rnd.agreement.zero_()
        r.rnd.D_in.copy_(r.D)
        r.rnd.set_inputs(r.blk.z_d, r.blk.z_t, r.blk.x, seed=r.seed, round_=r.round_)
        sdd.block_pipelined(r.rnd, None if prev is None else prev.rnd)
        torch.cuda.synchronize()
        if prev is not None:
            _check(prev, tally)
        prev = r
    sdd.block_pipelined(None, prev.rnd)
    torch.cuda.synchronize()
    _check(prev, tally)
    return tally


def _small_rounds(n, greedy, B=12, gamma=16, V=12007, stride=12008):
    taus, ells, ks = (0.5, 0.9, 0.95, 1.0), (1.0, 0.5), (2, 5)
    pair = [sdd.BlockRound(B, gamma, V, taus=taus, ells=ells, ks=ks, greedy=greedy, K_min=2, S_max=64)
            for _ in range(2)]
    g = torch.Generator().manual_seed(11)
    out = []
    for i in range(n):
        blk = synth.make_block("c3", device="cpu", B=B, gamma=gamma, V=V, greedy_drafts=greedy, round_=i)
        z_d, z_t = _padded(blk.z_d.to(DEV), stride), _padded(blk.z_t.to(DEV), stride)
        blk = synth.Block(z_d=z_d, z_t=z_t, x=blk.x.to(DEV), peaked=blk.peaked)
        D = torch.randint(0, 70, (B,), dtype=torch.int32, generator=g)
        out.append(_Round(pair[i % 2], blk, 77 + i, i, taus, ells, ks, greedy, 2, 64, D))
    return out


@pytest.mark.parametrize("greedy", [False, True])
def test_pipelined_rounds_vs_oracle(greedy):
    tally = _run_sequence(_small_rounds(4, greedy))
    print("pipelined rounds", tally)


def test_pipelined_c3_rounds_vs_oracle():
    """Three rounds of the 16-block workload (gamma = 32, V = 151,936 bf16,
    strict sampling + lenience + top-k) in the benchmark's launch
    configuration: every block of every round against the oracle."""
    wl = synth.WORKLOADS["c3"]
    ells = tuple(synth.paper_ell(e) for e in wl.ells)
    ks = tuple(wl.topks)
    pair = [sdd.BlockRound(wl.B, wl.gamma, wl.V, dtype=wl.dtype, taus=wl.taus, ells=ells, ks=ks, K_min=6, S_max=64)
            for _ in range(2)]
    rounds = [_Round(pair[i % 2], synth.make_block(wl, device=DEV, round_=i), wl.seed, i, wl.taus, ells, ks, False,
                     6, 64, torch.zeros(wl.B, dtype=torch.int32)) for i in range(3)]
    tally = _run_sequence(rounds)
    print("pipelined c3", tally)


def test_pipelined_mixed_shapes_and_more_blocks_than_ctas():
    """Rounds of different shapes follow one another; a round of 40 one-token
    blocks over an 8-entry vocabulary streams on 4 CTAs, so each CTA's decide
    warps take ten of its blocks in turn."""
    taus, ells, ks = (0.9,), (0.5,), (2,)
    shapes = [(40, 1, 8, torch.bfloat16), (5, 8, 30011, torch.float32), (40, 1, 8, torch.bfloat16),
              (7, 32, 20000, torch.bfloat16)]
    rounds = []
    g = torch.Generator().manual_seed(5)
    for i, (B, gamma, V, dt) in enumerate(shapes):
        rnd = sdd.BlockRound(B, gamma, V, dtype=dt, taus=taus, ells=ells, ks=ks, K_min=0, S_max=64)
        blk = synth.make_block("c3", device=DEV, B=B, gamma=gamma, V=V, dtype=dt, round_=i)
        esz = 2 if dt == torch.bfloat16 else 4
        stride = -(-V * esz // 16) * 16 // esz   # rows padded to 16 bytes
        if stride != V:
            blk = synth.Block(z_d=_padded(blk.z_d, stride), z_t=_padded(blk.z_t, stride), x=blk.x, peaked=blk.peaked)
        D = torch.randint(0, 10, (B,), dtype=torch.int32, generator=g)
        rounds.append(_Round(rnd, blk, 3 + i, i, taus, ells, ks, False, 0, 64, D))
    tally = _run_sequence(rounds)
    print("pipelined mixed shapes", tally)


def test_pipelined_large_and_small_rounds_alternate():
    """Rounds above 512 MiB of logits (48 blocks of the 16-block workload's
    rows: 948 MB) stream on all sixteen warps and are decided by the decide
    kernel; smaller ones run in the pipelined kernel.  A sequence alternating
    the two hands each kind of round to the other kind of call; sampled
    blocks of the large rounds and every block of the small one against the
    oracle."""
    wl = synth.WORKLOADS["c3"]
    ells = tuple(synth.paper_ell(e) for e in wl.ells)
    ks = tuple(wl.topks)
    rounds = []
    for i, B in enumerate((48, 16, 48)):
        rnd = sdd.BlockRound(B, wl.gamma, wl.V, dtype=wl.dtype, taus=wl.taus, ells=ells, ks=ks, K_min=6, S_max=64)
        blk = synth.make_block(wl, device=DEV, B=B, round_=i)
        sample = None if B == 16 else (0, 13, 30, 47)
        rounds.append(_Round(rnd, blk, wl.seed, i, wl.taus, ells, ks, False, 6, 64,
                             torch.zeros(B, dtype=torch.int32), sample=sample))
    tally = _run_sequence(rounds)
    print("pipelined large / small", tally)


def test_pipelined_rejects_one_round_as_both():
    rnd = sdd.BlockRound(2, 4, 1000, taus=(0.9,))
    with pytest.raises(ValueError):
        sdd.block_pipelined(rnd, rnd)
    with pytest.raises(sdd.SddError):
        sdd.block_pipelined(None, None)
