"""Helpers for the GPU-vs-oracle parity tests.

Everything expected comes from ``oracle/`` on the same seeded inputs the CUDA
path receives.  Decision outputs (accepted lengths, tokens, skip lengths) must
match exactly except on rows where the oracle reports a compared quantity
within NEAR = 1e-6 of its threshold; those rows are counted ("flagged"), and
mismatches among them are reported, not failed.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch

import oracle as orc

NEAR = 1e-6
RTOL = {torch.bfloat16: 2e-3, torch.float32: 1e-5}
ATOL = 1e-7


def host(z: torch.Tensor) -> np.ndarray:
    """What the oracle reads: bf16 bits as uint16, or fp32."""
    z = z.detach().cpu().contiguous()
    if z.dtype == torch.bfloat16:
        return z.view(torch.int16).numpy().view(np.uint16)
    return z.numpy()


def assert_close_stats(name, got: torch.Tensor, want: np.ndarray, dtype, mask=None):
    g = got.detach().cpu().double().numpy()
    w = np.asarray(want, np.float64)
    if mask is not None:
        g, w = g[mask], w[mask]
    both_nan = np.isnan(g) & np.isnan(w)
    g, w = g[~both_nan], w[~both_nan]
    tol = RTOL[dtype] * np.abs(w) + ATOL
    err = np.abs(g - w)
    bad = ~(err <= tol)
    assert not bad.any(), (f"{name}: {bad.sum()} of {bad.size} outside rtol {RTOL[dtype]}; worst "
                           f"rel {np.max(err / np.maximum(np.abs(w), 1e-30)):.3e}")
    return float(np.max(err / np.maximum(np.abs(w), 1e-30))) if err.size else 0.0


def assert_close_logratio(name, got: torch.Tensor, want: np.ndarray, dtype):
    """A log-probability: its absolute error is the relative error of the
    probability, so it is held to the relative tolerance as an absolute one."""
    g = got.detach().cpu().double().numpy()
    w = np.asarray(want, np.float64)
    both_nan = np.isnan(g) & np.isnan(w)
    err = np.abs(g - w)[~both_nan]
    bad = ~(err <= RTOL[dtype])
    assert not bad.any(), f"{name}: {bad.sum()} of {bad.size} outside {RTOL[dtype]}; worst {err.max():.3e}"
    return float(err.max()) if err.size else 0.0


@dataclass
class Tally:
    compared: int = 0
    flagged: int = 0
    flagged_mismatch: int = 0
    notes: list = field(default_factory=list)

    def check(self, what, ok: bool, margin: float):
        self.compared += 1
        if margin < NEAR:
            self.flagged += 1
            if not ok:
                self.flagged_mismatch += 1
            return
        assert ok, f"{what}: mismatch at a row whose oracle margin is {margin:.3e} >= {NEAR}"


@dataclass
class OracleBlock:
    stats: orc.RowStats
    facts: list                     # per block TargetFacts
    strict: list                    # per block (L, tokens, margin)
    greedy: list
    lenient: dict                   # ell -> list per block
    topk: dict                      # k -> list per block
    sched: dict                     # (eb, ec) -> (K_hat, K, D_out, margin)


def oracle_block(z_d, z_t, x, *, seed=0, round_=0, pairs=(), signal=0, K_min=6, S_max=64, D_in=None,
                 ells=(), ks=(), blocks=None, sampling=True, guard=None, force_strict=None) -> OracleBlock:
    """Run the oracle on blocks `blocks` (default all) of the batch.  The
    tensors always hold the whole batch, so that each block keeps its batch
    index b (its Philox stream)."""
    B = x.shape[0]
    blocks = list(range(B)) if blocks is None else list(blocks)
    zd, zt = host(z_d[blocks]), host(z_t[blocks])
    xx = x[blocks].detach().cpu().numpy().astype(np.int32)
    st = orc.row_stats(zd, tokens=xx)
    facts, strict, greedy = [], [], []
    lenient = {e: [] for e in ells}
    topk = {k: [] for k in ks}
    for i, b in enumerate(blocks):
        f = orc.target_facts(zt[i], xx[i])
        facts.append(f)
        greedy.append(orc.verify_greedy(f, xx[i]))
        if sampling:
            strict.append(orc.verify_strict(zt[i], zd[i], xx[i], seed=seed, b=b, round_=round_))
        for e in ells:
            lenient[e].append(orc.verify_lenient(f, xx[i], e))
        for k in ks:
            topk[k].append(orc.verify_topk(f, xx[i], k))
    sched = {}
    D = None if D_in is None else np.asarray(D_in)[blocks]
    g = None if guard is None else np.asarray(guard)[blocks]
    fs = None if force_strict is None else np.asarray(force_strict)[blocks]
    for (eb, ec) in pairs:
        sched[(eb, ec)] = orc.schedule(st.q, signal, eb, ec, K_min, S_max, guard=g, force_strict=fs, D_in=D)
    return OracleBlock(stats=st, facts=facts, strict=strict, greedy=greedy, lenient=lenient, topk=topk, sched=sched)


def compare_rule(tally: Tally, name, L_gpu, tok_gpu, oracle_list, blocks):
    L_gpu = L_gpu.detach().cpu().numpy()
    tok_gpu = tok_gpu.detach().cpu().numpy()
    for idx, b in enumerate(blocks):
        L, tok, mg = oracle_list[idx]
        ok = (int(L_gpu[b]) == L) and np.array_equal(tok_gpu[b], tok)
        tally.check(f"{name} block {b} (gpu L={int(L_gpu[b])} tok={tok_gpu[b][:L_gpu[b]+1].tolist()[-3:]} ; "
                    f"oracle L={L} tok={tok[:L+1].tolist()[-3:]})", ok, mg)


def row_stats_threads(zd, tokens, threads=None):
    """orc.row_stats over the leading (batch) axis split across host threads
    (the oracle's C calls release the interpreter lock); same result as one
    call over the whole array."""
    import os
    from concurrent.futures import ThreadPoolExecutor
    B = zd.shape[0]
    threads = max(1, min(B, threads or os.cpu_count() or 1))
    cuts = np.linspace(0, B, threads + 1).astype(int)
    parts = [(a, b) for a, b in zip(cuts[:-1], cuts[1:]) if b > a]
    with ThreadPoolExecutor(max_workers=len(parts)) as ex:
        res = list(ex.map(lambda ab: orc.row_stats(zd[ab[0]:ab[1]], tokens=tokens[ab[0]:ab[1]]), parts))
    cat = lambda name: np.concatenate([getattr(r, name) for r in res], axis=0)   # noqa: E731
    return orc.RowStats(m=cat("m"), lse=cat("lse"), q=cat("q"), logq=cat("logq"), maxprob=cat("maxprob"),
                        entropy=cat("entropy"), argmax=cat("argmax"))
