"""Decode-loop simulation of the path (the decode-loop workload).

Every round a batch of B draft blocks of gamma positions is scored twice --
raw confidence q = p_draft(x_j) from the drafter logits (Sec. 4.2) and a
learned-style survival score from the drafter hidden states and scalar
features (the scorer of App. A.7: by default its full shape, (3584 + 19) ->
256 -> 256 -> 256 -> 1, fed the row statistics the confidence pass also
returns; here with random-init stand-in weights) -- and the prefix schedule of
Sec. 4.1 picks K per block for each signal, with each policy's staleness
counter D carried across rounds.  The raw-confidence policy drives the round:
blocks with K = 0 go to the strict verifier (Sec. 3.1), which reads only
their target rows (row compaction); the committed tokens are x_1..x_K for a
skipped block and the verified tokens otherwise.  The survival-score policy
and the confidence-free periodic baseline of the appendix (a skip of K_min
tokens once every `period` rounds) run in shadow (their decisions and
verifier calls saved are counted).

Every step runs in libsdd.so through the binding; this module only sequences
the calls.  One device-to-host read per round (how many blocks to verify)
stands in for the host deciding whether to call the verifier at all.

    python -m paper_2608_14787_gb300.loop --rounds 256     # prints one JSON line
"""
from __future__ import annotations

import argparse
import json
import time
from dataclasses import dataclass, field

import torch

from . import binding as sdd
from . import synth


@dataclass
class RoundOut:
    K_raw: torch.Tensor        # [B] K under raw confidence (drives the round)
    K_mlp: torch.Tensor        # [B] K under the survival score (shadow)
    K_per: torch.Tensor        # [B] K under the periodic baseline (shadow)
    L: torch.Tensor            # [B] strict accepted length (-2 for skipped blocks)
    tokens: torch.Tensor       # [B, gamma+1] committed tokens (-1 padded)
    n: torch.Tensor            # [B] committed count
    n_verified: int
    score: torch.Tensor = None  # [B, gamma] the survival scorer's output


@dataclass
class LoopStats:
    rounds: int = 0
    blocks: int = 0
    verified: int = 0
    skipped_raw: int = 0
    skipped_mlp: int = 0
    skipped_per: int = 0
    committed_tokens: int = 0
    device_seconds: float = 0.0
    per_round_verified: list = field(default_factory=list)


class DecodeLoop:
    """State of one decode loop: workspace, D per policy, scorer weights."""

    def __init__(self, B: int, gamma: int, V: int, *, tau: float = 0.9, tau_mlp: float = 0.9, K_min: int = 6,
                 S_max: int = 64, greedy: bool = False, seed: int = 4, hidden: int = synth.HIDDEN, period: int = 4,
                 scorer: str = "deep", device="cuda"):
        self.B, self.gamma, self.V = B, gamma, V
        self.tau, self.tau_mlp, self.K_min, self.S_max = tau, tau_mlp, K_min, S_max
        self.greedy, self.seed, self.period = greedy, seed, period
        dev = torch.device(device)
        self.device = dev
        self.ws = sdd.Workspace(B, gamma, V, dev)
        self.status = sdd.new_status(dev)
        self.D_raw = torch.zeros(B, dtype=torch.int32, device=dev)
        self.D_mlp = torch.zeros(B, dtype=torch.int32, device=dev)
        self.D_per = torch.zeros(B, dtype=torch.int32, device=dev)
        self.scorer = scorer
        if scorer == "deep":
            self.deep = synth.make_scorer_deep(device=dev, seed=seed, hidden=hidden)
            self.feat = torch.zeros(B * gamma, sdd.MLP_HIDDEN, dtype=torch.bfloat16, device=dev)
            self.act = torch.empty(B * gamma, sdd.MLP_HIDDEN, dtype=torch.bfloat16, device=dev)
        elif scorer == "mlp":
            self.W1, self.b1, self.w2, b2 = synth.make_mlp(device=dev, seed=seed, hidden=hidden)
            self.b2 = float(b2.item())
        else:
            raise ValueError(f"scorer {scorer!r}: 'deep' or 'mlp'")
        self.scorer_ws = sdd.scorer_workspace(B * gamma, dev)
        # per-round outputs, allocated once: the schedules' (K_hat, K, D_out)
        # alternate between two sets so that D_out never aliases D_in
        i32 = lambda *shape: torch.empty(*shape, dtype=torch.int32, device=dev)  # noqa: E731
        self._conf = sdd.confidence_buffers(B, gamma, dev, features=(scorer == "deep"))
        self._sched = {p: [(i32(1, B), i32(1, B), i32(1, B)) for _ in range(2)] for p in ("raw", "mlp", "per")}
        self._commit = (i32(B, gamma + 1), i32(B))
        self._flip = 0

    def features(self, conf, round_: int) -> torch.Tensor:
        """The scorer's scalar-feature block [B * gamma, 256] bf16 (sdd_scorer_features:
        19 columns in the order of App. A.7's list, zeros after them).  The
        diffusion-model quantities (reveal step and rank, parallelism, late
        reveal, step-0 values and their changes, segment position, dataset
        flags) are not available here and stay zero; the logits-side ones come
        from the confidence pass: top-1 probability, its log, entropy, its
        negative, probability margin, top-5 mass; then block position and
        generated length."""
        return sdd.scorer_features(conf, round_, out=self.feat)

    def step(self, z_d, z_t, x, h, round_: int) -> RoundOut:
        """One round.  The returned tensors (and the loop's D and feature
        block) live in buffers that the next step reuses."""
        B, gamma = self.B, self.gamma
        deep = self.scorer == "deep"
        o = self._flip
        self._flip ^= 1
        conf = sdd.confidence(z_d, x, ws=self.ws, status=self.status, features=deep, out=self._conf)
        if deep:
            s = sdd.scorer_deep(h, self.features(conf, round_), *self.deep, act=self.act, status=self.status,
                                workspace=self.scorer_ws).reshape(B, gamma)
        else:
            s = sdd.survival_mlp(h, self.W1, self.b1, self.w2, self.b2, status=self.status,
                                 workspace=self.scorer_ws).reshape(B, gamma)
        _, K_raw, D_raw = sdd.schedule_prefix(conf.q, [self.tau], [self.tau], signal=sdd.SIG_RAW, logq=conf.logq,
                                              K_min=self.K_min, S_max=self.S_max, D_in=self.D_raw,
                                              status=self.status, out=self._sched["raw"][o])
        _, K_mlp, D_mlp = sdd.schedule_prefix(s, [self.tau_mlp], [self.tau_mlp], signal=sdd.SIG_CONDITIONAL,
                                              K_min=self.K_min, S_max=self.S_max, D_in=self.D_mlp,
                                              status=self.status, out=self._sched["mlp"][o])
        _, K_per, D_per = sdd.schedule_periodic(B, gamma, [self.period], K_skip=max(self.K_min, 1), round_=round_,
                                                K_min=self.K_min, S_max=self.S_max, D_in=self.D_per,
                                                status=self.status, device=self.device,
                                                out=self._sched["per"][o])
        K = K_raw[0]
        rows = torch.nonzero(K == 0).flatten().to(torch.int32)    # the host's verify decision
        n_rows = int(rows.numel())
        L, tok, n = sdd.verify_strict(z_t, x, z_d=z_d, draft=conf, greedy=self.greedy, seed=self.seed, round_=round_,
                                      rows=rows, ws=self.ws, status=self.status)
        tokens, n_commit = sdd.commit(K, x, tok, n, out=self._commit)
        self.D_raw, self.D_mlp, self.D_per = D_raw[0], D_mlp[0], D_per[0]
        return RoundOut(K_raw=K, K_mlp=K_mlp[0], K_per=K_per[0], L=L, tokens=tokens, n=n_commit, n_verified=n_rows,
                        score=s)


def run(rounds: int = 256, workload: str = "c5", warmup: int = 2, scorer: str = "deep", device="cuda") -> dict:
    """The decode-loop workload: `rounds` rounds of fresh synthetic logits and
    hidden states (generated before each round, untimed)."""
    wl = synth.WORKLOADS[workload]
    B, gamma, V = wl.B, wl.gamma, wl.V
    loop = DecodeLoop(B, gamma, V, tau=wl.taus[0], device=device, seed=wl.seed, scorer=scorer)
    st = LoopStats()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    for r in range(-warmup, rounds):
        rr = max(r, 0)
        blk = synth.make_block(wl, device=device, round_=rr)
        h = synth.make_hidden(B * gamma, device=device, seed=wl.seed, round_=rr)
        torch.cuda.synchronize()
        e0.record()
        out = loop.step(blk.z_d, blk.z_t, blk.x, h, round_=rr)
        e1.record()
        torch.cuda.synchronize()
        if r < 0:
            loop.D_raw.zero_()
            loop.D_mlp.zero_()
            loop.D_per.zero_()
            continue
        st.rounds += 1
        st.blocks += B
        st.device_seconds += e0.elapsed_time(e1) / 1e3
        st.verified += out.n_verified
        st.per_round_verified.append(out.n_verified)
        st.skipped_raw += int((out.K_raw > 0).sum().item())
        st.skipped_mlp += int((out.K_mlp > 0).sum().item())
        st.skipped_per += int((out.K_per > 0).sum().item())
        st.committed_tokens += int(out.n.sum().item())
        del blk, h
    status = int(loop.status.item())
    return {
        "workload": f"{wl.name}: B={B}, gamma={gamma}, V={V}, {rounds} rounds",
        "rounds": st.rounds, "blocks": st.blocks,
        "blocks_per_s": st.blocks / st.device_seconds if st.device_seconds > 0 else None,
        "ms_per_round": 1e3 * st.device_seconds / max(st.rounds, 1),
        "verifier_calls": st.verified,
        "verifier_calls_saved_raw": st.skipped_raw / max(st.blocks, 1),
        "verifier_calls_saved_mlp_shadow": st.skipped_mlp / max(st.blocks, 1),
        "scorer": "(3584 + 19) -> 256 -> 256 -> 256 -> 1 (sdd_scorer_deep)" if scorer == "deep"
        else "3584 -> 256 -> 1 (sdd_survival_mlp)",
        "verifier_calls_saved_periodic_shadow": st.skipped_per / max(st.blocks, 1),
        "periodic_P": loop.period,
        "committed_tokens_per_block": st.committed_tokens / max(st.blocks, 1),
        "device_status": status,
    }


def main():
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--rounds", type=int, default=256)
    ap.add_argument("--workload", default="c5")
    args = ap.parse_args()
    sdd.load()
    t0 = time.time()
    res = run(args.rounds, args.workload)
    res["wall_s"] = time.time() - t0
    print(json.dumps(res), flush=True)


if __name__ == "__main__":
    main()
