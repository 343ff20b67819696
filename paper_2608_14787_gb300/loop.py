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
the calls.  The blocks to verify and their count stay on the device
(sdd_select_rows, sdd_verify_strict_listed), so a round needs no host round
trip and rounds queue back to back.

    python -m paper_2608_14787_gb300.loop --rounds 256     # prints one JSON line
"""
from __future__ import annotations

import argparse
import json
import time
from dataclasses import dataclass

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
    n_verified: torch.Tensor   # [1] blocks sent to the verifier (device)
    score: torch.Tensor = None  # [B, gamma] the survival scorer's output


class DecodeLoop:
    """State of one decode loop: workspace, D per policy, scorer weights, and
    `history` slots of per-round outputs (round r uses slot r mod history).
    Nothing in a round waits for the host: the blocks to verify are selected
    on the device (sdd_select_rows) and verified with their count read there
    (sdd_verify_strict_listed), so rounds queue back to back on the stream."""

    def __init__(self, B: int, gamma: int, V: int, *, tau: float = 0.9, tau_mlp: float = 0.9, K_min: int = 6,
                 S_max: int = 64, greedy: bool = False, seed: int = 4, hidden: int = synth.HIDDEN, period: int = 4,
                 scorer: str = "deep", history: int = 8, overlap: bool = True, device="cuda"):
        self.B, self.gamma, self.V = B, gamma, V
        self.tau, self.tau_mlp, self.K_min, self.S_max = tau, tau_mlp, K_min, S_max
        self.greedy, self.seed, self.period = greedy, seed, period
        dev = torch.device(device)
        self.device = dev
        self.ws = sdd.Workspace(B, gamma, V, dev)
        self.status = sdd.new_status(dev)
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
        self._conf = sdd.confidence_buffers(B, gamma, dev, features=(scorer == "deep"))
        self.score = torch.empty(B * gamma, dtype=torch.float32, device=dev)
        # per-round outputs in history slots (never aliasing the previous
        # round's D, which the next schedule reads)
        H = max(2, int(history))
        self.history = H
        i32 = lambda *shape: torch.empty(*shape, dtype=torch.int32, device=dev)  # noqa: E731
        self.hist = {p: (i32(H, 1, B), i32(H, 1, B), i32(H, 1, B)) for p in ("raw", "mlp", "per")}
        self.hist_L = torch.full((H, B), -2, dtype=torch.int32, device=dev)
        self.hist_vt = torch.full((H, B, gamma + 1), -2, dtype=torch.int32, device=dev)
        self.hist_vn = torch.full((H, B), -2, dtype=torch.int32, device=dev)
        self.hist_n_rows = i32(H, 1)
        self.hist_tokens = i32(H, B, gamma + 1)
        self.hist_n = i32(H, B)
        self.rows = i32(B)
        # the survival scorer and the two shadow schedules (scorer, periodic)
        # need only the confidence pass: with overlap they run on a second
        # stream beside the raw schedule and the verifier pass
        self.overlap = overlap
        self.side = torch.cuda.Stream(device=dev) if overlap else None
        self._conf_ready = torch.cuda.Event() if overlap else None
        self._side_done = torch.cuda.Event() if overlap else None
        self.reset()

    def reset(self):
        """Staleness counters back to 0 (a new loop)."""
        z = torch.zeros(self.B, dtype=torch.int32, device=self.device)
        self.D_raw, self.D_mlp, self.D_per = z, z.clone(), z.clone()
        self.rounds_run = 0

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
        """One round, enqueued without waiting for the device.  The returned
        tensors live in history slot round_ mod history."""
        B, gamma = self.B, self.gamma
        deep = self.scorer == "deep"
        k = round_ % self.history
        if self.rounds_run >= self.history:
            # the slot held an older round: unlisted blocks must read -2 again
            self.hist_L[k].fill_(-2)
            self.hist_vt[k].fill_(-2)
            self.hist_vn[k].fill_(-2)
        self.rounds_run += 1
        main = torch.cuda.current_stream(self.device)
        conf = sdd.confidence(z_d, x, ws=self.ws, status=self.status, features=deep, out=self._conf)
        o = lambda p: tuple(t[k] for t in self.hist[p])   # noqa: E731

        def scored():
            if deep:
                sc = sdd.scorer_deep(h, self.features(conf, round_), *self.deep, act=self.act, status=self.status,
                                     workspace=self.scorer_ws, out=self.score).reshape(B, gamma)
            else:
                sc = sdd.survival_mlp(h, self.W1, self.b1, self.w2, self.b2, status=self.status,
                                      workspace=self.scorer_ws, out=self.score).reshape(B, gamma)
            _, K_m, D_m = sdd.schedule_prefix(sc, [self.tau_mlp], [self.tau_mlp], signal=sdd.SIG_CONDITIONAL,
                                              K_min=self.K_min, S_max=self.S_max, D_in=self.D_mlp,
                                              status=self.status, out=o("mlp"))
            _, K_p, D_p = sdd.schedule_periodic(B, gamma, [self.period], K_skip=max(self.K_min, 1), round_=round_,
                                                K_min=self.K_min, S_max=self.S_max, D_in=self.D_per,
                                                status=self.status, device=self.device, out=o("per"))
            return sc, K_m, D_m, K_p, D_p

        if self.overlap:
            self._conf_ready.record(main)
            self.side.wait_event(self._conf_ready)
            with torch.cuda.stream(self.side):
                s, K_mlp, D_mlp, K_per, D_per = scored()
                self._side_done.record(self.side)
        else:
            s, K_mlp, D_mlp, K_per, D_per = scored()
        _, K_raw, D_raw = sdd.schedule_prefix(conf.q, [self.tau], [self.tau], signal=sdd.SIG_RAW, logq=conf.logq,
                                              K_min=self.K_min, S_max=self.S_max, D_in=self.D_raw,
                                              status=self.status, out=o("raw"))
        K = K_raw[0]
        rows, n_rows = sdd.select_rows(K, rows=self.rows, n_rows=self.hist_n_rows[k])
        L, tok, n = sdd.verify_strict_listed(z_t, x, rows, n_rows, z_d=z_d, draft=conf, greedy=self.greedy,
                                             seed=self.seed, round_=round_, ws=self.ws, status=self.status,
                                             out=(self.hist_L[k], self.hist_vt[k], self.hist_vn[k]))
        tokens, n_commit = sdd.commit(K, x, tok, n, out=(self.hist_tokens[k], self.hist_n[k]))
        if self.overlap:
            # later work on the stream (the next round's confidence pass, which
            # overwrites what the scorer read; any read of these outputs) comes
            # after the side stream's
            main.wait_event(self._side_done)
        self.D_raw, self.D_mlp, self.D_per = D_raw[0], D_mlp[0], D_per[0]
        return RoundOut(K_raw=K, K_mlp=K_mlp[0], K_per=K_per[0], L=L, tokens=tokens, n=n_commit,
                        n_verified=n_rows, score=s)

    def summary(self, rounds: int) -> dict:
        """Statistics of the last `rounds` rounds (all within the history), read
        from the device once."""
        if rounds > self.history:
            raise ValueError("the history holds fewer rounds")
        last = (self.rounds_run - 1) % self.history
        idx = [(last - i) % self.history for i in range(rounds)]
        sel = lambda t: t[idx].cpu()   # noqa: E731
        K_raw, K_mlp, K_per = (sel(self.hist[p][1]) for p in ("raw", "mlp", "per"))
        n_rows, n = sel(self.hist_n_rows), sel(self.hist_n)
        blocks = rounds * self.B
        return {
            "rounds": rounds, "blocks": blocks, "verifier_calls": int(n_rows.sum()),
            "verifier_calls_saved_raw": float((K_raw > 0).sum()) / blocks,
            "verifier_calls_saved_mlp_shadow": float((K_mlp > 0).sum()) / blocks,
            "verifier_calls_saved_periodic_shadow": float((K_per > 0).sum()) / blocks,
            "committed_tokens_per_block": float(n.sum()) / blocks,
        }


def run(rounds: int = 256, workload: str = "c5", warmup: int = 2, scorer: str = "deep", n_sets: int = 8,
        overlap: bool = True, device="cuda") -> dict:
    """The decode-loop workload over `rounds` rounds.  The seeded logits and
    hidden states of `n_sets` rounds are generated first (round r reads set
    r mod n_sets; the rounds still differ by their D, their Philox round index
    and their generated-length feature); then every round is enqueued back to
    back with no host round trip and timed with one pair of events.  A second
    pass times the same rounds with a synchronise after each, which exposes
    the host's launch time per round, and the host's own enqueue time is
    reported."""
    wl = synth.WORKLOADS[workload]
    B, gamma, V = wl.B, wl.gamma, wl.V
    loop = DecodeLoop(B, gamma, V, tau=wl.taus[0], device=device, seed=wl.seed, scorer=scorer, history=rounds,
                      overlap=overlap)
    sets = [(synth.make_block(wl, device=device, round_=r),
             synth.make_hidden(B * gamma, device=device, seed=wl.seed, round_=r)) for r in range(n_sets)]
    for r in range(warmup):
        blk, h = sets[r % n_sets]
        loop.step(blk.z_d, blk.z_t, blk.x, h, round_=r)
    torch.cuda.synchronize()
    loop.reset()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda._sleep(400_000)      # keep the stream busy while the first rounds are enqueued
    e0.record()
    t0 = time.perf_counter()
    for r in range(rounds):
        blk, h = sets[r % n_sets]
        loop.step(blk.z_d, blk.z_t, blk.x, h, round_=r)
    host_s = time.perf_counter() - t0
    e1.record()
    torch.cuda.synchronize()
    dev_ms = e0.elapsed_time(e1)
    stats = loop.summary(rounds)
    # the same rounds with a synchronise after each (host launch time exposed)
    loop.reset()
    sync_ms = 0.0
    for r in range(min(rounds, 64)):
        blk, h = sets[r % n_sets]
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        loop.step(blk.z_d, blk.z_t, blk.x, h, round_=r)
        b.record()
        torch.cuda.synchronize()
        sync_ms += a.elapsed_time(b)
    status = int(loop.status.item())
    return {
        "workload": f"{wl.name}: B={B}, gamma={gamma}, V={V}, {rounds} rounds ({n_sets} seeded input sets)",
        **stats,
        "blocks_per_s": stats["blocks"] / (dev_ms / 1e3),
        "ms_per_round": dev_ms / rounds,
        "ms_per_round_synchronised": sync_ms / min(rounds, 64),
        "host_enqueue_ms_per_round": 1e3 * host_s / rounds,
        "scorer": "(3584 + 19) -> 256 -> 256 -> 256 -> 1 (sdd_scorer_deep)" if scorer == "deep"
        else "3584 -> 256 -> 1 (sdd_survival_mlp)",
        "periodic_P": loop.period,
        "scorer_stream": "second stream beside the verifier pass" if overlap else "in line",
        "device_status": status,
    }


def main():
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--rounds", type=int, default=256)
    ap.add_argument("--workload", default="c5")
    ap.add_argument("--no-overlap", action="store_true", help="run the scorer in line on the main stream")
    args = ap.parse_args()
    sdd.load()
    t0 = time.time()
    res = run(args.rounds, args.workload, overlap=not args.no_overlap)
    res["wall_s"] = time.time() - t0
    print(json.dumps(res), flush=True)


if __name__ == "__main__":
    main()
