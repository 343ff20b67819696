"""Benchmark of the logits-side hot path of verifier-skipping SDD on GB300.

One step = one fused round of the whole path over one batch of draft blocks:
confidence statistics of every drafter row, the prefix skip schedule, strict
(shadow) verification of every block with residual / bonus resampling,
lenience and top-k acceptance on the same target read, agreement counters and
the committed tokens.  Rounds over independent batches are pipelined
(``sdd_block_pipelined``): each launch streams one round's logits and, on four
warps of every CTA, finishes the round before; K steps are K launches and one
closing decide.  The same rounds run unpipelined (``sdd_block_scan`` then
``sdd_block_decide``) are reported beside them.

Default workload (c3): B=16 blocks, gamma=32, V=151,936, bf16 drafter and
target logits; half the positions peaked, half flat; strict sampling, lenience
ell in {1.5, 2, 4} (paper convention 1/ell), top-k k in {2, 5, 10}, raw
confidence schedule at tau=0.9.  Inputs are seeded synthetic logits (no model
weights are available); three input sets of 316 MB each rotate, so every step
reads its logits from HBM, not L2.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference] [--workload c3] [--blocks B]
Prints one JSON line (rank 0).

Other rows of the path, one JSON line each (not the fused-round contract line):
  python bench.py --component mlp [--steps K]   the survival scorer alone (K launches)
  python bench.py --component loop [--steps R]  the decode-loop workload (R rounds, default 256)
  python bench.py --component features          drafter confidence with / without the extended features
  python bench.py --component scorer [--steps K] the deep scorer (K calls)
  python bench.py --component diag              the permutation diagnostic (Table 1 settings)
  python bench.py --component shard [--shards S] the vocabulary-sharded round (S ranks in turn on one GPU)
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "draft blocks verified+scheduled/sec at γ=32,V=151,936 bf16; achieved HBM GB/s vs peak"
UNIT = "blocks/s"
NEAR = 1e-6
# dram__bytes_read.sum + dram__bytes_write.sum of one launch on the c3
# workload, from one ncu capture of the kernel as it stands; reported as the
# "traffic" of that workload's rooflines only: the streaming kernel
# (318,294,528 B + 3,656,960 B) and the pipelined round's kernel
# (328,386,304 B + 3,987,968 B, three rotating input sets).
SCAN_TRAFFIC_C3 = 321_951_488
PIPE_TRAFFIC_C3 = 332_374_272


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def _workload_cfg(name, blocks=None):
    """A workload by name; `blocks` overrides its batch size B (a sweep of the
    same rows over more or fewer blocks)."""
    from paper_2608_14787_gb300 import synth
    wl = synth.WORKLOADS[name]
    if blocks is not None and blocks != wl.B:
        wl = synth.Workload(**{**wl.__dict__, "B": blocks, "name": f"{wl.name}-B{blocks}",
                               "description": wl.description.replace(f"B={wl.B},", f"B={blocks},")})
    ells = tuple(synth.paper_ell(e) for e in wl.ells)
    return wl, ells, tuple(wl.topks)


def _config_json(wl, ells, ks, n_sets=3):
    return {
        "workload": f"{wl.name}: {wl.description}",
        "B": wl.B, "gamma": wl.gamma, "V": wl.V, "dtype": "bf16" if "bfloat16" in str(wl.dtype) else "fp32",
        "taus": list(wl.taus), "ell_paper": [round(e, 6) for e in ells], "topk": list(ks),
        "strict": "sampling with residual/bonus resampling, shadow-verifies every block",
        "K_min": 6, "S_max": 64,
        "l2": f"inputs larger than L2: {n_sets} rotating input set(s) of (2*gamma+1)*V*2*B bytes each",
    }


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""

    FIELDS = ("index,pci.bus_id,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, bus_id: str | None):
        self.bus_id = (bus_id or "").lower()
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        time.sleep(0.2)
        self.lines = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        rows = []
        for l in getattr(self, "lines", []):
            f = [x.strip() for x in l.split(",")]
            if len(f) < 10:
                continue
            if self.bus_id and self.bus_id not in f[1].lower() and f[1].lower() not in self.bus_id:
                continue
            rows.append(f)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no nvidia-smi samples"], "samples": 0}
        sm = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        mx = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[6 + i].lower() == "active"})
        pw = [float(r[4]) for r in rows if r[4].replace(".", "").isdigit()]
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows), "power_w_max": max(pw) if pw else None}


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _host_info():
    """Host cores (nproc) and CPU model, for the oracle baseline."""
    nproc = os.cpu_count() or 1
    model = None
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                key = line.split(":")[0].strip().lower()
                if key in ("model name", "cpu part", "hardware") and ":" in line:
                    model = line.split(":", 1)[1].strip()
                    if key == "model name":
                        break
    except OSError:
        pass
    if model is None:
        try:
            out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
            for line in out.splitlines():
                if line.lower().startswith("model name"):
                    model = line.split(":", 1)[1].strip()
                    break
        except Exception:
            pass
    return nproc, model or "unknown"


def _oracle_one_block(wl, ells, ks, zd, zt, xs, b, round_):
    """Every rule of the path for one block through the fp64 oracle: the raw
    schedule per tau (K, margin), strict sampling, lenience per ell and top-k
    per k (L, tokens, margin)."""
    import oracle as orc
    st = orc.row_stats(zd[b:b + 1], tokens=xs[b:b + 1])
    sched = [orc.schedule(st.q, 0, tau, tau, 6, 64) for tau in wl.taus]
    out = {"K": [(int(k[1][0]), float(k[3][0])) for k in sched],
           "strict": orc.verify_strict(zt[b], zd[b], xs[b], seed=wl.seed, b=b, round_=round_)}
    f = orc.target_facts(zt[b], xs[b])
    out["lenient"] = [orc.verify_lenient(f, xs[b], e) for e in ells]
    out["topk"] = [orc.verify_topk(f, xs[b], k) for k in ks]
    return out


def _oracle_blocks(wl, ells, ks, host, blocks, threads, round_=0):
    """The oracle over `blocks` of one input set, split over `threads` host
    threads (the oracle's C calls release the interpreter lock, so the threads
    run on separate cores).  Returns (seconds, {block: results})."""
    from concurrent.futures import ThreadPoolExecutor
    zd, zt, xs = host["z_d"], host["z_t"], host["x"]
    t0 = time.perf_counter()
    if threads <= 1:
        res = [_oracle_one_block(wl, ells, ks, zd, zt, xs, b, round_) for b in blocks]
    else:
        with ThreadPoolExecutor(max_workers=threads) as ex:
            res = list(ex.map(lambda b: _oracle_one_block(wl, ells, ks, zd, zt, xs, b, round_), blocks))
    return time.perf_counter() - t0, dict(zip(blocks, res))


def _host_block(blk, wl):
    import numpy as np
    import torch

    def h(t):
        t = t.detach().cpu()
        return t.view(torch.int16).numpy().view(np.uint16) if t.dtype == torch.bfloat16 else t.numpy()
    return {"z_d": h(blk.z_d), "z_t": h(blk.z_t), "x": blk.x.detach().cpu().numpy()}


def run_reference(args):
    """The fp64 CPU oracle, as it stands, on the host's cores: each step is a
    bounded sample of the workload (one block per host thread, all rules)."""
    ws, rank, _ = _dist()
    if rank != 0:
        return 0
    from paper_2608_14787_gb300 import synth
    wl, ells, ks = _workload_cfg(args.workload, args.blocks)
    nproc, model = _host_info()
    threads = max(1, min(nproc, args.ref_threads or nproc))
    host = _host_block(synth.make_block(wl, device="cpu", round_=0), wl)

    def step(s):
        blocks = [(s * threads + t) % wl.B for t in range(threads)]
        _oracle_blocks(wl, ells, ks, host, blocks, threads)

    for s in range(args.warmup):
        step(s)
    t0 = time.perf_counter()
    for s in range(args.steps):
        step(s)
    dt = time.perf_counter() - t0
    value = args.steps * threads / dt
    sample = (f"{threads} {wl.name} blocks per step (gamma={wl.gamma}, V={wl.V}), one per host thread, "
              f"all rules")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": _config_json(wl, ells, ks),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": sample,
                         "nproc": nproc, "cpu_model": model},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def _cpu_baseline(wl, ells, ks, host, n_single):
    """The oracle timed on a bounded sample of one input set: one thread over
    the first n_single blocks, and all host cores over every block.  Returns
    (cpu_baseline dict, the all-core run's per-block results)."""
    nproc, model = _host_info()
    dt1, _ = _oracle_blocks(wl, ells, ks, host, list(range(n_single)), 1)
    blocks = list(range(wl.B))
    dtn, res = _oracle_blocks(wl, ells, ks, host, blocks, nproc)
    base = {"value": len(blocks) / dtn, "unit": UNIT, "cores": min(nproc, len(blocks)), "kind": "oracle",
            "sample": f"all {wl.B} blocks of one {wl.name} input set, all rules, one block per thread on "
                      f"{min(nproc, len(blocks))} of {nproc} host cores ({dtn:.1f} s)",
            "nproc": nproc, "cpu_model": model,
            "single_thread": {"value": n_single / dt1, "unit": UNIT, "cores": 1,
                              "sample": f"the first {n_single} blocks, one thread ({dt1:.1f} s)"}}
    return base, res


def _parity_sample(got, res, ells, ks):
    """Compare one round's device decisions (host copies) with the oracle's
    results for the same blocks (bit-exact; a decision whose oracle margin is
    within 1e-6 of its threshold is counted as flagged, not compared)."""
    import numpy as np
    compared = flagged = mismatched = 0

    def check(ok, margin):
        nonlocal compared, flagged, mismatched
        compared += 1
        if margin < NEAR:
            flagged += 1
        elif not ok:
            mismatched += 1
    for b, r in res.items():
        for t, (K, mg) in enumerate(r["K"]):
            check(got["K"][t, b] == K, mg)
        L, tok, mg = r["strict"]
        check(got["L"][b] == L and np.array_equal(got["tok"][b], tok), mg)
        for e in range(len(ells)):
            L, tok, mg = r["lenient"][e]
            check(got["Ll"][e, b] == L and np.array_equal(got["tl"][e, b], tok), mg)
        for k in range(len(ks)):
            L, tok, mg = r["topk"][k]
            check(got["Lk"][k, b] == L and np.array_equal(got["tk"][k, b], tok), mg)
    return {"blocks": len(res), "decisions": compared, "near_threshold": flagged, "mismatches": mismatched}


def _e2e(args, ws, dev, stream, sets, rnd, wl, B):
    """The same round end to end through the C ABI: inputs copied from pinned
    host buffers and results copied back inside the timed region.  Two device
    input buffers alternate: step i + 1's host-to-device copy (on a copy
    stream) overlaps step i's round, and a buffer is refilled only after the
    round that read it (events); every step's copies are inside the region."""
    import torch
    from paper_2608_14787_gb300 import shard
    if ws > 1:
        import torch.distributed as dist
    hz_d = sets[0].z_d.cpu().pin_memory()
    hz_t = sets[0].z_t.cpu().pin_memory()
    hx = sets[0].x.cpu().pin_memory()
    bufs = [(st.z_d, st.z_t, st.x) for st in sets[:2]]
    if len(bufs) < 2:   # (a single input set: a second device buffer for the copies)
        bufs.append(tuple(torch.empty_like(t) for t in bufs[0]))
    outs = [rnd.L_strict, rnd.tokens_strict, rnd.K, rnd.commit_tokens, rnd.commit_n, rnd.q]
    h_outs = [torch.empty(o.shape, dtype=o.dtype, pin_memory=True) for o in outs]
    e2e_steps = max(3, min(args.steps, 200))
    h2d = hz_d.numel() * hz_d.element_size() + hz_t.numel() * hz_t.element_size() + hx.numel() * 4
    d2h = sum(o.numel() * o.element_size() for o in outs)
    main = torch.cuda.current_stream()
    copy = torch.cuda.Stream()
    ready = [torch.cuda.Event() for _ in range(2)]
    done = [torch.cuda.Event() for _ in range(2)]
    for ev in done:
        ev.record(main)

    def issue_copy(i):
        b = i % 2
        copy.wait_event(done[b])               # the round that last read this buffer has finished
        with torch.cuda.stream(copy):
            for d, h in zip(bufs[b], (hz_d, hz_t, hx)):
                d.copy_(h, non_blocking=True)
        ready[b].record(copy)

    def e2e_round(i):
        b = i % 2
        main.wait_event(ready[b])
        dz_d, dz_t, dx = bufs[b]
        rnd.set_inputs(dz_d, dz_t, dx, seed=wl.seed, round_=i)
        rnd.run()
        for h, d in zip(h_outs, outs):
            h.copy_(d, non_blocking=True)
        done[b].record(main)

    def run(n):
        copy.wait_stream(main)   # the copies start after everything issued so far (the start event)
        issue_copy(0)
        for i in range(n):
            if i + 1 < n:
                issue_copy(i + 1)
            e2e_round(i)

    run(2)
    torch.cuda.synchronize()
    if ws > 1:
        dist.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(main)
    run(e2e_steps)
    e1.record(main)
    torch.cuda.synchronize()
    e2e_ms = shard.max_over_ranks(e0.elapsed_time(e1), device=dev)
    return ws * B * e2e_steps / (e2e_ms / 1e3), h2d, d2h


def run_gpu(args):
    import torch
    import paper_2608_14787_gb300 as sdd
    from paper_2608_14787_gb300 import build as sdd_build
    from paper_2608_14787_gb300 import shard, synth

    ws, rank, local = _dist()
    torch.cuda.set_device(local)   # before the process group: NCCL binds each rank to its current device
    dev = torch.device("cuda", local)
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    if rank == 0:
        sdd_build.build()
    if ws > 1:
        dist.barrier()
    sdd.load()

    wl, ells, ks = _workload_cfg(args.workload, args.blocks)
    B, gamma, V = wl.B, wl.gamma, wl.V
    n_sets = max(1, args.sets)
    sets = [synth.make_block(wl, device=dev, round_=r + 1000 * rank) for r in range(n_sets)]
    pair = tuple(sdd.BlockRound(B, gamma, V, dtype=wl.dtype, taus=wl.taus, ells=ells, ks=ks, K_min=6, S_max=64,
                                device=dev) for _ in range(2))
    rnd = pair[0]
    esz = 2 if wl.dtype == torch.bfloat16 else 4
    scan_bytes = (2 * gamma + 1) * V * esz * B          # every logit read once
    draw_bytes = 2 * V * esz * B                         # the decide's two draw rows per block
    # (the library runs rounds of at most 512 MiB of logits in the pipelined
    # kernel, larger ones as its streaming and decide kernels; rows padded to
    # 16 bytes)
    pipelined_kernel = (2 * gamma + 1) * B * (-(-V * esz // 16) * 16) <= (512 << 20)
    stream = torch.cuda.current_stream()
    props = torch.cuda.get_device_properties(dev)
    bus = getattr(props, "pci_bus_id", None)

    # A step is one round over one batch.  Rounds over independent batches are
    # pipelined (sdd_block_pipelined): launch i streams round i and, on four
    # warps of each CTA, finishes round i - 1; a last call finishes the last
    # round.  K steps = K launches + that last call, all inside the region.
    def pstep(i):
        r = pair[i % 2]
        s = sets[i % n_sets]
        r.set_inputs(s.z_d, s.z_t, s.x, seed=wl.seed, round_=i)
        sdd.block_pipelined(r, pair[(i - 1) % 2] if i > 0 else None)

    def pflush(i_last):
        sdd.block_pipelined(None, pair[i_last % 2])

    def pipelined_region(k, first):
        """k pipelined steps (rounds first .. first + k - 1) and the closing
        decide under one event pair; also an event before the closing decide
        (the k launches' own span)."""
        t0, t_mid, t1 = (torch.cuda.Event(enable_timing=True) for _ in range(3))
        torch.cuda._sleep(int(args.prefill_us * 2.0e3))    # ~prefill_us at 2 GHz: rounds queue behind it
        t0.record(stream)
        for i in range(k):
            pstep(first + i)
        t_mid.record(stream)
        pflush(first + k - 1)
        t1.record(stream)
        torch.cuda.synchronize()
        return t0.elapsed_time(t1), t0.elapsed_time(t_mid)

    graph = None
    if args.graph:
        # small rounds outrun the host's launches: the timed steps replay a CUDA
        # graph of --graph pipelined steps (an even number, so that a replay's
        # first launch finishes the round the previous replay streamed last)
        if args.graph % 2 or args.steps % args.graph:
            raise SystemExit("--graph must be even and divide --steps")
        for i in range(args.warmup):
            pstep(i)
        side = torch.cuda.Stream(device=dev)
        side.wait_stream(stream)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=side):
            for j in range(args.graph):
                pstep(args.warmup + j)
        for _ in range(2):
            graph.replay()
        last = args.warmup + args.graph - 1

        def pipelined_region(k, first):   # noqa: F811 -- the graph's rounds replayed
            t0, t_mid, t1 = (torch.cuda.Event(enable_timing=True) for _ in range(3))
            torch.cuda._sleep(int(args.prefill_us * 2.0e3))
            t0.record(stream)
            for _ in range(k // args.graph):
                graph.replay()
            t_mid.record(stream)
            pflush(last)
            t1.record(stream)
            torch.cuda.synchronize()
            return t0.elapsed_time(t1), t0.elapsed_time(t_mid)
    else:
        for i in range(args.warmup):
            pstep(i)
        pflush(args.warmup - 1)
    torch.cuda.synchronize()
    if int(rnd.status.item()) | int(pair[1].status.item()):
        raise RuntimeError("device status set after warm-up")

    # ---- device-resident timed region: exactly K rounds ----
    if ws > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(bus) as clk:
        total_ms, launches_ms = pipelined_region(args.steps, 0)
    if ws > 1:
        dist.barrier()
    total_ms = shard.max_over_ranks(total_ms, device=dev)   # blocks shard by rank: no data-path exchange
    ms_per_step = total_ms / args.steps
    value = ws * B * args.steps / (total_ms / 1e3)
    pipe_avg_ms = launches_ms / args.steps                # one pipelined launch, back to back
    status = int(rnd.status.item()) | int(pair[1].status.item())

    # ---- the same rounds unpipelined: sdd_block_scan then sdd_block_decide
    # per round (each round complete before the next one's streaming pass) ----
    def step(i):
        s = sets[i % n_sets]
        rnd.set_inputs(s.z_d, s.z_t, s.x, seed=wl.seed, round_=i)
        rnd.scan()
        rnd.decide()

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    u0, u1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(bus) as uclk:
        torch.cuda._sleep(int(args.prefill_us * 2.0e3))
        u0.record(stream)
        for i in range(args.steps):
            step(args.warmup + i)
        u1.record(stream)
        torch.cuda.synchronize()
    u_ms = shard.max_over_ranks(u0.elapsed_time(u1), device=dev)
    unpipelined = {"value": ws * B * args.steps / (u_ms / 1e3), "unit": UNIT, "ms_per_step": u_ms / args.steps,
                   "launches": 2 * args.steps, "clocks": uclk.summary(),
                   "what": "sdd_block_scan + sdd_block_decide per round, rounds in series"}

    # ---- the streaming kernel alone: N back-to-back launches (rotating input
    # sets) under one event pair ----
    n_scan = max(50, args.scan_launches)
    for i in range(3):
        s = sets[i % n_sets]
        rnd.set_inputs(s.z_d, s.z_t, s.x, seed=wl.seed, round_=i)
        rnd.scan()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda._sleep(int(args.prefill_us * 2.0e3))
    e0.record(stream)
    for i in range(n_scan):
        s = sets[i % n_sets]
        rnd.set_inputs(s.z_d, s.z_t, s.x, seed=wl.seed, round_=i)
        rnd.scan()
    e1.record(stream)
    torch.cuda.synchronize()
    scan_avg_ms = e0.elapsed_time(e1) / n_scan

    # ---- one untimed pipelined round on input set 0 for the oracle parity
    # sample (its decisions are copied out before the end-to-end leg) ----
    pair[0].set_inputs(sets[0].z_d, sets[0].z_t, sets[0].x, seed=wl.seed, round_=0)
    sdd.block_pipelined(pair[0], None)
    sdd.block_pipelined(None, pair[0])
    torch.cuda.synchronize()
    decisions = {"K": rnd.K.cpu().numpy(), "L": rnd.L_strict.cpu().numpy(), "tok": rnd.tokens_strict.cpu().numpy(),
                 "Ll": rnd.L_lenient.cpu().numpy(), "tl": rnd.tokens_lenient.cpu().numpy(),
                 "Lk": rnd.L_topk.cpu().numpy(), "tk": rnd.tokens_topk.cpu().numpy()}

    if args.no_e2e:
        e2e = None
    else:
        e2e_value, h2d, d2h = _e2e(args, ws, dev, stream, sets, rnd, wl, B)
        e2e = {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}

    peak, peak_kind = _peaks()
    pipe_bytes = scan_bytes + draw_bytes
    achieved = pipe_bytes / (pipe_avg_ms / 1e3) / 1e9
    scan_achieved = scan_bytes / (scan_avg_ms / 1e3) / 1e9
    if rank == 0:
        cpu = parity = None
        if ws == 1 and not args.no_cpu_baseline:
            cpu, res = _cpu_baseline(wl, ells, ks, _host_block(sets[0], wl), min(args.cpu_blocks, B))
            parity = _parity_sample(decisions, res, ells, ks)
        roofline = {"bound": "hbm", "kernel": "pipe_kernel (sdd_block_pipelined)", "achieved": achieved,
                    "peak": peak, "unit": "GB/s", "frac": achieved / peak, "traffic": args.traffic,
                    "peak_source": f"{peak_kind} hbm_gbs (burst copy)",
                    "bytes_per_launch": pipe_bytes, "avg_launch_ms": pipe_avg_ms,
                    "launches_timed": args.steps,
                    "bytes": "every logit of round i once + the two draw rows per block of round i - 1"}
        if not pipelined_kernel:
            # rounds above the pipelined kernel's size run as the streaming and
            # decide kernels: the streaming kernel dominates
            roofline = {"bound": "hbm", "kernel": "scan_kernel (sdd_block_pipelined on a large round)",
                        "achieved": scan_achieved, "peak": peak, "unit": "GB/s", "frac": scan_achieved / peak,
                        "traffic": None, "peak_source": f"{peak_kind} hbm_gbs (burst copy)",
                        "bytes_per_launch": scan_bytes, "avg_launch_ms": scan_avg_ms, "launches_timed": n_scan}
            pipe_avg_ms = scan_avg_ms
        if pipe_avg_ms > ms_per_step:
            # the dominant kernel cannot take longer than the step that contains it
            roofline = {"bound": "hbm", "achieved": None, "peak": peak, "unit": "GB/s", "frac": None,
                        "traffic": args.traffic, "invalid": f"launch {pipe_avg_ms:.4f} ms > step {ms_per_step:.4f} ms"}
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
            # the arithmetic of the path: fp32 with double-float (fp32 pairs) sums
            # and normalisers; the logits' storage type is config.dtype
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {**_config_json(wl, ells, ks, n_sets),
                       "launch": ("pipelined rounds (sdd_block_pipelined): K calls each streaming one round "
                                  "and finishing the one before, + one closing decide, "
                                  + ("in one launch per call (pipe_kernel), " if pipelined_kernel else
                                     "as the decide and streaming kernels (a round above 512 MiB), ")
                                  + (f"as replays of a CUDA graph of {args.graph} calls" if args.graph
                                     else "queued behind a device spin"))},
            "achieved_gbs_step": ws * scan_bytes / (ms_per_step / 1e3) / 1e9,
            "frac_of_8tbs_step": ws * scan_bytes / (ms_per_step / 1e3) / 8e12,
            "roofline": roofline,
            "roofline_scan_kernel": {"bound": "hbm", "kernel": "scan_kernel (sdd_block_scan)",
                                     "achieved": scan_achieved, "peak": peak, "unit": "GB/s",
                                     "frac": scan_achieved / peak,
                                     "traffic": SCAN_TRAFFIC_C3 if args.c3 else None,
                                     "bytes_per_launch": scan_bytes, "avg_launch_ms": scan_avg_ms,
                                     "launches_timed": n_scan},
            "round_unpipelined": unpipelined,
            "cpu_baseline": cpu,
            "parity_sample": parity,
            "e2e": e2e,
            "gpu_launches": (args.steps + 1) if pipelined_kernel else 2 * args.steps,
            "clocks": clk.summary(),
            "device_status": status,
        }
        print(json.dumps(line), flush=True)
    if ws > 1:
        dist.barrier()
        dist.destroy_process_group()
    return 0


def _peak_tflops():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"]), "measured"
    except Exception:
        return 1900.0, "fallback"


def run_component_mlp(args):
    """The stand-in survival scorer alone (decode-loop batch: 4096 positions,
    hidden 3584 -> 256 -> 1), device time from CUDA-graph replays of 16 launches
    over 8 rotating hidden-state buffers (8 x 29 MB > L2)."""
    import torch
    import paper_2608_14787_gb300 as sdd
    from paper_2608_14787_gb300 import build as sdd_build
    from paper_2608_14787_gb300 import synth
    sdd_build.build()
    sdd.load()
    M, K, N = 128 * 32, synth.HIDDEN, 256
    W1, b1, w2, b2 = synth.make_mlp(device="cuda", hidden=K)
    b2 = float(b2.item())
    hs = [synth.make_hidden(M, device="cuda", round_=r) for r in range(8)]
    out = torch.empty(M, device="cuda")
    ws = sdd.scorer_workspace(M, torch.device("cuda"))
    status = sdd.new_status(torch.device("cuda"))
    for i in range(max(args.warmup, 3)):
        sdd.survival_mlp(hs[i % 8], W1, b1, w2, b2, out=out, status=status, workspace=ws)
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        for i in range(16):
            sdd.survival_mlp(hs[i % 8], W1, b1, w2, b2, out=out, status=status, workspace=ws)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    reps = max(1, args.steps // 16)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(None) as clk:
        e0.record()
        for _ in range(reps):
            g.replay()
        e1.record()
        torch.cuda.synchronize()
    t = e0.elapsed_time(e1) / (reps * 16) / 1e3
    flops = 2.0 * M * K * N
    nbytes = M * K * 2 + N * K * 2 + M * 4
    tpk, tkind = _peak_tflops()
    hbm, hkind = _peaks()
    cpu = None
    if not args.no_cpu_baseline:
        import numpy as np
        import oracle as orc
        rows = 512
        t0 = time.perf_counter()
        orc.survival_mlp(synth.bf16_bits(hs[0][:rows]), synth.bf16_bits(W1), b1.cpu().numpy(), synth.bf16_bits(w2), b2)
        dt = time.perf_counter() - t0
        cpu = {"value": rows / dt, "unit": "positions/s", "cores": 1, "kind": "oracle",
               "sample": f"{rows} of the {M} positions, fp64 loops, single thread ({dt:.1f} s)"}
        del np
    line = {
        "component": "a8 survival scorer (sdd_survival_mlp)", "metric": "positions scored/s", "unit": "positions/s",
        "value": M / t, "us_per_call": t * 1e6, "config": {"M": M, "K": K, "N": N, "dtype": "bf16 in, fp32 acc"},
        "roofline": {"bound": "hbm", "achieved_gbs": nbytes / t / 1e9, "peak_gbs": hbm, "frac_hbm": nbytes / t / 1e9 / hbm,
                     "achieved_tflops": flops / t / 1e12, "peak_tflops": tpk,
                     "frac_tensor": flops / t / 1e12 / tpk, "bytes": nbytes, "flops": flops,
                     "peak_source": f"{hkind} hbm_gbs / {tkind} bf16_tflops",
                     "note": "intensity 242 FLOP/B is below the ridge: bytes bound"},
        "cpu_baseline": cpu, "clocks": clk.summary(), "device_status": int(status.item()),
    }
    print(json.dumps(line), flush=True)
    return 0


def run_component_scorer(args):
    """The deep scorer (learned scorer's shape, App. A.7: (3584 + 19) -> 256 ->
    256 -> 256 -> 1) on the decode-loop batch (4096 positions), device time from
    CUDA-graph replays of 16 calls (two launches each) over 8 rotating
    hidden-state buffers (8 x 29 MB > L2)."""
    import torch
    import paper_2608_14787_gb300 as sdd
    from paper_2608_14787_gb300 import build as sdd_build
    from paper_2608_14787_gb300 import synth
    sdd_build.build()
    sdd.load()
    M, Kh, N = 128 * 32, synth.HIDDEN, 256
    w = synth.make_scorer_deep(device="cuda", hidden=Kh)
    hs = [synth.make_hidden(M, device="cuda", round_=r) for r in range(8)]
    fs = [synth.make_features(M, device="cuda", round_=r) for r in range(8)]
    act = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    out = torch.empty(M, device="cuda")
    ws = sdd.scorer_workspace(M, torch.device("cuda"))
    status = sdd.new_status(torch.device("cuda"))
    for i in range(max(args.warmup, 3)):
        sdd.scorer_deep(hs[i % 8], fs[i % 8], *w, act=act, out=out, status=status, workspace=ws)
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        for i in range(16):
            sdd.scorer_deep(hs[i % 8], fs[i % 8], *w, act=act, out=out, status=status, workspace=ws)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    reps = max(1, args.steps // 16)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(None) as clk:
        e0.record()
        for _ in range(reps):
            g.replay()
        e1.record()
        torch.cuda.synchronize()
    t = e0.elapsed_time(e1) / (reps * 16) / 1e3
    K1 = Kh + N
    flops = 2.0 * M * (K1 * N + 2 * N * N + N)
    nbytes = M * K1 * 2 + N * K1 * 2 + 2 * N * N * 2 + 2 * M * N * 2 + M * 4
    tpk, tkind = _peak_tflops()
    hbm, hkind = _peaks()
    cpu = None
    if not args.no_cpu_baseline:
        import oracle as orc
        rows = 128
        x = torch.cat([hs[0][:rows], fs[0][:rows]], dim=-1)
        bits = synth.bf16_bits
        W1, b1, W2, b2, W3, b3, w4, b4 = w
        t0 = time.perf_counter()
        orc.scorer_deep(bits(x), bits(W1), b1.cpu().numpy(), bits(W2), b2.cpu().numpy(), bits(W3), b3.cpu().numpy(),
                        bits(w4), b4)
        dt = time.perf_counter() - t0
        cpu = {"value": rows / dt, "unit": "positions/s", "cores": 1, "kind": "oracle",
               "sample": f"{rows} of the {M} positions, fp64 loops, single thread ({dt:.1f} s)"}
    line = {
        "component": "NEXT-2 deep scorer (sdd_scorer_deep)", "metric": "positions scored/s", "unit": "positions/s",
        "value": M / t, "us_per_call": t * 1e6,
        "config": {"M": M, "K": f"{Kh} + 256 (19 features, zero padded)", "layers": "3840 -> 256 -> 256 -> 256 -> 1",
                   "dtype": "bf16 operands, fp32 accumulation"},
        "roofline": {"bound": "hbm", "achieved_gbs": nbytes / t / 1e9, "peak_gbs": hbm, "frac_hbm": nbytes / t / 1e9 / hbm,
                     "achieved_tflops": flops / t / 1e12, "peak_tflops": tpk, "frac_tensor": flops / t / 1e12 / tpk,
                     "bytes": nbytes, "flops": flops, "peak_source": f"{hkind} hbm_gbs / {tkind} bf16_tflops"},
        "cpu_baseline": cpu, "clocks": clk.summary(), "device_status": int(status.item()),
    }
    print(json.dumps(line), flush=True)
    return 0


def run_component_diag(args):
    """NEXT-4: the permutation diagnostic of Sec. 5 (Table 1's settings: 100
    repetitions; raw (0.90, 0.93), marginal 0.90, conditional (0.90, 0.90)) and
    the positionwise metrics on a synthetic log: raw confidence and
    shadow-verified strict L of 32 fused c3 rounds (512 blocks, gamma = 32).
    The signals all read the raw-confidence log (no trained scorer exists here)."""
    import numpy as np
    import torch
    import paper_2608_14787_gb300 as sdd
    from paper_2608_14787_gb300 import build as sdd_build
    from paper_2608_14787_gb300 import synth
    sdd_build.build()
    sdd.load()
    wl = synth.WORKLOADS["c3"]
    B, gamma, V = wl.B, wl.gamma, wl.V
    rnd = sdd.BlockRound(B, gamma, V, taus=wl.taus, K_min=6, S_max=64)
    qs, Ls = [], []
    for r in range(32):
        blk = synth.make_block(wl, device="cuda", round_=r)
        rnd.set_inputs(blk.z_d, blk.z_t, blk.x, seed=wl.seed, round_=r)
        rnd.run()
        qs.append(rnd.q.clone())
        Ls.append(rnd.L_strict.clone())
        del blk
    q, L = torch.cat(qs), torch.cat(Ls)
    torch.cuda.synchronize()
    nb = q.shape[0]
    settings = [("raw", 0, 0.90, 0.93), ("marginal", 1, 0.90, 0.90), ("conditional", 2, 0.90, 0.90)]
    res, times = {}, []
    with ClockSampler(None) as clk:
        for name, sig, eb, ec in settings:
            sums = sdd.permutation_diagnostic(q, L, signal=sig, eta_b=eb, eta_c=ec, n_rep=100, seed=0)   # warm-up
            torch.cuda.synchronize()
            # device time per call: replays of a CUDA graph of 4 calls (the
            # binding's allocations and marshalling stay outside the timed region)
            side = torch.cuda.Stream()
            side.wait_stream(torch.cuda.current_stream())
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=side):
                for _ in range(4):
                    sdd.permutation_diagnostic(q, L, signal=sig, eta_b=eb, eta_c=ec, n_rep=100, seed=0)
            g.replay()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for _ in range(5):
                g.replay()
            e1.record()
            torch.cuda.synchronize()
            times.append(e0.elapsed_time(e1) / 1e3 / 20)
            s = sums.cpu().numpy()
            res[name] = {"original": float(s[-1]) / nb, "permuted_mean": float(s[:-1].mean()) / nb}
        bce, base, auc, npos, nneg = sdd.position_metrics(q, L)
        torch.cuda.synchronize()
    cpu = None
    if not args.no_cpu_baseline:
        import oracle as orc
        t0 = time.perf_counter()
        orc.permutation_diagnostic(q.double().cpu().numpy(), L.cpu().numpy(), 0, 0.90, 0.93, 10, 0)
        dt = time.perf_counter() - t0
        cpu = {"value": 10 * nb / dt, "unit": "block-repetitions/s", "cores": 1, "kind": "oracle",
               "sample": f"10 of the 100 repetitions of the raw setting over {nb} blocks ({dt:.2f} s)"}
    t_mean = sum(times) / len(times)
    line = {
        "component": "NEXT-4 permutation diagnostic (sdd_permutation_diagnostic)",
        "metric": "block-repetitions/s", "unit": "block-repetitions/s", "value": 100 * nb / t_mean,
        "us_per_call": t_mean * 1e6, "blocks": nb, "gamma": gamma, "repetitions": 100,
        "feasible_prefix_mean": res,
        "mean_bce": float(np.nanmean(bce.cpu().numpy())), "mean_bce_position_only": float(np.nanmean(base.cpu().numpy())),
        "mean_auroc": float(np.nanmean(auc.cpu().numpy())),
        "note": "synthetic raw-confidence log (32 c3 rounds); the paper's Table 1 needs its HumanEval logs",
        "cpu_baseline": cpu, "clocks": clk.summary(),
    }
    print(json.dumps(line), flush=True)
    return 0


def run_component_shard(args):
    """The vocabulary-sharded round on the benchmark's workload (c3: B=16,
    gamma=32, V=151,936 bf16, every rule) with S = --shards ranks played in
    turn on one GPU (vocab_shard.run_local: the exchanges are device-memory
    concatenations and maxima, timed with the rest): blocks/s of the whole
    round, and the per-slice partials kernel alone (bytes of one slice's logits
    over its launch time)."""
    import torch
    import paper_2608_14787_gb300 as sdd
    from paper_2608_14787_gb300 import build as sdd_build
    from paper_2608_14787_gb300 import synth, vocab_shard
    sdd_build.build()
    sdd.load()
    wl, ells, ks = _workload_cfg("c3")
    S = args.shards
    bounds = vocab_shard.slice_bounds(wl.V, S)
    blk = synth.make_block(wl, device="cuda", round_=0)
    sd = [vocab_shard.slice_logits(blk.z_d, v0, v1) for v0, v1 in bounds]
    st = [vocab_shard.slice_logits(blk.z_t, v0, v1) for v0, v1 in bounds]
    ranks = [vocab_shard.ShardRound(wl.B, wl.gamma, wl.V, v0, v1, taus=wl.taus, ells=ells, ks=ks, K_min=6)
             for v0, v1 in bounds]
    for r in range(3):
        vocab_shard.run_local(ranks, sd, st, blk.x, seed=wl.seed, round_=r)
    torch.cuda.synchronize()
    n = max(10, min(args.steps, 200))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(None) as clk:
        torch.cuda._sleep(int(args.prefill_us * 2.0e3))
        e0.record()
        for r in range(n):
            vocab_shard.run_local(ranks, sd, st, blk.x, seed=wl.seed, round_=r)
        e1.record()
        torch.cuda.synchronize()
    round_ms = e0.elapsed_time(e1) / n
    # one slice's partials kernel, back to back
    r0 = ranks[0]
    a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda._sleep(int(2000 * 2.0e3))   # ~2 ms: the 50 launches queue behind it, no host gaps
    a0.record()
    for _ in range(50):
        r0.partials()
    a1.record()
    torch.cuda.synchronize()
    part_ms = a0.elapsed_time(a1) / 50
    w = bounds[0][1] - bounds[0][0]
    slice_bytes = wl.B * (2 * wl.gamma + 1) * w * 2
    peak, kind = _peaks()
    status = max(int(r.status.item()) for r in ranks)
    line = {"component": f"vocabulary-sharded round, S = {S} ranks played in turn on one GPU",
            "metric": "blocks/s", "unit": "blocks/s", "value": wl.B / (round_ms / 1e3), "ms_per_round": round_ms,
            "config": {"workload": "c3", "B": wl.B, "gamma": wl.gamma, "V": wl.V, "shards": S,
                       "slices": [list(b) for b in bounds]},
            "partials_kernel": {"ms": part_ms, "bytes": slice_bytes, "achieved_gbs": slice_bytes / (part_ms / 1e3) / 1e9,
                                "peak": peak, "frac": slice_bytes / (part_ms / 1e3) / 1e9 / peak,
                                "peak_source": f"{kind} hbm_gbs"},
            "clocks": clk.summary(), "device_status": status}
    print(json.dumps(line), flush=True)
    return 0


def run_component_features(args):
    """Drafter confidence with and without the extended features (App. A.7:
    probability margin, top-5 mass) on the drafter half of the c3 workload
    (16 blocks x 32 rows x 151,936 bf16 = 155.6 MB), 3 rotating input sets
    (> L2); device time per call (streaming + decide kernels) from CUDA events
    around replays of a CUDA graph of 24 calls (the binding's per-call output
    allocations and argument marshalling stay out of the timed region)."""
    import torch
    import paper_2608_14787_gb300 as sdd
    from paper_2608_14787_gb300 import build as sdd_build
    from paper_2608_14787_gb300 import synth
    sdd_build.build()
    sdd.load()
    wl = synth.WORKLOADS["c3"]
    B, gamma, V = wl.B, wl.gamma, wl.V
    sets = [synth.make_block(wl, device="cuda", round_=r) for r in range(3)]
    ws = sdd.Workspace(B, gamma, V, torch.device("cuda"))
    status = sdd.new_status(torch.device("cuda"))
    steps = max(args.steps // 8, 64)

    def timed(features):
        for i in range(max(args.warmup, 3)):
            sdd.confidence(sets[i % 3].z_d, sets[i % 3].x, ws=ws, status=status, features=features)
        torch.cuda.synchronize()
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=side):
            for i in range(24):
                sdd.confidence(sets[i % 3].z_d, sets[i % 3].x, ws=ws, status=status, features=features)
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        reps = max(1, steps // 24)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            g.replay()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / (24 * reps) / 1e3
    with ClockSampler(None) as clk:
        t_plain = timed(False)
        t_feat = timed(True)
    nbytes = B * gamma * V * 2
    hbm, hkind = _peaks()
    cpu = None
    if not args.no_cpu_baseline:
        import oracle as orc
        rows = 16
        t0 = time.perf_counter()
        orc.row_features(synth.bf16_bits(sets[0].z_d[0, :rows]))
        orc.row_stats(synth.bf16_bits(sets[0].z_d[0, :rows]), tokens=sets[0].x[0, :rows].cpu().numpy())
        dt = time.perf_counter() - t0
        cpu = {"value": rows / dt, "unit": "rows/s", "cores": 1, "kind": "oracle",
               "sample": f"{rows} drafter rows of one block, stats + features, single thread ({dt:.2f} s)"}
    line = {
        "component": "NEXT-2 extended features (sdd_confidence_features)", "metric": "drafter rows scored/s",
        "unit": "rows/s", "value": B * gamma / t_feat, "us_per_call": t_feat * 1e6,
        "us_per_call_without_features": t_plain * 1e6,
        "config": {"B": B, "gamma": gamma, "V": V, "dtype": "bf16", "rows": B * gamma},
        "roofline": {"bound": "hbm", "achieved": nbytes / t_feat / 1e9, "peak": hbm, "unit": "GB/s",
                     "frac": nbytes / t_feat / 1e9 / hbm, "bytes": nbytes, "peak_source": f"{hkind} hbm_gbs",
                     "note": "whole call (streaming + decide kernels) per launch pair"},
        "cpu_baseline": cpu, "clocks": clk.summary(), "device_status": int(status.item()),
    }
    print(json.dumps(line), flush=True)
    return 0


def run_component_loop(args):
    """The decode-loop workload (B=128, gamma=32, V=151,936 bf16): `--steps`
    rounds (default 256, the workload's count), enqueued back to back with no
    host round trip (inputs: 8 seeded sets generated before the timed region)."""
    import torch
    from paper_2608_14787_gb300 import build as sdd_build
    from paper_2608_14787_gb300 import loop as sdd_loop
    from paper_2608_14787_gb300 import synth
    sdd_build.build()
    rounds = args.steps if args.steps != 4000 else 256
    with ClockSampler(None) as clk:
        res = sdd_loop.run(rounds, "c5", warmup=max(2, min(args.warmup, 4)))
    cpu = None
    if not args.no_cpu_baseline:
        import numpy as np
        import oracle as orc
        wl = synth.WORKLOADS["c5"]
        blk = synth.make_block(wl, device="cuda", round_=0, B=1)
        zd, zt, x = synth.bf16_bits(blk.z_d[0]), synth.bf16_bits(blk.z_t[0]), blk.x[0].cpu().numpy()
        t0 = time.perf_counter()
        st = orc.row_stats(zd, tokens=x)
        orc.schedule(st.q[None], orc.SIG_RAW, 0.9, 0.9, 6, 64)
        orc.verify_strict(zt, zd, x, seed=wl.seed, b=0, round_=0)
        dt = time.perf_counter() - t0
        cpu = {"value": 1.0 / dt, "unit": "blocks/s", "cores": 1, "kind": "oracle",
               "sample": f"one block of one round (confidence, schedule, strict verification), single thread "
                         f"({dt:.1f} s)"}
        del np
    res.update({"component": "decode loop (c5)", "metric": "blocks/s", "unit": "blocks/s",
                "value": res["blocks_per_s"], "cpu_baseline": cpu, "clocks": clk.summary()})
    torch.cuda.synchronize()
    print(json.dumps(res), flush=True)
    return 0


def _launch_ranks(n: int) -> int:
    """`--gpus N` without a launcher around it: start N ranks of this same
    command, one per GPU, through torch.distributed.run on 127.0.0.1 (each rank
    reads RANK / LOCAL_RANK / WORLD_SIZE; rank 0 prints the line)."""
    import socket
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as sk:
        sk.bind(("127.0.0.1", 0))
        port = sk.getsockname()[1]
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={n}",
           "--master-addr=127.0.0.1", f"--master-port={port}", os.path.abspath(__file__)] + sys.argv[1:]
    return subprocess.call(cmd)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=4000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--workload", default="c3")
    ap.add_argument("--blocks", type=int, default=None, help="override the workload's batch size B")
    ap.add_argument("--graph", type=int, default=0, help="replay a CUDA graph of this many rounds (small workloads)")
    ap.add_argument("--cpu-blocks", type=int, default=8, help="blocks of the single-thread oracle sample")
    ap.add_argument("--ref-threads", type=int, default=0, help="host threads of --impl reference (0: all cores)")
    ap.add_argument("--scan-launches", type=int, default=60, help="back-to-back streaming launches for the roofline")
    ap.add_argument("--prefill-us", type=float, default=200.0, help="device spin before the start event")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--sets", type=int, default=3, help="rotating input sets (3 x 316 MB exceeds L2)")
    ap.add_argument("--traffic", type=float, default=None,
                    help="dram bytes per scan launch from an ncu capture of the current kernel")
    ap.add_argument("--shards", type=int, default=2, help="--component shard: vocabulary slices")
    ap.add_argument("--component", default=None, choices=["mlp", "loop", "features", "scorer", "diag", "shard"],
                    help="measure one other row of the path instead of the fused round")
    args = ap.parse_args()
    if args.gpus > 1 and "WORLD_SIZE" not in os.environ:
        return _launch_ranks(args.gpus)
    if args.component == "mlp":
        return run_component_mlp(args)
    if args.component == "loop":
        return run_component_loop(args)
    if args.component == "features":
        return run_component_features(args)
    if args.component == "scorer":
        return run_component_scorer(args)
    if args.component == "diag":
        return run_component_diag(args)
    if args.component == "shard":
        return run_component_shard(args)
    if args.traffic is None and args.workload == "c3" and args.blocks in (None, 16):
        args.traffic = PIPE_TRAFFIC_C3
    args.c3 = args.workload == "c3" and args.blocks in (None, 16)
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        return run_reference(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())
