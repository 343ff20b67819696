"""The vocabulary-sharded round (a tensor-parallel LM head, each rank holding a
contiguous vocabulary slice of every row) against the fp64 oracle on the
whole rows: S ranks are played one after another on one GPU
(vocab_shard.run_local: the exchanges are device-memory concatenations and
maxima), and, separately, as two processes on the one GPU exchanging through
gloo.  Decisions bit-exact outside the flagged band, statistics within the
float tolerance, and the sharded outputs equal to the one-GPU sdd_block's."""
import os

import numpy as np
import pytest
import torch

import paper_2608_14787_gb300 as sdd
from paper_2608_14787_gb300 import synth, vocab_shard
from parity_util import Tally, assert_close_stats, compare_rule, oracle_block

pytestmark = pytest.mark.gpu


def _sharded(blk, S, *, taus, ells, ks, greedy=False, seed=7, round_=1, K_min=2, bounds=None):
    B, gamma, V = blk.x.shape[0], blk.x.shape[1], blk.z_d.shape[-1]
    bounds = bounds or vocab_shard.slice_bounds(V, S)
    ranks = [vocab_shard.ShardRound(B, gamma, V, v0, v1, dtype=blk.z_d.dtype, taus=taus, ells=ells, ks=ks,
                                    greedy=greedy, K_min=K_min) for v0, v1 in bounds]
    sd = [vocab_shard.slice_logits(blk.z_d, v0, v1) for v0, v1 in bounds]
    st = [vocab_shard.slice_logits(blk.z_t, v0, v1) for v0, v1 in bounds]
    vocab_shard.run_local(ranks, sd, st, blk.x, seed=seed, round_=round_)
    torch.cuda.synchronize()
    for r in ranks:
        assert int(r.status.item()) == 0
    return ranks


def _rows16(z):
    """The same logits with rows padded to a 16-byte multiple (+inf padding,
    never read into a result), as the one-GPU call requires."""
    B, P, V = z.shape
    esz = z.element_size()
    stride = -(-V * esz // 16) * 16 // esz
    if stride == V:
        return z
    buf = torch.full((B, P, stride), float("inf"), dtype=z.dtype, device=z.device)
    buf[..., :V] = z
    return buf[..., :V]


def _compare_with_oracle(r0, blk, taus, ells, ks, greedy, seed, round_, K_min):
    ob = oracle_block(blk.z_d, blk.z_t, blk.x, seed=seed, round_=round_, pairs=[(t, t) for t in taus],
                      K_min=K_min, S_max=64, ells=ells, ks=ks, sampling=not greedy)
    dt = blk.z_d.dtype
    for name in ("q", "maxprob", "lse", "entropy"):
        assert_close_stats(name, getattr(r0, name), getattr(ob.stats, name), dt)
    np.testing.assert_array_equal(r0.argmax.cpu().numpy(), ob.stats.argmax)
    B = blk.x.shape[0]
    blocks = list(range(B))
    tally = Tally()
    compare_rule(tally, "strict", r0.L_strict, r0.tokens_strict, ob.greedy if greedy else ob.strict, blocks)
    for i, e in enumerate(ells):
        compare_rule(tally, f"lenient {e}", r0.L_lenient[i], r0.tokens_lenient[i], ob.lenient[e], blocks)
    for i, k in enumerate(ks):
        compare_rule(tally, f"top-{k}", r0.L_topk[i], r0.tokens_topk[i], ob.topk[k], blocks)
    for t, tau in enumerate(taus):
        oKh, oK, oD, mg = ob.sched[(tau, tau)]
        for b in blocks:
            tally.check(f"schedule {tau} block {b}", r0.K[t, b].item() == oK[b] and r0.K_hat[t, b].item() == oKh[b],
                        mg[b])
    return tally, ob


def _same_as_one_gpu(ranks, blk, taus, ells, ks, greedy, seed, round_, K_min, ob):
    """The sharded outputs equal sdd_block's on the whole rows; blocks whose
    strict decision or schedule lies within 1e-6 of a threshold in the oracle
    are left out (the two sum the same terms in different orders)."""
    B, gamma, V = blk.x.shape[0], blk.x.shape[1], blk.z_d.shape[-1]
    rnd = sdd.BlockRound(B, gamma, V, dtype=blk.z_d.dtype, taus=taus, ells=ells, ks=ks, greedy=greedy, K_min=K_min)
    rnd.set_inputs(_rows16(blk.z_d), _rows16(blk.z_t), blk.x, seed=seed, round_=round_)
    rnd.run()
    torch.cuda.synchronize()
    strict = ob.greedy if greedy else ob.strict
    sure = [b for b in range(B) if strict[b][2] >= 1e-6 and all(ob.sched[(t, t)][3][b] >= 1e-6 for t in taus)]
    assert len(sure) >= B // 2
    block_dim = {"L_strict": 0, "tokens_strict": 0, "n_strict": 0, "commit_tokens": 0, "commit_n": 0, "K": 1,
                 "K_hat": 1, "L_lenient": 1, "tokens_lenient": 1, "L_topk": 1, "tokens_topk": 1}
    idx = torch.tensor(sure, device=blk.x.device)
    for r in ranks:
        for name, dim in block_dim.items():
            a, c = getattr(r, name), getattr(rnd, name)
            assert torch.equal(a.index_select(dim, idx), c.index_select(dim, idx)), name
        assert torch.equal(r.argmax, rnd.argmax)


@pytest.mark.parametrize("S", [2, 3, 8])
def test_sharded_round_full_vocabulary(S):
    """B = 6 blocks of gamma = 32 over V = 151,936 bf16 (the benchmark's
    shapes), strict sampling, lenience and top-k grids, tau grid."""
    blk = synth.make_block("c3", device="cuda", B=6, gamma=32, round_=S)
    taus, ells, ks = (0.5, 0.9), (1.0, 0.5, 0.25), (2, 5, 10)
    ranks = _sharded(blk, S, taus=taus, ells=ells, ks=ks)
    tally, ob = _compare_with_oracle(ranks[0], blk, taus, ells, ks, False, 7, 1, 2)
    print(f"S={S}", tally)
    _same_as_one_gpu(ranks, blk, taus, ells, ks, False, 7, 1, 2, ob)
    for r in ranks[1:]:   # every rank ends the round with the same outputs
        assert torch.equal(r.tokens_strict, ranks[0].tokens_strict) and torch.equal(r.q, ranks[0].q)


def test_sharded_greedy_and_ragged_fp32():
    """Greedy strict with fp32 logits, V = 20,011 cut into uneven slices (the
    last one not a whole number of vectors), padded strides."""
    blk = synth.make_block("c3", device="cuda", B=5, gamma=12, V=20_011, dtype=torch.float32, greedy_drafts=True)
    taus, ells, ks = (0.8,), (0.5,), (1, 3, 16)
    bounds = [(0, 4096), (4096, 4104), (4104, 13000), (13000, 20_011)]
    ranks = _sharded(blk, 4, taus=taus, ells=ells, ks=ks, greedy=True, bounds=bounds)
    _, ob = _compare_with_oracle(ranks[0], blk, taus, ells, ks, True, 7, 1, 2)
    _same_as_one_gpu(ranks, blk, taus, ells, ks, True, 7, 1, 2, ob)


def test_sharded_rounds_reuse_their_workspaces():
    """The same ranks (workspaces, arrival counters) serve two rounds in a
    row: the draw's counters are left at zero by every call, so the second
    round matches the oracle as the first does."""
    blk = synth.make_block("c3", device="cuda", B=5, gamma=12, V=40_000, round_=9)
    taus, ells, ks = (0.6,), (0.5,), (3,)
    bounds = vocab_shard.slice_bounds(40_000, 3)
    ranks = [vocab_shard.ShardRound(5, 12, 40_000, v0, v1, dtype=blk.z_d.dtype, taus=taus, ells=ells, ks=ks, K_min=2)
             for v0, v1 in bounds]
    sd = [vocab_shard.slice_logits(blk.z_d, v0, v1) for v0, v1 in bounds]
    st = [vocab_shard.slice_logits(blk.z_t, v0, v1) for v0, v1 in bounds]
    for seed, round_ in ((7, 1), (8, 2)):
        vocab_shard.run_local(ranks, sd, st, blk.x, seed=seed, round_=round_)
        torch.cuda.synchronize()
        for r in ranks:
            assert int(r.status.item()) == 0
        _compare_with_oracle(ranks[0], blk, taus, ells, ks, False, seed, round_, 2)


def test_sharded_bonus_draw_identical_rows():
    """p_t = p_d: every position accepts and the bonus token is drawn from p_t
    of row gamma + 1 across the slices (Sec. 3.1)."""
    blk = synth.make_block("c3", device="cuda", B=4, gamma=8, V=30_000)
    blk.z_t = torch.cat([blk.z_d, blk.z_d[:, -1:]], dim=1).contiguous()
    ranks = _sharded(blk, 3, taus=(0.9,), ells=(), ks=())
    assert torch.all(ranks[0].L_strict == 8)
    _compare_with_oracle(ranks[0], blk, (0.9,), (), (), False, 7, 1, 2)


def test_sharded_tokens_on_slice_boundaries():
    """Drafted tokens at the first and last index of every slice."""
    blk = synth.make_block("c3", device="cuda", B=3, gamma=8, V=12_000)
    bounds = vocab_shard.slice_bounds(12_000, 3)
    edges = [v for b in bounds for v in (b[0], b[1] - 1)]
    x = blk.x.clone()
    for i in range(x.numel()):
        x.view(-1)[i] = edges[i % len(edges)]
    blk.x = x
    ranks = _sharded(blk, 3, taus=(0.5,), ells=(0.5,), ks=(2, 16), bounds=bounds)
    _compare_with_oracle(ranks[0], blk, (0.5,), (0.5,), (2, 16), False, 7, 1, 2)


def _two_process_worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    torch.cuda.set_device(0)
    sdd.load()
    blk = synth.make_block("c3", device="cuda", B=4, gamma=16, V=50_000, round_=5)
    v0, v1 = vocab_shard.slice_bounds(50_000, world)[rank]
    r = vocab_shard.ShardRound(4, 16, 50_000, v0, v1, taus=(0.9,), ells=(0.5,), ks=(5,), K_min=2)
    vocab_shard.run_distributed(r, vocab_shard.slice_logits(blk.z_d, v0, v1), vocab_shard.slice_logits(blk.z_t, v0, v1),
                                blk.x, seed=3, round_=2)
    torch.cuda.synchronize()
    q.put((rank, int(r.status.item()), r.L_strict.cpu(), r.tokens_strict.cpu(), r.K.cpu(), r.commit_tokens.cpu(),
           r.L_topk.cpu(), r.tokens_topk.cpu()))
    dist.barrier()
    dist.destroy_process_group()


def test_two_processes_exchange_through_gloo():
    """Two ranks as two processes on the one GPU (no kernel waits on another:
    every exchange is a gloo collective between launches); both end with the
    outputs of the single-process sharded round."""
    import socket
    import torch.multiprocessing as mp
    with socket.socket() as sk:
        sk.bind(("127.0.0.1", 0))
        port = sk.getsockname()[1]
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_two_process_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted([q.get(timeout=300) for _ in procs], key=lambda t: t[0])
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    blk = synth.make_block("c3", device="cuda", B=4, gamma=16, V=50_000, round_=5)
    ranks = _sharded(blk, 2, taus=(0.9,), ells=(0.5,), ks=(5,), seed=3, round_=2)
    for _, status, L, tok, K, ct, Lk, tk in res:
        assert status == 0
        assert torch.equal(L, ranks[0].L_strict.cpu()) and torch.equal(tok, ranks[0].tokens_strict.cpu())
        assert torch.equal(K, ranks[0].K.cpu()) and torch.equal(ct, ranks[0].commit_tokens.cpu())
        assert torch.equal(Lk, ranks[0].L_topk.cpu()) and torch.equal(tk, ranks[0].tokens_topk.cpu())
    _compare_with_oracle(ranks[0], blk, (0.9,), (0.5,), (5,), False, 3, 2, 2)
