"""Multi-rank host logic on CPU (two gloo ranks): blocks shard across ranks
with no data-path exchange; the agreement counters of Sec. 3.2 (Eq. 1-2) and
timings are the only cross-rank reductions, and their sum over ranks must
equal the single-rank counters of the whole batch (oracle)."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

from paper_2608_14787_gb300 import shard

WORLD = 2
N_TAU, B, GAMMA = 3, 37, 32


def _free_port():
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _inputs():
    rng = np.random.default_rng(2608)
    K = rng.integers(0, GAMMA + 1, size=(N_TAU, B)).astype(np.int32)
    K[:, ::5] = 0                      # some verified (not skipped) blocks
    L = rng.integers(0, GAMMA + 1, size=B).astype(np.int32)
    return K, L


def _worker(rank, port, outdir):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    import torch.distributed as dist
    import oracle
    dist.init_process_group("gloo", rank=rank, world_size=WORLD)
    try:
        K, L = _inputs()
        s, e = shard.block_range(B, rank, WORLD)
        acc = torch.from_numpy(np.stack([oracle.agreement(K[t, s:e], L[s:e]) for t in range(N_TAU)]))
        tot = shard.sum_counters(acc)
        mx = shard.max_over_ranks(1.5 * (rank + 1))
        np.save(os.path.join(outdir, f"tot{rank}.npy"), tot.numpy())
        np.save(os.path.join(outdir, f"max{rank}.npy"), np.array([mx]))
        np.save(os.path.join(outdir, f"local{rank}.npy"), acc.numpy())
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_block_range_partitions():
    for n in (0, 1, 7, 16, 37, 4096):
        for w in (1, 2, 3, 8):
            got = [shard.block_range(n, r, w) for r in range(w)]
            assert got[0][0] == 0 and got[-1][1] == n
            assert all(got[r][1] == got[r + 1][0] for r in range(w - 1))
            sizes = [e - s for s, e in got]
            assert max(sizes) - min(sizes) <= 1
    with pytest.raises(ValueError):
        shard.block_range(4, 2, 2)


def test_single_rank_is_identity(orc):
    K, L = _inputs()
    acc = torch.from_numpy(np.stack([orc.agreement(K[t], L) for t in range(N_TAU)]))
    assert torch.equal(shard.sum_counters(acc), acc)
    assert shard.max_over_ranks(3.25) == 3.25


def test_agreement_rates_from_counters():
    acc = torch.tensor([[6, 8, 1, 2], [0, 0, 0, 0]], dtype=torch.int64)
    (st, fp, n), (st2, fp2, n2) = shard.agreement_rates(acc)
    assert (st, fp, n) == (0.75, 0.5, 2)
    assert np.isnan(st2) and np.isnan(fp2) and n2 == 0


def test_two_gloo_ranks_sum_to_whole_batch(orc, tmp_path):
    K, L = _inputs()
    want = np.stack([orc.agreement(K[t], L) for t in range(N_TAU)])
    mp.spawn(_worker, args=(_free_port(), str(tmp_path)), nprocs=WORLD, join=True)
    locals_ = [np.load(tmp_path / f"local{r}.npy") for r in range(WORLD)]
    assert not np.array_equal(locals_[0], want)          # each rank saw only its shard
    for r in range(WORLD):
        np.testing.assert_array_equal(np.load(tmp_path / f"tot{r}.npy"), want)
        assert np.load(tmp_path / f"max{r}.npy")[0] == 1.5 * WORLD


# ---------------------------------------------------------------------------
# Vocabulary-sharded round: the exchanges between ranks (vocab_shard), with
# stand-in record bytes (the records themselves come from the GPU kernels and
# are checked by tests/test_gpu_shard.py)
# ---------------------------------------------------------------------------
ROWS = 13


def _records(rank):
    g = torch.Generator().manual_seed(100 + rank)
    return torch.randint(0, 256, (ROWS * 160,), dtype=torch.uint8, generator=g)


def _tokens(rank):
    # every rank holds -1 at the drawn positions except the rank that drew them
    t = torch.full((4, 9), -1, dtype=torch.int32)
    t[:, :3] = torch.arange(12, dtype=torch.int32).view(4, 3)
    t[rank, 3 + rank] = 1000 + rank
    return t


def _exchange_worker(rank, port, outdir):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    import torch.distributed as dist
    from paper_2608_14787_gb300 import vocab_shard
    dist.init_process_group("gloo", rank=rank, world_size=WORLD)
    try:
        allr = vocab_shard._all_gather(_records(rank), WORLD, None)
        mass = torch.tensor([[rank + 0.5, 2.0 * rank]] * 3, dtype=torch.float32)
        allm = vocab_shard._all_gather(mass.reshape(-1), WORLD, None).reshape(WORLD, 3, 2)
        tok = _tokens(rank)
        vocab_shard._all_reduce_max(tok, None)
        torch.save({"rec": allr, "mass": allm, "tok": tok}, os.path.join(outdir, f"ex{rank}.pt"))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_vocab_shard_exchanges_two_gloo_ranks(tmp_path):
    """All-gather of the record bytes (slice order), of the draw-row masses,
    and the MAX all-reduce that completes the drawn tokens: every rank ends
    with the same buffers, equal to the single-process concatenation."""
    mp.spawn(_exchange_worker, args=(_free_port(), str(tmp_path)), nprocs=WORLD, join=True)
    want_rec = torch.stack([_records(r) for r in range(WORLD)])
    want_tok = torch.stack([_tokens(r) for r in range(WORLD)]).amax(dim=0)
    for r in range(WORLD):
        got = torch.load(tmp_path / f"ex{r}.pt")
        assert torch.equal(got["rec"], want_rec)
        assert torch.equal(got["mass"][1, 0], torch.tensor([1.5, 2.0]))
        assert torch.equal(got["tok"], want_tok)
        assert got["tok"][0, 3] == 1000 and got["tok"][1, 4] == 1001


def test_slice_bounds_cover_the_vocabulary():
    from paper_2608_14787_gb300 import vocab_shard
    for V in (1, 7, 8, 1003, 151_936):
        for S in (1, 2, 3, 8):
            b = vocab_shard.slice_bounds(V, S)
            assert b[0][0] == 0 and b[-1][1] == V
            assert all(b[i][1] == b[i + 1][0] for i in range(len(b) - 1))
            assert all(v0 % 8 == 0 and v1 > v0 for v0, v1 in b)
