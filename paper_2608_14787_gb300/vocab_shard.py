"""The vocabulary-sharded round (a tensor-parallel LM head) through the C ABI.

Rank s of S holds the contiguous vocabulary slice [v0_s, v1_s) of every
drafter and target row.  A round is three library calls with an exchange after
each of the first two, and a MAX reduction of the token arrays at the end (see
sdd_shard_partials / sdd_shard_decide / sdd_shard_draw in include/sdd.h):

    records  = shard_partials(slice)            # [rows] sdd_shard_partial, 160 B each
    all      = all_gather(records)              # [S, rows]
    mass     = shard_decide(all)                # outputs of the round; [B, 2] draw-row masses
    all_mass = all_gather(mass)                 # [S, B, 2]      (strict sampling only)
    shard_draw(all_mass)                        # the owning rank writes the drawn tokens
    all_reduce_max(tokens_strict, commit_tokens)

Every step runs in libsdd.so; this module sizes the buffers, slices the
vocabulary and moves the bytes between ranks (torch.distributed: all-gather
and a MAX all-reduce; gloo or NCCL, no peer loads).  `run_local` plays the S
ranks one after another on one device with the exchanges done in device
memory.
"""
from __future__ import annotations

import ctypes

import torch

from . import binding as sdd

RECORD_BYTES = 160


def slice_bounds(V: int, S: int):
    """Contiguous slices [v0, v1) covering [0, V), as equal as possible, each
    start a multiple of 8 entries (so that a slice copied out of a row keeps
    16-byte aligned vectors)."""
    q = 8
    units = -(-V // q)
    cuts = [min(V, (units * s // S) * q) for s in range(S + 1)]
    cuts[-1] = V
    return [(cuts[s], cuts[s + 1]) for s in range(S) if cuts[s + 1] > cuts[s]]


def slice_logits(z: torch.Tensor, v0: int, v1: int) -> torch.Tensor:
    """Columns [v0, v1) of logits [B, P, V] as a rank would hold them: their own
    array, rows padded to a 16-byte multiple."""
    B, P, _ = z.shape
    esz = z.element_size()
    w = v1 - v0
    stride = -(-w * esz // 16) * 16 // esz
    out = torch.empty(B, P, stride, dtype=z.dtype, device=z.device)
    out[..., :w] = z[..., v0:v1]
    if stride > w:
        out[..., w:] = float("nan")      # padding: never read into a result
    return out[..., :w]


def workspace_bytes(B: int) -> int:
    n = ctypes.c_size_t(0)
    sdd._check(sdd.load().sdd_shard_workspace_size(B, ctypes.byref(n)), "sdd_shard_workspace_size")
    return int(n.value)


class ShardRound:
    """One rank's buffers for the sharded round of B blocks (its slice of the
    vocabulary [v0, v1) of V).  Outputs after the round have the names and
    layouts of binding.BlockRound's."""

    def __init__(self, B, gamma, V, v0, v1, *, dtype=torch.bfloat16, taus=(0.9,), ells=(), ks=(), greedy=False,
                 K_min=6, S_max=64, device="cuda"):
        self.B, self.gamma, self.V, self.v0, self.v1 = B, gamma, V, v0, v1
        self.rnd = sdd.BlockRound(B, gamma, V, dtype=dtype, taus=taus, ells=ells, ks=ks, greedy=greedy,
                                  K_min=K_min, S_max=S_max, device=device)
        dev = torch.device(device)
        self.greedy = greedy
        self.rows = B * (2 * gamma + 1)
        self.records = torch.empty(self.rows * RECORD_BYTES, dtype=torch.uint8, device=dev)
        self.mass = torch.zeros(B, 2, dtype=torch.float32, device=dev)
        nb = workspace_bytes(B)
        self.ws = torch.zeros(max(nb, 16) + 256, dtype=torch.uint8, device=dev)
        off = (-self.ws.data_ptr()) % 256
        self.rnd.args.workspace = self.ws.data_ptr() + off
        self.rnd.args.workspace_bytes = nb

    def __getattr__(self, name):
        # outputs (q, L_strict, tokens_strict, K, ...) live in the BlockRound
        return getattr(self.__dict__["rnd"], name)

    def set_inputs(self, z_d_slice, z_t_slice, x, *, seed=0, round_=0):
        """z_d_slice [B, gamma, w], z_t_slice [B, gamma+1, w]: this rank's columns
        (w = v1 - v0; rows 16-byte aligned, any padded stride)."""
        a = self.rnd.args
        Vs, stride = sdd._logits_layout(z_d_slice, "z_d")
        Vt, stride_t = sdd._logits_layout(z_t_slice, "z_t")
        if (Vs, stride) != (Vt, stride_t) or Vs != self.v1 - self.v0:
            raise ValueError("slices must be [., ., v1 - v0] with one row stride")
        a.draft_logits, a.target_logits, a.draft_tokens = z_d_slice.data_ptr(), z_t_slice.data_ptr(), x.data_ptr()
        a.row_stride = stride
        a.seed, a.round = seed, round_
        self._keep = (z_d_slice, z_t_slice, x)

    def partials(self, stream=None):
        sdd._check(sdd.load().sdd_shard_partials(ctypes.byref(self.rnd.args), self.v0, self.v1,
                                                 ctypes.c_void_p(self.records.data_ptr()), sdd._stream(stream)),
                   "sdd_shard_partials")
        return self.records

    def decide(self, all_records: torch.Tensor, n_shards: int, stream=None):
        sdd._check(sdd.load().sdd_shard_decide(ctypes.byref(self.rnd.args), self.v0, self.v1, n_shards,
                                               ctypes.c_void_p(all_records.data_ptr()),
                                               ctypes.c_void_p(self.mass.data_ptr()), sdd._stream(stream)),
                   "sdd_shard_decide")
        return self.mass

    def draw(self, all_mass: torch.Tensor, n_shards: int, shard: int, stream=None):
        sdd._check(sdd.load().sdd_shard_draw(ctypes.byref(self.rnd.args), self.v0, self.v1, n_shards, shard,
                                             ctypes.c_void_p(all_mass.data_ptr()), sdd._stream(stream)),
                   "sdd_shard_draw")

    @property
    def sampling(self):
        return not self.greedy


def run_local(ranks, slices_d, slices_t, x, *, seed=0, round_=0):
    """Play S ranks (ShardRound objects in slice order) on one device: each
    rank's calls run in turn, and the exchanges are concatenations and
    element-wise maxima of device tensors.  Returns the ranks."""
    S = len(ranks)
    for r, zd, zt in zip(ranks, slices_d, slices_t):
        r.set_inputs(zd, zt, x, seed=seed, round_=round_)
        r.partials()
    all_rec = torch.cat([r.records for r in ranks])
    for r in ranks:
        r.decide(all_rec, S)
    if ranks[0].sampling:
        all_mass = torch.stack([r.mass for r in ranks])
        for s, r in enumerate(ranks):
            r.draw(all_mass, S, s)
        for name in ("tokens_strict", "commit_tokens"):
            top = torch.stack([getattr(r, name) for r in ranks]).amax(dim=0)
            for r in ranks:
                getattr(r, name).copy_(top)
    return ranks


def run_distributed(rank_round: ShardRound, z_d_slice, z_t_slice, x, group=None, *, seed=0, round_=0):
    """This process's part of the sharded round under torch.distributed (one
    rank per slice, ranks in slice order).  Exchanges go through
    all_gather / all_reduce(MAX) on the tensors' device, or
    through host copies when the group's backend is gloo and the data is on
    a GPU."""
    import torch.distributed as dist
    S = dist.get_world_size(group)
    me = dist.get_rank(group)
    r = rank_round
    r.set_inputs(z_d_slice, z_t_slice, x, seed=seed, round_=round_)
    rec = r.partials()
    all_rec = _all_gather(rec, S, group)
    r.decide(all_rec, S)
    if r.sampling:
        all_mass = _all_gather(r.mass.reshape(-1), S, group).reshape(S, r.B, 2)
        r.draw(all_mass, S, me)
        for name in ("tokens_strict", "commit_tokens"):
            _all_reduce_max(getattr(r, name), group)
    return r


def _on_host(group):
    import torch.distributed as dist
    return dist.get_backend(group) == "gloo"


def _all_gather(t: torch.Tensor, S: int, group):
    import torch.distributed as dist
    src = (t.cpu() if (_on_host(group) and t.is_cuda) else t).contiguous()
    parts = [torch.empty_like(src) for _ in range(S)]
    dist.all_gather(parts, src, group=group)
    return torch.stack(parts).to(t.device)


def _all_reduce_max(t: torch.Tensor, group):
    import torch.distributed as dist
    if _on_host(group) and t.is_cuda:
        h = t.cpu()
        dist.all_reduce(h, op=dist.ReduceOp.MAX, group=group)
        t.copy_(h)
    else:
        dist.all_reduce(t, op=dist.ReduceOp.MAX, group=group)
