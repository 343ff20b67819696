"""Seeded synthetic inputs shaped like the paper's drafter/target logits.

The paper decodes with DiffuCoder-7B (drafter) and Qwen3-32B (verifier) on
HumanEval (Sec. 5.1); those weights and that dataset are not available here, so
these generators stand in for them: logits with the Qwen vocabulary size
(151,936), the paper's block length (gamma = 32, Sec. 5.1) and structure that
exercises both confident (skippable) and flat (non-skippable) positions.

This module only draws random numbers with torch generators and shapes them.
It computes none of the path's statistics or decisions; both the CUDA path and
the CPU oracle receive the identical tensors it returns.

Recipes (per workload):

* ``tiny``  -- B=1, gamma=8, V=32,000, fp32.  Rows ~ N(0, 2) (2 is the
  standard deviation) with +6 added at one seeded token per row; target =
  drafter + N(0, 0.5).
* ``c2``    -- B=1, gamma=32, V=151,936, bf16.  n ~ N(0, 1) with a planted top
  token 2 above the row's largest other entry; drafter = n / T_j with
  T_j ~ U[0.3, 1.5]; target = 0.9 * drafter + N(0, 0.7).
* ``c3``    -- B=16, gamma=32, V=151,936, bf16.  Per batch row, break points
  a ~ U{0..gamma/2}, f ~ U{1..gamma/2}; positions [0, a) and [a+f, gamma/2+f)
  are peaked, the rest flat.  Peaked rows: N(0, 1) plus one planted token at
  ln(V-1) + 1/2 + 8, i.e. 8 nats above the expected log-sum-exp of the other
  V-1 entries (E exp(N(0,1)) = e^(1/2)), so its probability is close to
  sigmoid(8).  Flat rows: N(0, 0.5).  Target = drafter + N(0, 0.5).
* ``c4``    -- B=64, gamma=64: as c3 with the target noise scale drawn per batch
  row from U[0.2, 1.2].
* ``c5``    -- B=128, gamma=32: c3-style logits drawn afresh every round, plus
  drafter hidden states h ~ N(0, 1) [B*gamma, 3584] and a random-init survival
  MLP 3584 -> 256 -> 1 (W1, b1 ~ U(+-1/sqrt(3584)), w2, b2 ~ U(+-1/16)).

Every workload has gamma+1 target rows per block (row gamma+1 serves the bonus
token) and gamma drafter rows.  Drafted tokens are drawn from the drafter
softmax with the Gumbel-max construction (argmax of logits plus Gumbel noise),
which samples exactly that softmax; ``greedy_drafts=True`` takes the drafter
argmax instead.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch

QWEN_VOCAB = 151_936
HIDDEN = 3584
MLP_HIDDEN = 256


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    gamma: int
    V: int
    dtype: torch.dtype
    seed: int
    kind: str                      # "tiny" | "temp" | "runs"
    sigma: float = 0.5             # target noise scale for "runs"
    sigma_range: tuple | None = None  # per-row target noise range (c4)
    rounds: int = 1
    taus: tuple = (0.9,)
    ells: tuple = ()               # lenience factors as listed per workload (>= 1: paper ell = 1/value)
    topks: tuple = ()
    description: str = ""


WORKLOADS = {
    "tiny": Workload("tiny", 1, 8, 32_000, torch.float32, 0, "tiny", taus=(0.9,),
                     description="B=1, gamma=8, V=32,000 fp32; strict sampling; raw schedule tau=0.9"),
    "c2": Workload("c2", 1, 32, QWEN_VOCAB, torch.bfloat16, 1, "temp", taus=(0.8, 0.9, 0.95),
                   description="B=1, gamma=32, V=151,936 bf16; per-position temperature; strict + residual"),
    "c3": Workload("c3", 16, 32, QWEN_VOCAB, torch.bfloat16, 2, "runs", sigma=0.5, taus=(0.9,),
                   ells=(1.5, 2.0, 4.0), topks=(2, 5, 10),
                   description="B=16, gamma=32, V=151,936 bf16; half peaked in two runs, half flat; "
                               "strict + lenient {1.5,2,4} + top-k {2,5,10}; tau=0.9"),
    "c4": Workload("c4", 64, 64, QWEN_VOCAB, torch.bfloat16, 3, "runs", sigma_range=(0.2, 1.2),
                   taus=(0.50, 0.60, 0.70, 0.80, 0.85, 0.90, 0.93, 0.95, 0.97, 0.98, 0.99, 0.995, 0.998,
                         0.999, 0.9995, 1.0),
                   description="B=64, gamma=64, V=151,936 bf16; per-row target noise U[0.2,1.2]; 16-value tau grid"),
    "c5": Workload("c5", 128, 32, QWEN_VOCAB, torch.bfloat16, 4, "runs", sigma=0.5, rounds=256, taus=(0.9,),
                   description="B=128, gamma=32, V=151,936 bf16, 256 rounds; raw + stand-in MLP schedules"),
}


@dataclass
class Block:
    """One batch of draft blocks: drafter logits [B, gamma, V], target logits
    [B, gamma+1, V], drafted tokens [B, gamma] int32."""
    z_d: torch.Tensor
    z_t: torch.Tensor
    x: torch.Tensor
    peaked: torch.Tensor | None = None   # [B, gamma+1] bool, structure marker (not used by the path)
    extras: dict = field(default_factory=dict)


def _gen(device, *ids) -> torch.Generator:
    """A torch generator seeded from a tuple of small integers."""
    s = 0x9E3779B97F4A7C15
    for i in ids:
        s = (s * 6364136223846793005 + (int(i) & 0xFFFFFFFF) + 1442695040888963407) & 0xFFFFFFFFFFFFFFFF
    g = torch.Generator(device=device)
    g.manual_seed(s & 0x7FFFFFFFFFFFFFFF)
    return g


def _gumbel_draft(z_d: torch.Tensor, gen: torch.Generator, greedy: bool) -> torch.Tensor:
    """Sample one token per row of z_d from its softmax (Gumbel-max), row by row
    to bound temporary memory."""
    B, G, V = z_d.shape
    out = torch.empty(B, G, dtype=torch.int32, device=z_d.device)
    for b in range(B):
        zf = z_d[b].float()
        if greedy:
            out[b] = torch.argmax(zf, dim=-1).to(torch.int32)
            continue
        u = torch.rand(zf.shape, generator=gen, device=z_d.device, dtype=torch.float32)
        u = u.clamp_(min=1e-12, max=1.0 - 1e-7)
        gumbel = -torch.log(-torch.log(u))
        out[b] = torch.argmax(zf + gumbel, dim=-1).to(torch.int32)
    return out


def _rows_tiny(wl: Workload, B, G1, V, device, round_):
    g = _gen(device, wl.seed, round_, 1)
    base = torch.randn(B, G1, V, generator=g, device=device) * 2.0
    t = torch.randint(0, V, (B, G1), generator=g, device=device)
    base.scatter_add_(2, t.unsqueeze(-1), torch.full((B, G1, 1), 6.0, device=device))
    noise = torch.randn(B, G1, V, generator=g, device=device) * 0.5
    return base, base + noise, None


def _rows_temp(wl: Workload, B, G1, V, device, round_):
    g = _gen(device, wl.seed, round_, 2)
    n = torch.randn(B, G1, V, generator=g, device=device)
    t = torch.randint(0, V, (B, G1), generator=g, device=device)
    n.scatter_(2, t.unsqueeze(-1), torch.full((B, G1, 1), -float("inf"), device=device))
    top = n.amax(dim=-1, keepdim=True) + 2.0
    n.scatter_(2, t.unsqueeze(-1), top)
    T = torch.rand(B, G1, 1, generator=g, device=device) * 1.2 + 0.3
    zd = (n / T).to(wl.dtype).float()
    zt = 0.9 * zd + torch.randn(B, G1, V, generator=g, device=device) * 0.7
    return zd, zt, None


def _rows_runs(wl: Workload, B, G1, V, device, round_):
    gamma = G1 - 1
    g = _gen(device, wl.seed, round_, 3)
    half = gamma // 2
    a = torch.randint(0, half + 1, (B,), generator=g, device=device)
    f = torch.randint(1, max(half, 1) + 1, (B,), generator=g, device=device)
    pos = torch.arange(G1, device=device).unsqueeze(0)
    peaked = (pos < a.unsqueeze(1)) | ((pos >= (a + f).unsqueeze(1)) & (pos < (half + f).unsqueeze(1)))
    peaked[:, gamma] = False
    if wl.sigma_range is not None:
        lo, hi = wl.sigma_range
        sig = torch.rand(B, 1, 1, generator=g, device=device) * (hi - lo) + lo
    else:
        sig = torch.full((B, 1, 1), wl.sigma, device=device)
    zd = torch.empty(B, G1, V, device=device)
    zt = torch.empty(B, G1, V, device=device)
    plant = math.log(max(V - 1, 1)) + 0.5 + 8.0
    for b in range(B):   # per batch row keeps fp32 temporaries small
        pk = peaked[b].view(G1, 1)
        base = torch.randn(G1, V, generator=g, device=device)
        rows = torch.where(pk, base, base * 0.5)
        t = torch.randint(0, V, (G1,), generator=g, device=device)
        idx = torch.arange(G1, device=device)
        planted = torch.where(peaked[b], torch.full((G1,), plant, device=device), rows[idx, t])
        rows[idx, t] = planted
        rows = rows.to(wl.dtype).float()
        zd[b] = rows
        zt[b] = rows + torch.randn(G1, V, generator=g, device=device) * sig[b]
    return zd, zt, peaked


_KINDS = {"tiny": _rows_tiny, "temp": _rows_temp, "runs": _rows_runs}


def make_block(wl: Workload | str, device="cpu", round_: int = 0, greedy_drafts: bool = False,
               B: int | None = None, gamma: int | None = None, V: int | None = None,
               dtype: torch.dtype | None = None) -> Block:
    """Draw one batch of blocks for a workload (optionally with overridden sizes)."""
    if isinstance(wl, str):
        wl = WORKLOADS[wl]
    B = wl.B if B is None else B
    gamma = wl.gamma if gamma is None else gamma
    V = wl.V if V is None else V
    dtype = wl.dtype if dtype is None else dtype
    wl = Workload(**{**wl.__dict__, "B": B, "gamma": gamma, "V": V, "dtype": dtype})
    G1 = gamma + 1
    zd, zt, peaked = _KINDS[wl.kind](wl, B, G1, V, device, round_)
    z_d = zd[:, :gamma].to(dtype).clone(memory_format=torch.contiguous_format)
    z_t = zt.to(dtype).clone(memory_format=torch.contiguous_format)
    del zd, zt
    x = _gumbel_draft(z_d, _gen(device, wl.seed, round_, 7), greedy_drafts)
    return Block(z_d=z_d, z_t=z_t, x=x, peaked=peaked)


def make_mlp(device="cpu", seed: int = 4, hidden: int = HIDDEN, width: int = MLP_HIDDEN):
    """Random-init stand-in survival scorer: W1 [width, hidden] bf16 (one row per
    hidden unit, the Linear layout), b1 [width] fp32, w2 [width] bf16, b2 scalar fp32;
    W1, b1 ~ U(+-1/sqrt(hidden)), w2, b2 ~ U(+-1/16)."""
    g = _gen(device, seed, 0xA11CE)
    a = 1.0 / math.sqrt(hidden)
    W1 = ((torch.rand(width, hidden, generator=g, device=device) * 2 - 1) * a).to(torch.bfloat16)
    b1 = (torch.rand(width, generator=g, device=device) * 2 - 1) * a
    w2 = ((torch.rand(width, generator=g, device=device) * 2 - 1) / 16.0).to(torch.bfloat16)
    b2 = (torch.rand(1, generator=g, device=device) * 2 - 1) / 16.0
    return W1.contiguous(), b1.contiguous(), w2.contiguous(), b2.contiguous()


def make_scorer_deep(device="cpu", seed: int = 5, hidden: int = HIDDEN, n_feat: int = 19, width: int = MLP_HIDDEN):
    """Random-init stand-in weights of the learned scorer's shape (App. A.7:
    (hidden + n_feat) -> width -> width -> width -> 1): W1 [width, hidden + width]
    bf16 whose columns past hidden + n_feat are zero (the feature block is padded
    to width columns), W2, W3 [width, width] bf16, w4 [width] bf16, b1..b3 fp32,
    b4 float; U(+-1/sqrt(fan_in)) like a default Linear init."""
    g = _gen(device, seed, 0xDEE9)
    u = lambda *s, a: ((torch.rand(*s, generator=g, device=device) * 2 - 1) * a)   # noqa: E731
    K1 = hidden + n_feat
    W1 = torch.zeros(width, hidden + width, device=device)
    W1[:, :K1] = u(width, K1, a=1.0 / math.sqrt(K1))
    b1 = u(width, a=1.0 / math.sqrt(K1))
    W2, b2 = u(width, width, a=1.0 / math.sqrt(width)), u(width, a=1.0 / math.sqrt(width))
    W3, b3 = u(width, width, a=1.0 / math.sqrt(width)), u(width, a=1.0 / math.sqrt(width))
    w4, b4 = u(width, a=1.0 / math.sqrt(width)), u(1, a=1.0 / math.sqrt(width))
    bf = lambda t: t.to(torch.bfloat16).contiguous()   # noqa: E731
    return (bf(W1), b1.contiguous(), bf(W2), b2.contiguous(), bf(W3), b3.contiguous(), bf(w4), float(b4.item()))


def make_features(rows: int, device="cpu", seed: int = 5, round_: int = 0, n_feat: int = 19, width: int = MLP_HIDDEN):
    """Synthetic scalar features [rows, width] bf16: n_feat standard-normal
    columns, zeros after them (the padded feature block of the deep scorer)."""
    g = _gen(device, seed, round_, 0xFEA7)
    f = torch.zeros(rows, width, device=device)
    f[:, :n_feat] = torch.randn(rows, n_feat, generator=g, device=device)
    return f.to(torch.bfloat16).contiguous()


def make_hidden(rows: int, device="cpu", seed: int = 4, round_: int = 0, hidden: int = HIDDEN):
    g = _gen(device, seed, round_, 0x41DD)
    return torch.randn(rows, hidden, generator=g, device=device).to(torch.bfloat16).contiguous()


def paper_ell(listed: float) -> float:
    """Lenience factors listed >= 1 are read as the paper's ell = 1/listed (App. A.6
    uses ell <= 1 with threshold log ell)."""
    return 1.0 / listed if listed >= 1.0 else listed


def bf16_bits(t: torch.Tensor):
    """numpy uint16 view of a bf16 tensor (what the oracle reads), or float32 numpy."""
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view("uint16")
    return t.float().numpy()
