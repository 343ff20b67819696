"""ctypes binding of libsdd.so (include/sdd.h).

Argument marshalling only: every step of the path runs in the library's CUDA
kernels.  PyTorch provides device memory (output tensors, the workspace) and
the current stream.  If the library is missing or fails to load, every entry
point raises; there is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libsdd.so")

SDD_OK = 0
SDD_ERR_DEVICE = 5
SDD_F32 = 0
SDD_BF16 = 1
SIG_RAW, SIG_MARGINAL, SIG_CONDITIONAL, SIG_PERIODIC = 0, 1, 2, 3
DEV_NONFINITE, DEV_BAD_TOKEN, DEV_TIMEOUT = 1, 2, 4
MAX_GAMMA = 128
MAX_GRID = 32

_lib = None

c_i32p = ctypes.POINTER(ctypes.c_int32)
c_f32p = ctypes.POINTER(ctypes.c_float)
c_f64p = ctypes.POINTER(ctypes.c_double)
c_u8p = ctypes.POINTER(ctypes.c_uint8)
c_i64p = ctypes.POINTER(ctypes.c_int64)
VP = ctypes.c_void_p


class BlockArgs(ctypes.Structure):
    """Mirror of sdd_block_args (field order and types as in include/sdd.h)."""
    _fields_ = [
        ("draft_logits", VP), ("target_logits", VP), ("draft_tokens", VP),
        ("dtype", ctypes.c_int32), ("B", ctypes.c_int32), ("gamma", ctypes.c_int32), ("V", ctypes.c_int32),
        ("row_stride", ctypes.c_int64),
        ("signal", ctypes.c_int32), ("n_tau", ctypes.c_int32), ("eta_b", c_f64p), ("eta_c", c_f64p),
        ("period", c_i32p), ("K_skip", ctypes.c_int32), ("reserved1", ctypes.c_int32),
        ("K_min", ctypes.c_int32), ("S_max", ctypes.c_int32),
        ("guard", VP), ("force_strict", VP), ("D_in", VP),
        ("greedy", ctypes.c_int32), ("reserved0", ctypes.c_int32),
        ("seed", ctypes.c_uint64), ("round", ctypes.c_uint64),
        ("n_ell", ctypes.c_int32), ("n_k", ctypes.c_int32), ("ell", c_f64p), ("topk", c_i32p),
        ("q", VP), ("logq", VP), ("maxprob", VP), ("lse", VP), ("entropy", VP), ("argmax", VP),
        ("K_hat", VP), ("K", VP), ("D_out", VP),
        ("L_strict", VP), ("tokens_strict", VP), ("n_strict", VP),
        ("L_lenient", VP), ("tokens_lenient", VP), ("n_lenient", VP),
        ("L_topk", VP), ("tokens_topk", VP), ("n_topk", VP),
        ("commit_tokens", VP), ("commit_n", VP),
        ("agreement", VP),
        ("workspace", VP), ("workspace_bytes", ctypes.c_size_t),
        ("status", VP),
    ]


def load(path: str | None = None):
    """Load libsdd.so (built in-tree by paper_2608_14787_gb300.build)."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or LIB_PATH
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with paper_2608_14787_gb300.build.build()")
    L = ctypes.CDLL(path)
    I = ctypes.c_int
    i64 = ctypes.c_int64
    u64 = ctypes.c_uint64
    L.sdd_version.restype = I
    L.sdd_last_error.restype = ctypes.c_char_p
    L.sdd_workspace_size.argtypes = [I, I, I, ctypes.POINTER(ctypes.c_size_t)]
    L.sdd_confidence.argtypes = [VP, I, I, I, I, i64, VP, VP, VP, VP, VP, VP, VP, VP, ctypes.c_size_t, VP, VP]
    L.sdd_confidence_features.argtypes = [VP, I, I, I, I, i64, VP, VP, VP, VP, VP, VP, VP, VP, VP, VP,
                                          ctypes.c_size_t, VP, VP]
    L.sdd_schedule_prefix.argtypes = [VP, VP, I, I, I, c_f64p, c_f64p, I, I, I, VP, VP, VP, VP, VP, VP, VP, VP]
    L.sdd_schedule_periodic.argtypes = [I, I, c_i32p, I, I, u64, I, I, VP, VP, VP, VP, VP, VP, VP, VP]
    L.sdd_verify_strict.argtypes = [VP, VP, I, I, I, I, i64, VP, VP, I, u64, u64, VP, I, VP, VP, VP, VP,
                                    ctypes.c_size_t, VP, VP]
    L.sdd_verify_lenient.argtypes = [VP, I, I, I, I, i64, VP, c_f64p, I, VP, I, VP, VP, VP, VP, ctypes.c_size_t,
                                     VP, VP]
    L.sdd_verify_topk.argtypes = [VP, I, I, I, I, i64, VP, c_i32p, I, VP, I, VP, VP, VP, VP, ctypes.c_size_t,
                                  VP, VP]
    L.sdd_agreement.argtypes = [VP, VP, I, I, VP, VP]
    L.sdd_commit.argtypes = [VP, VP, VP, VP, I, I, VP, VP, VP]
    L.sdd_uniforms.argtypes = [u64, VP, VP, VP, VP, i64, VP, VP]
    L.sdd_confidence_noalloc.argtypes = [VP, I, I, I, I, i64, VP, VP, VP, VP, VP, VP, VP, VP, VP]
    L.sdd_confidence_noalloc.restype = I
    L.sdd_scorer_features.argtypes = [VP, VP, VP, VP, I, I, i64, VP, VP]
    L.sdd_scorer_features.restype = I
    L.sdd_scorer_workspace_size.argtypes = [I, ctypes.POINTER(ctypes.c_size_t)]
    L.sdd_scorer_workspace_size.restype = I
    L.sdd_survival_mlp.argtypes = [VP, I, I, VP, VP, VP, ctypes.c_float, VP, VP, ctypes.c_size_t, VP, VP]
    L.sdd_survival_mlp.restype = I
    L.sdd_scorer_deep.argtypes = [VP, I, VP, I, VP, VP, VP, VP, VP, VP, VP, ctypes.c_float, VP, VP, VP,
                                  ctypes.c_size_t, VP, VP]
    L.sdd_scorer_deep.restype = I
    L.sdd_permutation_workspace_size.argtypes = [I, I, I, ctypes.POINTER(ctypes.c_size_t)]
    L.sdd_permutation_workspace_size.restype = I
    L.sdd_permutation_diagnostic.argtypes = [VP, VP, I, I, I, ctypes.c_double, ctypes.c_double, I, u64, VP, VP,
                                             ctypes.c_size_t, VP]
    L.sdd_permutation_diagnostic.restype = I
    L.sdd_position_metrics.argtypes = [VP, VP, I, I, I, VP, VP, VP, VP, VP, VP]
    L.sdd_position_metrics.restype = I
    L.sdd_test_wait_hooks.argtypes = [ctypes.c_uint32, I]
    L.sdd_status_from_device.argtypes = [VP, I, ctypes.POINTER(ctypes.c_uint32), VP]
    L.sdd_test_wait_hooks.restype = I
    L.sdd_select_rows.argtypes = [VP, I, VP, VP, VP]
    L.sdd_select_rows.restype = I
    L.sdd_verify_strict_listed.argtypes = [VP, VP, I, I, I, I, i64, VP, VP, I, u64, u64, VP, VP, VP, VP, VP, VP,
                                           ctypes.c_size_t, VP, VP]
    L.sdd_verify_strict_listed.restype = I
    L.sdd_shard_workspace_size.argtypes = [I, ctypes.POINTER(ctypes.c_size_t)]
    L.sdd_shard_workspace_size.restype = I
    L.sdd_shard_partials.argtypes = [ctypes.POINTER(BlockArgs), I, I, VP, VP]
    L.sdd_shard_partials.restype = I
    L.sdd_shard_decide.argtypes = [ctypes.POINTER(BlockArgs), I, I, I, VP, VP, VP]
    L.sdd_shard_decide.restype = I
    L.sdd_shard_draw.argtypes = [ctypes.POINTER(BlockArgs), I, I, I, I, VP, VP]
    L.sdd_shard_draw.restype = I
    for fn in ("sdd_block", "sdd_block_scan", "sdd_block_decide"):
        getattr(L, fn).argtypes = [ctypes.POINTER(BlockArgs), VP]
    L.sdd_block_pipelined.argtypes = [ctypes.POINTER(BlockArgs), ctypes.POINTER(BlockArgs), VP]
    L.sdd_block_pipelined.restype = I
    for fn in ("sdd_workspace_size", "sdd_confidence", "sdd_confidence_features", "sdd_schedule_prefix",
               "sdd_schedule_periodic",
               "sdd_verify_strict",
               "sdd_verify_lenient", "sdd_verify_topk", "sdd_agreement", "sdd_commit", "sdd_uniforms", "sdd_block",
               "sdd_block_scan", "sdd_block_decide"):
        getattr(L, fn).restype = I
    _lib = L
    return L


class SddError(RuntimeError):
    pass


def _check(rc: int, what: str):
    if rc != SDD_OK:
        msg = load().sdd_last_error().decode(errors="replace")
        raise SddError(f"{what} failed (status {rc}): {msg}")


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return SDD_BF16
    if t.dtype == torch.float32:
        return SDD_F32
    raise TypeError(f"logits must be bfloat16 or float32, got {t.dtype}")


def _logits_layout(z: torch.Tensor, npos_name: str):
    """(V, row_stride) of a [B, P, V] tensor whose last dim is contiguous and
    whose rows are evenly spaced."""
    if z.dim() != 3:
        raise ValueError(f"{npos_name} must be [B, P, V]")
    B, P, V = z.shape
    if z.stride(2) != 1 and V > 1:
        raise ValueError(f"{npos_name} must have unit stride over V")
    stride = z.stride(1) if P > 1 or B == 1 else z.stride(0) // max(P, 1)
    if B > 1 and z.stride(0) != stride * P:
        raise ValueError(f"{npos_name} must have evenly spaced rows (stride(0) == stride(1) * P)")
    return V, stride


def workspace_bytes(B: int, gamma: int, V: int) -> int:
    n = ctypes.c_size_t(0)
    _check(load().sdd_workspace_size(B, gamma, V, ctypes.byref(n)), "sdd_workspace_size")
    return int(n.value)


class Workspace:
    """256-byte aligned device scratch for any call with at most B blocks of at
    most gamma positions (its contents need no initialisation)."""

    def __init__(self, B: int, gamma: int, V: int, device=None):
        self.nbytes = workspace_bytes(B, gamma, V)
        buf = torch.zeros(self.nbytes + 256, dtype=torch.uint8, device=device or "cuda")
        off = (-buf.data_ptr()) % 256
        self._buf = buf
        self.tensor = buf[off:off + self.nbytes]

    @property
    def ptr(self):
        return ctypes.c_void_p(self.tensor.data_ptr())


def new_status(device=None) -> torch.Tensor:
    return torch.zeros(1, dtype=torch.int32, device=device or "cuda")


@dataclass
class Confidence:
    q: torch.Tensor
    logq: torch.Tensor
    maxprob: torch.Tensor
    lse: torch.Tensor
    entropy: torch.Tensor
    argmax: torch.Tensor
    margin: torch.Tensor | None = None   # extended features (confidence(..., features=True))
    top5: torch.Tensor | None = None


def confidence_buffers(B: int, gamma: int, device, features: bool = False) -> Confidence:
    """Output tensors for confidence(..., out=): [B, gamma] each (lse fp64, argmax int32)."""
    f32 = lambda: torch.empty(B, gamma, dtype=torch.float32, device=device)  # noqa: E731
    out = Confidence(q=f32(), logq=f32(), maxprob=f32(), lse=torch.empty(B, gamma, dtype=torch.float64, device=device),
                     entropy=f32(), argmax=torch.empty(B, gamma, dtype=torch.int32, device=device))
    if features:
        out.margin, out.top5 = f32(), f32()
    return out


def confidence(z_d: torch.Tensor, x: torch.Tensor, ws: Workspace | None = None, status=None,
               stream=None, features: bool = False, out: Confidence | None = None) -> Confidence:
    """sdd_confidence over drafter logits z_d [B, gamma, V] and drafted tokens x [B, gamma];
    with features=True sdd_confidence_features (also margin and top5 [B, gamma]).
    `out`: tensors from confidence_buffers (filled and returned) instead of new ones."""
    B, gamma = x.shape
    V, stride = _logits_layout(z_d, "z_d")
    dev = z_d.device
    ws = ws or Workspace(B, gamma, V, dev)
    status = new_status(dev) if status is None else status
    if out is None:
        out = confidence_buffers(B, gamma, dev, features)
    elif out.q.shape != (B, gamma) or (features and (out.margin is None or out.top5 is None)):
        raise ValueError("out must come from confidence_buffers(B, gamma, device, features)")
    if features:
        rc = load().sdd_confidence_features(_p(z_d), _dtype_code(z_d), B, gamma, V, stride, _p(x), _p(out.q),
                                            _p(out.logq), _p(out.maxprob), _p(out.lse), _p(out.entropy),
                                            _p(out.argmax), _p(out.margin), _p(out.top5), ws.ptr, ws.nbytes,
                                            _p(status), _stream(stream))
        _check(rc, "sdd_confidence_features")
        return out
    rc = load().sdd_confidence(_p(z_d), _dtype_code(z_d), B, gamma, V, stride, _p(x), _p(out.q), _p(out.logq),
                               _p(out.maxprob), _p(out.lse), _p(out.entropy), _p(out.argmax), ws.ptr, ws.nbytes,
                               _p(status), _stream(stream))
    _check(rc, "sdd_confidence")
    return out


def confidence_noalloc(z_d: torch.Tensor, x: torch.Tensor, status=None, stream=None) -> Confidence:
    """sdd_confidence_noalloc: the same statistics as confidence() with the
    library's fixed scratch instead of a workspace (B * gamma <= 8192)."""
    B, gamma = x.shape
    V, stride = _logits_layout(z_d, "z_d")
    dev = z_d.device
    status = new_status(dev) if status is None else status
    f32 = lambda: torch.empty(B, gamma, dtype=torch.float32, device=dev)  # noqa: E731
    out = Confidence(q=f32(), logq=f32(), maxprob=f32(), lse=torch.empty(B, gamma, dtype=torch.float64, device=dev),
                     entropy=f32(), argmax=torch.empty(B, gamma, dtype=torch.int32, device=dev))
    rc = load().sdd_confidence_noalloc(_p(z_d), _dtype_code(z_d), B, gamma, V, stride, _p(x), _p(out.q),
                                       _p(out.logq), _p(out.maxprob), _p(out.lse), _p(out.entropy), _p(out.argmax),
                                       _p(status), _stream(stream))
    _check(rc, "sdd_confidence_noalloc")
    return out


def _f64_array(vals):
    arr = (ctypes.c_double * len(vals))(*[float(v) for v in vals])
    return arr


def schedule_prefix(q, eta_b, eta_c, *, signal=SIG_RAW, logq=None, K_min=6, S_max=64, guard=None,
                    force_strict=None, D_in=None, status=None, stream=None, out=None):
    """sdd_schedule_prefix; returns (K_hat, K, D_out), each [n_tau, B] int32 (`out`:
    three such tensors to fill instead; D_out must not alias D_in)."""
    B, gamma = q.shape
    n_tau = len(eta_b)
    dev = q.device
    if out is None:
        Kh, K, Do = (torch.empty(n_tau, B, dtype=torch.int32, device=dev) for _ in range(3))
    else:
        Kh, K, Do = out
    eb, ec = _f64_array(eta_b), _f64_array(eta_c)
    rc = load().sdd_schedule_prefix(_p(q), _p(logq), B, gamma, signal, eb, ec, n_tau, K_min, S_max, _p(guard),
                                    _p(force_strict), _p(D_in), _p(Kh), _p(K), _p(Do), _p(status), _stream(stream))
    _check(rc, "sdd_schedule_prefix")
    return Kh, K, Do


def schedule_periodic(B, gamma, periods, *, K_skip=6, round_=0, K_min=6, S_max=64, guard=None, force_strict=None,
                      D_in=None, status=None, stream=None, device="cuda", out=None):
    """sdd_schedule_periodic; returns (K_hat, K, D_out), each [n_p, B] int32 (`out`:
    three such tensors to fill instead; D_out must not alias D_in)."""
    n_p = len(periods)
    if out is None:
        Kh, K, Do = (torch.empty(n_p, B, dtype=torch.int32, device=device) for _ in range(3))
    else:
        Kh, K, Do = out
    per = (ctypes.c_int32 * n_p)(*[int(x) for x in periods])
    rc = load().sdd_schedule_periodic(B, gamma, per, n_p, K_skip, round_, K_min, S_max, _p(guard), _p(force_strict),
                                      _p(D_in), _p(Kh), _p(K), _p(Do), _p(status), _stream(stream))
    _check(rc, "sdd_schedule_periodic")
    return Kh, K, Do


def verify_strict(z_t, x, *, z_d=None, draft=None, greedy=False, seed=0, round_=0, rows=None,
                  ws: Workspace | None = None, status=None, stream=None, out=None):
    """sdd_verify_strict; returns (L [B], tokens [B, gamma+1], n_commit [B])."""
    B, gamma = x.shape
    V, stride = _logits_layout(z_t, "z_t")
    dev = z_t.device
    ws = ws or Workspace(B, gamma, V, dev)
    status = new_status(dev) if status is None else status
    if out is None:
        out = (torch.full((B,), -2, dtype=torch.int32, device=dev),
               torch.full((B, gamma + 1), -2, dtype=torch.int32, device=dev),
               torch.full((B,), -2, dtype=torch.int32, device=dev))
    L, tok, n = out
    n_rows = B if rows is None else rows.numel()
    lse = None if draft is None else draft.lse
    rc = load().sdd_verify_strict(_p(z_t), _p(z_d), _dtype_code(z_t), B, gamma, V, stride, _p(x), _p(lse),
                                  1 if greedy else 0, seed, round_, _p(rows), n_rows, _p(L), _p(tok), _p(n),
                                  ws.ptr, ws.nbytes, _p(status), _stream(stream))
    _check(rc, "sdd_verify_strict")
    return L, tok, n


def select_rows(K, rows=None, n_rows=None, stream=None):
    """sdd_select_rows: (rows [B] int32, n_rows [1] int32), both on the device."""
    B = K.numel()
    rows = torch.empty(B, dtype=torch.int32, device=K.device) if rows is None else rows
    n_rows = torch.empty(1, dtype=torch.int32, device=K.device) if n_rows is None else n_rows
    _check(load().sdd_select_rows(_p(K), B, _p(rows), _p(n_rows), _stream(stream)), "sdd_select_rows")
    return rows, n_rows


def verify_strict_listed(z_t, x, rows, n_rows, *, z_d=None, draft=None, greedy=False, seed=0, round_=0,
                         ws: Workspace | None = None, status=None, stream=None, out=None):
    """sdd_verify_strict_listed: the blocks rows[0..n_rows[0]) with the count on the
    device; returns (L [B], tokens [B, gamma+1], n_commit [B])."""
    B, gamma = x.shape
    V, stride = _logits_layout(z_t, "z_t")
    dev = z_t.device
    ws = ws or Workspace(B, gamma, V, dev)
    status = new_status(dev) if status is None else status
    if out is None:
        out = (torch.full((B,), -2, dtype=torch.int32, device=dev),
               torch.full((B, gamma + 1), -2, dtype=torch.int32, device=dev),
               torch.full((B,), -2, dtype=torch.int32, device=dev))
    L, tok, n = out
    lse = None if draft is None else draft.lse
    rc = load().sdd_verify_strict_listed(_p(z_t), _p(z_d), _dtype_code(z_t), B, gamma, V, stride, _p(x), _p(lse),
                                         1 if greedy else 0, seed, round_, _p(rows), _p(n_rows), _p(L), _p(tok),
                                         _p(n), ws.ptr, ws.nbytes, _p(status), _stream(stream))
    _check(rc, "sdd_verify_strict_listed")
    return L, tok, n


def verify_lenient(z_t, x, ells, *, rows=None, ws=None, status=None, stream=None):
    """sdd_verify_lenient with ell in the paper's convention (0 < ell <= 1)."""
    B, gamma = x.shape
    V, stride = _logits_layout(z_t, "z_t")
    dev = z_t.device
    ws = ws or Workspace(B, gamma, V, dev)
    status = new_status(dev) if status is None else status
    n = len(ells)
    L = torch.full((n, B), -2, dtype=torch.int32, device=dev)
    tok = torch.full((n, B, gamma + 1), -2, dtype=torch.int32, device=dev)
    nc = torch.full((n, B), -2, dtype=torch.int32, device=dev)
    n_rows = B if rows is None else rows.numel()
    rc = load().sdd_verify_lenient(_p(z_t), _dtype_code(z_t), B, gamma, V, stride, _p(x), _f64_array(ells), n,
                                   _p(rows), n_rows, _p(L), _p(tok), _p(nc), ws.ptr, ws.nbytes, _p(status),
                                   _stream(stream))
    _check(rc, "sdd_verify_lenient")
    return L, tok, nc


def verify_topk(z_t, x, ks, *, rows=None, ws=None, status=None, stream=None):
    B, gamma = x.shape
    V, stride = _logits_layout(z_t, "z_t")
    dev = z_t.device
    ws = ws or Workspace(B, gamma, V, dev)
    status = new_status(dev) if status is None else status
    n = len(ks)
    L = torch.full((n, B), -2, dtype=torch.int32, device=dev)
    tok = torch.full((n, B, gamma + 1), -2, dtype=torch.int32, device=dev)
    nc = torch.full((n, B), -2, dtype=torch.int32, device=dev)
    n_rows = B if rows is None else rows.numel()
    karr = (ctypes.c_int32 * n)(*[int(k) for k in ks])
    rc = load().sdd_verify_topk(_p(z_t), _dtype_code(z_t), B, gamma, V, stride, _p(x), karr, n, _p(rows), n_rows,
                                _p(L), _p(tok), _p(nc), ws.ptr, ws.nbytes, _p(status), _stream(stream))
    _check(rc, "sdd_verify_topk")
    return L, tok, nc


def agreement(K, L_strict, acc=None, stream=None):
    n_tau, B = K.shape
    acc = torch.zeros(n_tau, 4, dtype=torch.int64, device=K.device) if acc is None else acc
    _check(load().sdd_agreement(_p(K), _p(L_strict), B, n_tau, _p(acc), _stream(stream)), "sdd_agreement")
    return acc


def commit(K, x, verified_tokens, verified_n, stream=None, out=None):
    """sdd_commit; returns (tokens [B, gamma+1], n [B]) int32 (`out`: two such tensors to fill)."""
    B, gamma = x.shape
    if out is None:
        out_t = torch.empty(B, gamma + 1, dtype=torch.int32, device=x.device)
        out_n = torch.empty(B, dtype=torch.int32, device=x.device)
    else:
        out_t, out_n = out
    _check(load().sdd_commit(_p(K), _p(x), _p(verified_tokens), _p(verified_n), B, gamma, _p(out_t), _p(out_n),
                             _stream(stream)), "sdd_commit")
    return out_t, out_n


MLP_HIDDEN = 256
MLP_KSTEP = 64


def scorer_features(conf, round_: int, *, out=None, stream=None):
    """sdd_scorer_features: the scorer's scalar-feature block [B * gamma, 256] bf16
    from a Confidence computed with features=True (App. A.7's column order)."""
    B, gamma = conf.maxprob.shape
    if conf.margin is None or conf.top5 is None:
        raise ValueError("the confidence must be computed with features=True")
    f = torch.empty(B * gamma, MLP_HIDDEN, dtype=torch.bfloat16, device=conf.maxprob.device) if out is None else out
    _check(load().sdd_scorer_features(_p(conf.maxprob), _p(conf.entropy), _p(conf.margin), _p(conf.top5), B, gamma,
                                      int(round_), _p(f), _stream(stream)), "sdd_scorer_features")
    return f


def scorer_workspace(M, device):
    """A device workspace for the scorers over M positions (sdd_scorer_workspace_size bytes)."""
    nbytes = ctypes.c_size_t(0)
    _check(load().sdd_scorer_workspace_size(int(M), ctypes.byref(nbytes)), "sdd_scorer_workspace_size")
    return torch.empty(max(nbytes.value, 16), dtype=torch.uint8, device=device)


def _scorer_ws(M, device, workspace):
    if workspace is None:
        return scorer_workspace(M, device)
    if workspace.dtype != torch.uint8 or not workspace.is_cuda or not workspace.is_contiguous():
        raise ValueError("workspace must be a contiguous CUDA uint8 tensor (see scorer_workspace)")
    return workspace


def survival_mlp(h, W1, b1, w2, b2: float, *, status=None, stream=None, out=None, workspace=None):
    """sdd_survival_mlp: sigmoid(w2 . GELU(W1 h + b1) + b2) per row of h.
    h bf16 [M, K] (or [B, gamma, K]), W1 bf16 [256, K], b1 fp32 [256], w2 bf16 [256];
    returns fp32 scores shaped like h without its last dimension.  `workspace`:
    from scorer_workspace(M) (allocated per call when omitted)."""
    lead = h.shape[:-1]
    K = h.shape[-1]
    h2 = h.reshape(-1, K)
    for t, name, dt in ((h2, "h", torch.bfloat16), (W1, "W1", torch.bfloat16), (w2, "w2", torch.bfloat16),
                        (b1, "b1", torch.float32)):
        if t.dtype != dt or not t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous CUDA {dt} tensor")
    if W1.shape != (MLP_HIDDEN, K) or b1.shape != (MLP_HIDDEN,) or w2.shape != (MLP_HIDDEN,):
        raise ValueError("W1 must be [256, K], b1 and w2 [256]")
    M = h2.shape[0]
    s = torch.empty(M, dtype=torch.float32, device=h.device) if out is None else out
    ws = _scorer_ws(M, h.device, workspace)
    _check(load().sdd_survival_mlp(_p(h2), M, K, _p(W1), _p(b1), _p(w2), float(b2), _p(s), _p(ws), ws.numel(),
                                   _p(status), _stream(stream)), "sdd_survival_mlp")
    return s.reshape(lead)


def scorer_deep(h, f, W1, b1, W2, b2, W3, b3, w4, b4, *, act=None, status=None, stream=None, out=None,
                workspace=None):
    """sdd_scorer_deep: h [..., Kh] bf16, f [..., 256] bf16 (features, zero padded),
    W1 [256, Kh + 256], W2 / W3 [256, 256], w4 [256] bf16; b1..b3 fp32 [256], b4 float.
    Returns s with h's leading shape.  `workspace`: from scorer_workspace(M)
    (allocated per call when omitted)."""
    lead = h.shape[:-1]
    Kh = h.shape[-1]
    h2 = h.reshape(-1, Kh).contiguous()
    f2 = f.reshape(-1, f.shape[-1]).contiguous()
    M = h2.shape[0]
    if f2.shape != (M, MLP_HIDDEN) or W1.shape != (MLP_HIDDEN, Kh + MLP_HIDDEN):
        raise ValueError("f must be [M, 256] and W1 [256, Kh + 256]")
    for t in (W2, W3):
        if t.shape != (MLP_HIDDEN, MLP_HIDDEN):
            raise ValueError("W2 and W3 must be [256, 256]")
    act = torch.empty(M, MLP_HIDDEN, dtype=torch.bfloat16, device=h.device) if act is None else act
    s = torch.empty(M, dtype=torch.float32, device=h.device) if out is None else out
    ws = _scorer_ws(M, h.device, workspace)
    _check(load().sdd_scorer_deep(_p(h2), Kh, _p(f2), M, _p(W1), _p(b1), _p(W2), _p(b2), _p(W3), _p(b3), _p(w4),
                                  float(b4), _p(act), _p(s), _p(ws), ws.numel(), _p(status), _stream(stream)),
           "sdd_scorer_deep")
    return s.reshape(lead)


def permutation_diagnostic(q, L, *, signal=SIG_RAW, eta_b=0.9, eta_c=0.93, n_rep=100, seed=0, stream=None):
    """sdd_permutation_diagnostic over logged blocks (q [B, gamma] fp32, L [B]
    int32): returns the int64 sums [n_rep + 1] of the feasible prefix lengths
    (the permutations, then the logged order); means are sums / B."""
    B, gamma = q.shape
    nbytes = ctypes.c_size_t(0)
    _check(load().sdd_permutation_workspace_size(B, gamma, n_rep, ctypes.byref(nbytes)),
           "sdd_permutation_workspace_size")
    ws = torch.empty(max(int(nbytes.value), 1), dtype=torch.uint8, device=q.device)
    sums = torch.empty(n_rep + 1, dtype=torch.int64, device=q.device)
    q = q.contiguous()
    L = L.to(torch.int32).contiguous()
    _check(load().sdd_permutation_diagnostic(_p(q), _p(L), B, gamma, signal, float(eta_b), float(eta_c), n_rep, seed,
                                             _p(sums), _p(ws), ws.numel(), _stream(stream)),
           "sdd_permutation_diagnostic")
    return sums


def position_metrics(q, L, *, conditional=False, stream=None):
    """sdd_position_metrics: (bce, bce_base, auroc) fp64 [gamma] and (n_pos, n_neg) int32 [gamma]."""
    B, gamma = q.shape
    dev = q.device
    out = [torch.empty(gamma, dtype=torch.float64, device=dev) for _ in range(3)]
    cnt = [torch.empty(gamma, dtype=torch.int32, device=dev) for _ in range(2)]
    q = q.contiguous()
    L = L.to(torch.int32).contiguous()
    _check(load().sdd_position_metrics(_p(q), _p(L), B, gamma, 1 if conditional else 0, *(_p(t) for t in out),
                                       *(_p(t) for t in cnt), _stream(stream)), "sdd_position_metrics")
    return (*out, *cnt)


def uniforms(seed, j, b, round_, purpose, stream=None):
    """sdd_uniforms: Philox uniforms for device arrays j, b, purpose (int32/uint32) and round (int64)."""
    n = j.numel()
    u = torch.empty(n, dtype=torch.float32, device=j.device)
    _check(load().sdd_uniforms(seed, _p(j), _p(b), _p(round_), _p(purpose), n, _p(u), _stream(stream)),
           "sdd_uniforms")
    return u


def test_wait_hooks(polls: int = 0, drop_copy: bool = False):
    """sdd_test_wait_hooks: the streaming kernel's ring-wait poll limit (0 =
    default) and the dropped-first-copy hook, for later calls of this process."""
    _check(load().sdd_test_wait_hooks(int(polls), 1 if drop_copy else 0), "sdd_test_wait_hooks")


test_wait_hooks.__test__ = False   # a library call, not a test


def status_from_device(status: torch.Tensor, clear: bool = False, stream=None):
    """sdd_status_from_device: the SDD_DEV_* bits of a device status word once
    the stream's calls complete (synchronises the stream); clear=True zeroes
    the word.  Returns (code, bits): code SDD_OK or SDD_ERR_DEVICE; raises
    SddError when the read itself fails."""
    bits = ctypes.c_uint32(0)
    rc = load().sdd_status_from_device(_p(status), 1 if clear else 0, ctypes.byref(bits), _stream(stream))
    if rc not in (SDD_OK, SDD_ERR_DEVICE):
        _check(rc, "sdd_status_from_device")
    return rc, int(bits.value)


class BlockRound:
    """Pre-allocated arguments and outputs of sdd_block for one (B, gamma, V) shape.

    Attributes after a call: q, logq, maxprob, lse, entropy, argmax [B, gamma];
    K_hat, K, D_out [n_tau, B]; L_strict [B], tokens_strict [B, gamma+1],
    n_strict [B]; L_lenient/tokens_lenient/n_lenient [n_ell, ...];
    L_topk/tokens_topk/n_topk [n_k, ...]; commit_tokens, commit_n;
    agreement [n_tau, 4] (accumulated across calls).
    """

    def __init__(self, B, gamma, V, *, dtype=torch.bfloat16, taus=(0.9,), eta_b=None, eta_c=None,
                 signal=SIG_RAW, K_min=6, S_max=64, ells=(), ks=(), greedy=False, periods=None, K_skip=6,
                 device="cuda"):
        """signal=SIG_PERIODIC schedules the periodic baseline: one pair per entry
        of `periods` (skip K_skip tokens once every P rounds); taus are unused."""
        dev = torch.device(device)
        self.B, self.gamma, self.V = B, gamma, V
        self.dtype = dtype
        if signal == SIG_PERIODIC:
            if not periods:
                raise ValueError("SIG_PERIODIC needs periods")
            eta_b = eta_c = [0.0] * len(periods)
        eta_b = list(taus) if eta_b is None else list(eta_b)
        eta_c = list(taus) if eta_c is None else list(eta_c)
        self.n_tau = len(eta_b)
        self.ws = Workspace(B, gamma, V, dev)
        self.status = new_status(dev)
        f32 = lambda *s: torch.zeros(*s, dtype=torch.float32, device=dev)   # noqa: E731
        i32 = lambda *s: torch.zeros(*s, dtype=torch.int32, device=dev)     # noqa: E731
        self.q, self.logq, self.maxprob, self.entropy = (f32(B, gamma) for _ in range(4))
        self.lse = torch.zeros(B, gamma, dtype=torch.float64, device=dev)
        self.argmax = i32(B, gamma)
        self.K_hat, self.K, self.D_out = (i32(self.n_tau, B) for _ in range(3))
        self.D_in = i32(B)
        self.L_strict, self.tokens_strict, self.n_strict = i32(B), i32(B, gamma + 1), i32(B)
        ne, nk = len(ells), len(ks)
        self.L_lenient, self.tokens_lenient, self.n_lenient = i32(max(ne, 1), B), i32(max(ne, 1), B, gamma + 1), \
            i32(max(ne, 1), B)
        self.L_topk, self.tokens_topk, self.n_topk = i32(max(nk, 1), B), i32(max(nk, 1), B, gamma + 1), \
            i32(max(nk, 1), B)
        self.commit_tokens, self.commit_n = i32(B, gamma + 1), i32(B)
        self.agreement = torch.zeros(self.n_tau, 4, dtype=torch.int64, device=dev)
        self._eta_b = _f64_array(eta_b)
        self._eta_c = _f64_array(eta_c)
        self._ell = _f64_array(list(ells) or [1.0])
        self._k = (ctypes.c_int32 * max(nk, 1))(*([int(k) for k in ks] or [1]))
        a = BlockArgs()
        a.dtype = SDD_BF16 if dtype == torch.bfloat16 else SDD_F32
        a.B, a.gamma, a.V = B, gamma, V
        a.signal, a.n_tau = signal, self.n_tau
        a.eta_b = ctypes.cast(self._eta_b, c_f64p)
        a.eta_c = ctypes.cast(self._eta_c, c_f64p)
        a.K_min, a.S_max = K_min, S_max
        if signal == SIG_PERIODIC:
            self._period = (ctypes.c_int32 * len(periods))(*[int(x) for x in periods])
            a.period = ctypes.cast(self._period, c_i32p)
            a.K_skip = int(K_skip)
        a.greedy = 1 if greedy else 0
        a.n_ell, a.n_k = ne, nk
        a.ell = ctypes.cast(self._ell, c_f64p)
        a.topk = ctypes.cast(self._k, c_i32p)
        for name in ("q", "logq", "maxprob", "lse", "entropy", "argmax", "K_hat", "K", "D_out", "L_strict",
                     "tokens_strict", "n_strict", "commit_tokens", "commit_n", "agreement"):
            setattr(a, name, getattr(self, name).data_ptr())
        if ne:
            a.L_lenient, a.tokens_lenient, a.n_lenient = (t.data_ptr() for t in
                                                          (self.L_lenient, self.tokens_lenient, self.n_lenient))
        if nk:
            a.L_topk, a.tokens_topk, a.n_topk = (t.data_ptr() for t in (self.L_topk, self.tokens_topk, self.n_topk))
        a.D_in = self.D_in.data_ptr()
        a.workspace = self.ws.tensor.data_ptr()
        a.workspace_bytes = self.ws.nbytes
        a.status = self.status.data_ptr()
        self.args = a

    def set_inputs(self, z_d, z_t, x, *, seed=0, round_=0, guard=None, force_strict=None):
        V, stride = _logits_layout(z_d, "z_d")
        Vt, stride_t = _logits_layout(z_t, "z_t")
        if (V, stride) != (Vt, stride_t) or V != self.V:
            raise ValueError("z_d and z_t must share V and row stride")
        a = self.args
        a.draft_logits, a.target_logits, a.draft_tokens = z_d.data_ptr(), z_t.data_ptr(), x.data_ptr()
        a.row_stride = stride
        a.seed, a.round = seed, round_
        a.guard = None if guard is None else guard.data_ptr()
        a.force_strict = None if force_strict is None else force_strict.data_ptr()
        self._keep = (z_d, z_t, x, guard, force_strict)

    def run(self, stream=None):
        _check(load().sdd_block(ctypes.byref(self.args), _stream(stream)), "sdd_block")

    def scan(self, stream=None):
        _check(load().sdd_block_scan(ctypes.byref(self.args), _stream(stream)), "sdd_block_scan")

    def decide(self, stream=None):
        _check(load().sdd_block_decide(ctypes.byref(self.args), _stream(stream)), "sdd_block_decide")


def block_pipelined(nxt, prev, stream=None):
    """sdd_block_pipelined: the streaming pass of BlockRound `nxt` and the
    decide work of BlockRound `prev` (streamed by the previous call on this
    stream) in one launch; either may be None (the first and the last call of
    a sequence).  The two rounds must be different BlockRound objects."""
    if nxt is not None and nxt is prev:
        raise ValueError("next and prev must be different BlockRound objects")
    a = None if nxt is None else ctypes.byref(nxt.args)
    b = None if prev is None else ctypes.byref(prev.args)
    _check(load().sdd_block_pipelined(a, b, _stream(stream)), "sdd_block_pipelined")
