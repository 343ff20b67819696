"""fp64 CPU oracle for the logits-side path of verifier-skipping speculative
diffusion decoding (arXiv 2608.14787).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The product library never calls it, and it imports nothing from the
product package: the two share no code.

The arithmetic lives in ``sdd_oracle.c`` (plain fp64 loops).  This module only
marshals numpy arrays into it and composes its steps in the paper's order:

* ``row_stats``          -- Sec. 4.2 raw confidence and softmax statistics.
* ``schedule``           -- Sec. 4.1 Eq. 3 and the commit rule (K_min, S_max, D).
* ``verify_strict``      -- Sec. 3.1 strict rule (speculative sampling, greedy).
* ``verify_lenient``     -- App. A.6 Eq. 9.
* ``verify_topk``        -- App. A.6 top-k acceptance.
* ``agreement``          -- Sec. 3.2 Eq. 1 (StrictToken) and Eq. 2 (FullPrefix).
* ``philox4x32_10`` / ``uniform`` -- the counter-based uniforms of the sampling rule.
* ``survival_mlp``       -- the decode-loop workload's stand-in survival scorer
                            sigmoid(w2 . GELU(W1 h + b1) + b2) (App. A.7 form).

Logit arrays are numpy ``float32`` (fp32 logits) or ``uint16`` (the raw bits of
bf16 logits); both are converted exactly to fp64 inside the C code.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "sdd_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")

ORC_F32 = 0
ORC_BF16 = 1

PURPOSE_ACCEPT = 0
PURPOSE_RESID = 1
PURPOSE_BONUS = 2
PURPOSE_DRAFT = 3

SIG_RAW = 0
SIG_MARGINAL = 1
SIG_CONDITIONAL = 2

_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (fp64, no FMA contraction) into oracle/_build."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
                               "-std=c11", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _P(t):
    return ctypes.POINTER(t)


def lib():
    global _lib
    if _lib is None:
        _lib = _bind(build())
    return _lib


def build_variant(replacements, out_dir: str) -> str:
    """Compile a copy of the oracle source with each (old, new) text
    replacement applied (every `old` must occur exactly once) into out_dir.
    Tests use it to plant a mistake in the oracle and check that a pin fails."""
    src = open(_SRC).read()
    for old, new in replacements:
        if src.count(old) != 1:
            raise ValueError(f"replacement target must occur once: {old!r}")
        src = src.replace(old, new)
    os.makedirs(out_dir, exist_ok=True)
    c_path = os.path.join(out_dir, "sdd_oracle_variant.c")
    so_path = os.path.join(out_dir, "liboracle_variant.so")
    with open(c_path, "w") as f:
        f.write(src)
    subprocess.check_call(["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared", "-std=c11",
                           "-o", so_path, c_path, "-lm"])
    return so_path


class using_library:
    """Context manager: route every oracle call through the library at `path`
    (a variant from build_variant) and restore the real one afterwards."""

    def __init__(self, path: str):
        self.path = path

    def __enter__(self):
        global _lib
        self.saved = lib()
        _lib = _bind(self.path)
        return self

    def __exit__(self, *exc):
        global _lib
        _lib = self.saved
        return False


def _bind(path: str):
    L = ctypes.CDLL(path)
    dp, ip32, ip64, up8, up32, up64 = (_P(ctypes.c_double), _P(ctypes.c_int32), _P(ctypes.c_int64),
                                       _P(ctypes.c_uint8), _P(ctypes.c_uint32), _P(ctypes.c_uint64))
    L.orc_philox4x32_10.argtypes = [up32, up32, up32]
    L.orc_philox4x32_10.restype = None
    L.orc_uniform.argtypes = [ctypes.c_uint64, ctypes.c_uint32, ctypes.c_uint32, ctypes.c_uint64, ctypes.c_uint32]
    L.orc_uniform.restype = ctypes.c_double
    L.orc_uniform_many.argtypes = [ctypes.c_int64, ctypes.c_uint64, up32, up32, up64, up32, dp]
    L.orc_uniform_many.restype = None
    L.orc_row_stats.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                                ip32, dp, dp, dp, dp, dp, dp, ip32]
    L.orc_row_stats.restype = None
    L.orc_row_features.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                                   dp, dp]
    L.orc_row_features.restype = None
    L.orc_row_probs.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_int64, dp]
    L.orc_row_probs.restype = None
    L.orc_rank.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64]
    L.orc_rank.restype = ctypes.c_int64
    L.orc_schedule.argtypes = [dp, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_double, ctypes.c_double,
                               ctypes.c_int, ctypes.c_int, up8, up8, ip32, ip32, ip32, ip32, dp]
    L.orc_schedule.restype = None
    L.orc_schedule_periodic.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_uint64,
                                        ctypes.c_int, ctypes.c_int, up8, up8, ip32, ip32, ip32, ip32]
    L.orc_schedule_periodic.restype = None
    L.orc_inverse_cdf.argtypes = [dp, ctypes.c_int64, ctypes.c_double, dp]
    L.orc_inverse_cdf.restype = ctypes.c_int64
    L.orc_verify_strict_sample.argtypes = [dp, dp, ip32, ctypes.c_int, ctypes.c_int64, dp, ctypes.c_double,
                                           ctypes.c_double, dp, ip32, ip32, dp]
    L.orc_verify_strict_sample.restype = None
    L.orc_verify_greedy_family.argtypes = [ctypes.c_int, ctypes.c_double, ctypes.c_int, ip32, ip64, dp, ip32,
                                           ip32, ip32, dp]
    L.orc_verify_greedy_family.restype = None
    L.orc_agreement.argtypes = [ip32, ip32, ctypes.c_int, ip64]
    L.orc_agreement.restype = None
    u16p, f32p, f64p = _P(ctypes.c_uint16), _P(ctypes.c_float), _P(ctypes.c_double)
    L.orc_survival_mlp.argtypes = [u16p, ctypes.c_int, ctypes.c_int, u16p, f32p, u16p, ctypes.c_double,
                                   ctypes.c_int, f64p]
    L.orc_survival_mlp.restype = None
    L.orc_scorer_deep.argtypes = [u16p, ctypes.c_int, ctypes.c_int, u16p, f32p, u16p, f32p, u16p, f32p, u16p,
                                  ctypes.c_double, ctypes.c_int, f64p, f64p, f64p]
    L.orc_scorer_deep.restype = None
    L.orc_permutation_diagnostic.argtypes = [dp, ip32, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_double,
                                             ctypes.c_double, ctypes.c_int, ctypes.c_uint64, ip64, dp, ip32, ip32,
                                             ip32, ip32]
    L.orc_permutation_diagnostic.restype = None
    L.orc_shuffle.argtypes = [ctypes.c_int, ctypes.c_uint64, ctypes.c_int, ctypes.c_int, ip32]
    L.orc_shuffle.restype = None
    return L


def _ptr(a, ct):
    return a.ctypes.data_as(_P(ct))


def _logits_arg(z):
    """Return (array, dtype-code) for a float32 or bf16-bits (uint16) array."""
    z = np.ascontiguousarray(z)
    if z.dtype == np.float32:
        return z, ORC_F32
    if z.dtype == np.uint16:
        return z, ORC_BF16
    raise TypeError(f"oracle logits must be float32 or uint16 (bf16 bits), got {z.dtype}")


# ----------------------------------------------------------------------------
# Philox uniforms
# ----------------------------------------------------------------------------

def philox4x32_10(ctr, key):
    ctr = np.ascontiguousarray(np.asarray(ctr, dtype=np.uint32).reshape(4))
    key = np.ascontiguousarray(np.asarray(key, dtype=np.uint32).reshape(2))
    out = np.zeros(4, dtype=np.uint32)
    lib().orc_philox4x32_10(_ptr(ctr, ctypes.c_uint32), _ptr(key, ctypes.c_uint32), _ptr(out, ctypes.c_uint32))
    return out


def uniform(seed: int, j: int, b: int, round_: int, purpose: int) -> float:
    return float(lib().orc_uniform(seed, j, b, round_, purpose))


def uniform_many(seed: int, j, b, round_, purpose) -> np.ndarray:
    j, b, r, p = np.broadcast_arrays(np.asarray(j, np.uint32), np.asarray(b, np.uint32),
                                     np.asarray(round_, np.uint64), np.asarray(purpose, np.uint32))
    j, b, r, p = (np.ascontiguousarray(x.ravel()) for x in (j, b, r, p))
    out = np.zeros(j.size, dtype=np.float64)
    lib().orc_uniform_many(j.size, seed, _ptr(j, ctypes.c_uint32), _ptr(b, ctypes.c_uint32),
                           _ptr(r, ctypes.c_uint64), _ptr(p, ctypes.c_uint32), _ptr(out, ctypes.c_double))
    return out


# ----------------------------------------------------------------------------
# Row statistics
# ----------------------------------------------------------------------------

@dataclass
class RowStats:
    m: np.ndarray
    lse: np.ndarray
    q: np.ndarray
    logq: np.ndarray
    maxprob: np.ndarray
    entropy: np.ndarray
    argmax: np.ndarray


def row_stats(z, tokens=None) -> RowStats:
    """Softmax statistics of every row of ``z`` ([..., V]); ``tokens`` has shape z.shape[:-1]."""
    z, dt = _logits_arg(z)
    lead = z.shape[:-1]
    V = z.shape[-1]
    n = int(np.prod(lead)) if lead else 1
    outs = [np.zeros(n, dtype=np.float64) for _ in range(6)]
    am = np.zeros(n, dtype=np.int32)
    tok = None
    if tokens is not None:
        tok = np.ascontiguousarray(np.asarray(tokens, dtype=np.int32).reshape(n))
    lib().orc_row_stats(z.ctypes.data, dt, n, V, V, _ptr(tok, ctypes.c_int32) if tok is not None else None,
                        *[_ptr(o, ctypes.c_double) for o in outs], _ptr(am, ctypes.c_int32))
    m, lse, q, logq, mp, H = (o.reshape(lead) for o in outs)
    return RowStats(m=m, lse=lse, q=q, logq=logq, maxprob=mp, entropy=H, argmax=am.reshape(lead))


def row_features(z):
    """Probability margin p_(1) - p_(2) and top-5 mass of every row of ``z``
    ([..., V]), fp64.  Returns (margin, top5) shaped z.shape[:-1]."""
    z, dt = _logits_arg(z)
    lead = z.shape[:-1]
    V = z.shape[-1]
    n = int(np.prod(lead)) if lead else 1
    mg = np.zeros(n, np.float64)
    t5 = np.zeros(n, np.float64)
    lib().orc_row_features(z.ctypes.data, dt, n, V, V, _ptr(mg, ctypes.c_double), _ptr(t5, ctypes.c_double))
    return mg.reshape(lead), t5.reshape(lead)


def row_probs(z_row) -> np.ndarray:
    z, dt = _logits_arg(z_row)
    V = z.shape[-1]
    p = np.zeros(V, dtype=np.float64)
    lib().orc_row_probs(z.ctypes.data, dt, V, 0, _ptr(p, ctypes.c_double))
    return p


def rank(z_row, token: int) -> int:
    z, dt = _logits_arg(z_row)
    return int(lib().orc_rank(z.ctypes.data, dt, z.shape[-1], 0, int(token)))


# ----------------------------------------------------------------------------
# Prefix schedule (Eq. 3)
# ----------------------------------------------------------------------------

def schedule(q, signal, eta_b, eta_c, K_min, S_max, guard=None, force_strict=None, D_in=None):
    """q: [B, gamma] fp64 scores.  Returns (K_hat, K, D_out, margin) for one threshold pair."""
    q = np.ascontiguousarray(np.asarray(q, dtype=np.float64))
    B, gamma = q.shape
    g = None if guard is None else np.ascontiguousarray(np.asarray(guard, dtype=np.uint8).reshape(B, gamma))
    f = None if force_strict is None else np.ascontiguousarray(np.asarray(force_strict, dtype=np.uint8).reshape(B))
    D = np.zeros(B, np.int32) if D_in is None else np.ascontiguousarray(np.asarray(D_in, dtype=np.int32).reshape(B))
    Kh = np.zeros(B, np.int32)
    K = np.zeros(B, np.int32)
    Do = np.zeros(B, np.int32)
    mg = np.zeros(B, np.float64)
    lib().orc_schedule(_ptr(q, ctypes.c_double), B, gamma, int(signal), float(eta_b), float(eta_c), int(K_min),
                       int(S_max), _ptr(g, ctypes.c_uint8) if g is not None else None,
                       _ptr(f, ctypes.c_uint8) if f is not None else None, _ptr(D, ctypes.c_int32),
                       _ptr(Kh, ctypes.c_int32), _ptr(K, ctypes.c_int32), _ptr(Do, ctypes.c_int32),
                       _ptr(mg, ctypes.c_double))
    return Kh, K, Do, mg


def schedule_periodic(B, gamma, P, K_skip, round_, K_min, S_max, guard=None, force_strict=None, D_in=None):
    """Periodic skipping baseline for one period P.  Returns (K_hat, K, D_out)."""
    g = None if guard is None else np.ascontiguousarray(np.asarray(guard, dtype=np.uint8).reshape(B, gamma))
    f = None if force_strict is None else np.ascontiguousarray(np.asarray(force_strict, dtype=np.uint8).reshape(B))
    D = np.zeros(B, np.int32) if D_in is None else np.ascontiguousarray(np.asarray(D_in, dtype=np.int32).reshape(B))
    Kh = np.zeros(B, np.int32)
    K = np.zeros(B, np.int32)
    Do = np.zeros(B, np.int32)
    lib().orc_schedule_periodic(B, gamma, int(P), int(K_skip), int(round_), int(K_min), int(S_max),
                                _ptr(g, ctypes.c_uint8) if g is not None else None,
                                _ptr(f, ctypes.c_uint8) if f is not None else None, _ptr(D, ctypes.c_int32),
                                _ptr(Kh, ctypes.c_int32), _ptr(K, ctypes.c_int32), _ptr(Do, ctypes.c_int32))
    return Kh, K, Do


# ----------------------------------------------------------------------------
# Inverse CDF and acceptance rules
# ----------------------------------------------------------------------------

def inverse_cdf(w, u):
    w = np.ascontiguousarray(np.asarray(w, dtype=np.float64))
    mg = ctypes.c_double(0.0)
    v = lib().orc_inverse_cdf(_ptr(w, ctypes.c_double), w.size, float(u), ctypes.byref(mg))
    return int(v), float(mg.value)


def strict_sample_probs(pt, pd, x, u_acc, u_res, u_bonus):
    """Speculative-sampling rule on explicit probabilities and uniforms (one block)."""
    pt = np.ascontiguousarray(np.asarray(pt, dtype=np.float64))
    pd = np.ascontiguousarray(np.asarray(pd, dtype=np.float64))
    gamma, V = pd.shape
    assert pt.shape == (gamma + 1, V)
    x = np.ascontiguousarray(np.asarray(x, dtype=np.int32).reshape(gamma))
    ua = np.ascontiguousarray(np.asarray(u_acc, dtype=np.float64).reshape(gamma))
    w = np.zeros(V, np.float64)
    L = ctypes.c_int32(0)
    tokens = np.zeros(gamma + 1, np.int32)
    mg = ctypes.c_double(0.0)
    lib().orc_verify_strict_sample(_ptr(pt, ctypes.c_double), _ptr(pd, ctypes.c_double), _ptr(x, ctypes.c_int32),
                                   gamma, V, _ptr(ua, ctypes.c_double), float(u_res), float(u_bonus),
                                   _ptr(w, ctypes.c_double), ctypes.byref(L), _ptr(tokens, ctypes.c_int32),
                                   ctypes.byref(mg))
    return int(L.value), tokens, float(mg.value)


def _greedy_family(mode, param, x, rank_, gap, target_argmax):
    gamma = len(x)
    x = np.ascontiguousarray(np.asarray(x, dtype=np.int32))
    rk = np.ascontiguousarray(np.asarray(rank_, dtype=np.int64))
    gp = np.ascontiguousarray(np.asarray(gap, dtype=np.float64))
    ta = np.ascontiguousarray(np.asarray(target_argmax, dtype=np.int32))
    assert ta.size == gamma + 1
    L = ctypes.c_int32(0)
    tokens = np.zeros(gamma + 1, np.int32)
    mg = ctypes.c_double(0.0)
    lib().orc_verify_greedy_family(int(mode), float(param), gamma, _ptr(x, ctypes.c_int32), _ptr(rk, ctypes.c_int64),
                                   _ptr(gp, ctypes.c_double), _ptr(ta, ctypes.c_int32), ctypes.byref(L),
                                   _ptr(tokens, ctypes.c_int32), ctypes.byref(mg))
    return int(L.value), tokens, float(mg.value)


@dataclass
class TargetFacts:
    """What the greedy-family rules read from the target rows of one block."""
    rank: np.ndarray     # [gamma] int64
    gap: np.ndarray      # [gamma] fp64, z(x_j) - max z
    argmax: np.ndarray   # [gamma+1] int32


def target_facts(zt_block, x) -> TargetFacts:
    """zt_block: [gamma+1, V] target logits of one block; x: [gamma] drafted tokens."""
    zt, _ = _logits_arg(zt_block)
    gamma = zt.shape[0] - 1
    st = row_stats(zt)
    rk = np.zeros(gamma, np.int64)
    gap = np.zeros(gamma, np.float64)
    for j in range(gamma):
        rk[j] = rank(zt[j], int(x[j]))
        zf = _to_f64(zt[j])
        gap[j] = zf[int(x[j])] - st.m[j]
    return TargetFacts(rank=rk, gap=gap, argmax=st.argmax.astype(np.int32))


def _to_f64(z):
    if z.dtype == np.uint16:
        return (z.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return z.astype(np.float64)


def verify_greedy(facts: TargetFacts, x):
    return _greedy_family(0, 0.0, x, facts.rank, facts.gap, facts.argmax)


def verify_lenient(facts: TargetFacts, x, ell: float):
    """ell in the paper's convention (0 < ell <= 1; accept iff gap >= log ell)."""
    return _greedy_family(1, float(ell), x, facts.rank, facts.gap, facts.argmax)


def verify_topk(facts: TargetFacts, x, k: int):
    return _greedy_family(2, float(k), x, facts.rank, facts.gap, facts.argmax)


def verify_strict(zt_block, zd_block, x, seed: int, b: int, round_: int):
    """Sampling form of Strict SDD for one block with the Philox uniforms of row b.

    zt_block: [gamma+1, V] target logits, zd_block: [gamma, V] drafter logits.
    Uniforms: u_j = U(seed, j, b, round, ACCEPT) for j = 1..gamma, the residual
    draw U(seed, L+1, b, round, RESID), the bonus draw U(seed, gamma+1, b, round, BONUS).
    """
    zt, _ = _logits_arg(zt_block)
    zd, _ = _logits_arg(zd_block)
    gamma = zd.shape[0]
    pt = np.stack([row_probs(zt[j]) for j in range(gamma + 1)])
    pd = np.stack([row_probs(zd[j]) for j in range(gamma)])
    u_acc = np.array([uniform(seed, j + 1, b, round_, PURPOSE_ACCEPT) for j in range(gamma)])
    # The residual draw's counter depends on L; compute L first with a placeholder, then redo.
    L, _, _ = strict_sample_probs(pt, pd, x, u_acc, 0.5, 0.5)
    u_res = uniform(seed, L + 1, b, round_, PURPOSE_RESID)
    u_bonus = uniform(seed, gamma + 1, b, round_, PURPOSE_BONUS)
    return strict_sample_probs(pt, pd, x, u_acc, u_res, u_bonus)


def survival_mlp(h_bits, W1_bits, b1, w2_bits, b2: float) -> np.ndarray:
    """fp64 sigmoid(w2 . GELU(W1 h + b1) + b2) per row of h.  h_bits [M, K] and
    W1_bits [N, K] / w2_bits [N] are the raw bits of bf16 arrays (uint16), b1 fp32 [N]."""
    h = np.ascontiguousarray(np.asarray(h_bits, dtype=np.uint16))
    W1 = np.ascontiguousarray(np.asarray(W1_bits, dtype=np.uint16))
    w2 = np.ascontiguousarray(np.asarray(w2_bits, dtype=np.uint16))
    b1 = np.ascontiguousarray(np.asarray(b1, dtype=np.float32))
    M, K = h.shape
    N = W1.shape[0]
    if W1.shape != (N, K) or w2.shape != (N,) or b1.shape != (N,):
        raise ValueError("shape mismatch")
    out = np.zeros(M, np.float64)
    lib().orc_survival_mlp(_ptr(h, ctypes.c_uint16), M, K, _ptr(W1, ctypes.c_uint16), _ptr(b1, ctypes.c_float),
                           _ptr(w2, ctypes.c_uint16), float(b2), N, _ptr(out, ctypes.c_double))
    return out


def scorer_deep(x_bits, W1_bits, b1, W2_bits, b2, W3_bits, b3, w4_bits, b4: float) -> np.ndarray:
    """fp64 sigmoid(w4 . GELU(W3 a2 + b3) + b4), a2 = GELU(W2 a1 + b2),
    a1 = GELU(W1 x + b1) per row of x, every activation in fp64.  x_bits [M, K], W1 [N, K], W2 and W3
    [N, N], w4 [N]: raw bf16 bits (uint16); biases fp32 [N]."""
    u16 = lambda a: np.ascontiguousarray(np.asarray(a, dtype=np.uint16))   # noqa: E731
    f32 = lambda a: np.ascontiguousarray(np.asarray(a, dtype=np.float32))  # noqa: E731
    x, W1, W2, W3, w4 = u16(x_bits), u16(W1_bits), u16(W2_bits), u16(W3_bits), u16(w4_bits)
    b1, b2, b3 = f32(b1), f32(b2), f32(b3)
    M, K = x.shape
    N = W1.shape[0]
    if W1.shape != (N, K) or W2.shape != (N, N) or W3.shape != (N, N) or w4.shape != (N,) or \
            b1.shape != (N,) or b2.shape != (N,) or b3.shape != (N,):
        raise ValueError("shape mismatch")
    out = np.zeros(M, np.float64)
    s1, s2 = np.zeros(N, np.float64), np.zeros(N, np.float64)
    u16p, f32p, dp = _P(ctypes.c_uint16), _P(ctypes.c_float), _P(ctypes.c_double)
    lib().orc_scorer_deep(x.ctypes.data_as(u16p), M, K, W1.ctypes.data_as(u16p), b1.ctypes.data_as(f32p),
                          W2.ctypes.data_as(u16p), b2.ctypes.data_as(f32p), W3.ctypes.data_as(u16p),
                          b3.ctypes.data_as(f32p), w4.ctypes.data_as(u16p), float(b4), N, out.ctypes.data_as(dp),
                          s1.ctypes.data_as(dp), s2.ctypes.data_as(dp))
    return out


def permutation_diagnostic(q, L, signal, eta_b, eta_c, n_rep, seed):
    """Sums of the feasible prefix lengths: [n_rep] under the permutations, then
    the logged order (length n_rep + 1)."""
    q = np.ascontiguousarray(np.asarray(q, dtype=np.float64))
    B, gamma = q.shape
    L = np.ascontiguousarray(np.asarray(L, dtype=np.int32).reshape(B))
    sums = np.zeros(n_rep + 1, np.int64)
    qp = np.zeros_like(q)
    lst, kh, k, d = (np.zeros(max(B, 1), np.int32) for _ in range(4))
    i32 = lambda a: _ptr(a, ctypes.c_int32)   # noqa: E731
    lib().orc_permutation_diagnostic(_ptr(q, ctypes.c_double), i32(L), B, gamma, int(signal), float(eta_b),
                                     float(eta_c), int(n_rep), ctypes.c_uint64(int(seed)), _ptr(sums, ctypes.c_int64),
                                     _ptr(qp, ctypes.c_double), i32(lst), i32(kh), i32(k), i32(d))
    return sums


def shuffle(n: int, seed: int, j0: int, r: int) -> np.ndarray:
    """The diagnostic's Fisher-Yates permutation of 0..n-1 for repetition r
    and 0-based position j0."""
    perm = np.zeros(max(n, 1), np.int32)
    lib().orc_shuffle(int(n), ctypes.c_uint64(int(seed)), int(j0), int(r), _ptr(perm, ctypes.c_int32))
    return perm[:n]


def position_metrics(q, L, conditional: bool):
    """Positionwise BCE, position-only baseline BCE and AUROC (fp64, plain
    loops over the definitions): labels y = 1{L >= j}, j 1-based; blocks with
    L >= j - 1 only when conditional.  Returns (bce, bce_base, auroc, n_pos, n_neg)."""
    q = np.asarray(q, dtype=np.float64)
    L = np.asarray(L, dtype=np.int64)
    B, gamma = q.shape
    out = [np.full(gamma, np.nan) for _ in range(3)]
    npos, nneg = np.zeros(gamma, np.int64), np.zeros(gamma, np.int64)
    for j in range(gamma):
        idx = [b for b in range(B) if not conditional or L[b] >= j]
        if not idx:
            continue
        y = [1 if L[b] >= j + 1 else 0 for b in idx]
        qc = [min(max(q[b, j], 1e-7), 1.0 - 1e-7) for b in idx]
        n = len(idx)
        out[0][j] = -sum(math.log(c) if t else math.log1p(-c) for c, t in zip(qc, y)) / n
        p = sum(y) / n
        out[1][j] = -(p * math.log(p) + (1 - p) * math.log1p(-p)) if 0.0 < p < 1.0 else 0.0
        pos = [q[b, j] for b, t in zip(idx, y) if t]
        neg = [q[b, j] for b, t in zip(idx, y) if not t]
        npos[j], nneg[j] = len(pos), len(neg)
        if pos and neg:
            gt = sum(1 for a in pos for c in neg if a > c)
            eq = sum(1 for a in pos for c in neg if a == c)
            out[2][j] = (gt + 0.5 * eq) / (len(pos) * len(neg))
    return out[0], out[1], out[2], npos, nneg


def agreement(K, L):
    K = np.ascontiguousarray(np.asarray(K, dtype=np.int32))
    L = np.ascontiguousarray(np.asarray(L, dtype=np.int32))
    acc = np.zeros(4, np.int64)
    lib().orc_agreement(_ptr(K, ctypes.c_int32), _ptr(L, ctypes.c_int32), K.size, _ptr(acc, ctypes.c_int64))
    return acc
