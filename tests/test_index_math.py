"""The kernels' division by launch constants (FastDiv in csrc/internal.h):
floor(n / d) = umulhi(n, M) >> s with s = floor(log2 d), M = ceil(2^(64+s) / d)
(a power of two is a shift).  Emulated here with Python integers, the same
construction must equal exact integer division for every n < 2^53 -- edge
values, random values, and the index ranges of the 64 x 64 workload."""
import numpy as np


def make_fastdiv(d: int):
    s = d.bit_length() - 1                     # floor(log2 d)
    if d & (d - 1) == 0:
        return 0, s, True
    return -(-(1 << (64 + s)) // d), s, False   # ceil(2^(64+s) / d)


def fast_div(n: int, f) -> int:
    M, s, pow2 = f
    if pow2:
        return n >> s
    assert M < (1 << 64)
    return ((n * M) >> 64) >> s                  # umulhi(n, M) >> s


def test_fastdiv_edges_and_random():
    rng = np.random.default_rng(0)
    ds = [1, 2, 3, 7, 33, 129, 2432, 4096, 18992, 2**24 + 1, 19751680, 2**31 - 1, 2**40 - 3, 2**52 + 7]
    ns = [0, 1, 2**24 + 1, 2**31 - 1, 2**40, 2**53 - 1]
    for d in ds:
        f = make_fastdiv(d)
        for n in ns + [d - 1, d, d + 1, 2**53 - 1 - (2**53 - 1) % d, 2**53 - 2 - (2**53 - 1) % d]:
            if 0 <= n < 2**53:
                assert fast_div(n, f) == n // d, (n, d)
    for _ in range(50000):
        d = int(rng.integers(1, 2**int(rng.integers(1, 53))))
        n = int(rng.integers(0, 2**53))
        assert fast_div(n, make_fastdiv(d)) == n // d, (n, d)


def test_partition_of_the_64x64_workload():
    # rows = 64 blocks x (2 * 64 + 1), 18992 vectors per row, 2432 warps
    T, W, RV = 64 * 129 * 18992, 2432, 18992
    fT, fW, fRV, fN = make_fastdiv(T), make_fastdiv(W), make_fastdiv(RV), make_fastdiv(65)
    rng = np.random.default_rng(1)
    for w in range(W + 1):
        assert fast_div(w * T, fW) == w * T // W
    for v in rng.integers(0, T, 20000):
        v = int(v)
        assert fast_div((v + 1) * W - 1, fT) == ((v + 1) * W - 1) // T
        assert fast_div(v, fRV) == v // RV
        assert fast_div(v % (64 * 129), fN) == (v % (64 * 129)) // 65


def _weighted(T0, T1, W, w0, w1, RV=None, R=0):
    """The cost-balanced partition of the streaming kernel (part_start /
    part_owner in csrc/internal.h), emulated with the same magic divisions:
    rows of RV vectors (group 0: T0 vectors, then group 1: T1), a group-g
    vector costing w_g and a row's first vector R more."""
    RV = RV or 1
    rows0, rows1 = T0 // RV, T1 // RV
    assert rows0 * RV == T0 and rows1 * RV == T1
    P = (w0 * RV + R, w1 * RV + R)
    wt = (w0, w1)
    T, C = T0 + T1, rows0 * P[0] + rows1 * P[1]
    fW, fC, fRV = make_fastdiv(W), make_fastdiv(C), make_fastdiv(RV)
    fWt = (make_fastdiv(w0), make_fastdiv(w1))
    fP = (make_fastdiv(P[0]), make_fastdiv(P[1]))
    c0 = rows0 * P[0]

    def start(w):
        c = fast_div(w * C, fW)
        g = 0 if c <= c0 else 1
        cg = c - c0 if g else c
        r = fast_div(cg, fP[g])
        rem = cg - r * P[g]
        k = 0
        if rem > 0:
            k = 1 if rem <= R else fast_div(rem - R + wt[g] - 1, fWt[g])
        return (T0 if g else 0) + r * RV + k

    def owner(v):
        g = 0 if v < T0 else 1
        u = v - T0 if g else v
        r = fast_div(u, fRV)
        k = u - r * RV
        cost = (c0 if g else 0) + r * P[g] + (R + k * wt[g] if k > 0 else 0)
        return fast_div((cost + 1) * W - 1, fC)

    def cost(v):   # plain definition: the costs of the vectors before v
        tot = 0
        for g, (lo, hi) in enumerate(((0, T0), (T0, T))):
            for x in range(lo, min(v, hi)):
                tot += wt[g] + (R if (x - lo) % RV == 0 else 0)
        return tot
    return T, start, owner, cost, C


def test_cost_weighted_partition():
    rng = np.random.default_rng(2)
    cases = [(16 * 32 * 18992, 16 * 33 * 18992, 2432, 10, 9, 18992, 0),   # the 16 x 32 block workload
             (16 * 33 * 18992, 16 * 32 * 18992, 2432, 9, 10, 18992, 0),   # target rows first
             (5 * 1001, 0, 37, 1, 1, 1001, 0), (3, 4, 3, 10, 9, 1, 0), (8, 9, 8, 10, 9, 1, 0),
             (16 * 32 * 18992, 16 * 33 * 18992, 2432, 10, 9, 18992, 4000)]   # with a row-start cost
    for _ in range(20):
        T0, T1 = int(rng.integers(1, 50000)), int(rng.integers(1, 50000))
        cases.append((T0, T1, int(rng.integers(1, (T0 + T1) // 2 + 1)), 10, 9, 1, 0))
    for _ in range(20):
        # rows with a row-start cost inside the bound that set_divisors keeps
        # (wmin RV + R >= 16 (R + 2 wmax)); W at most 16 per row
        RV = int(rng.integers(32, 3000))
        rows0, rows1 = int(rng.integers(1, 12)), int(rng.integers(0, 12))
        R = int(rng.integers(0, max(1, (9 * RV - 16 * 20) // 15)))
        W = int(rng.integers(1, 16 * (rows0 + rows1) + 1))
        cases.append((rows0 * RV, rows1 * RV, W, 10, 9, RV, R))
    for T0, T1, W, w0, w1, RV, R in cases:
        if (w0, w1) != (1, 1) and R == 0:
            W = max(1, min(W, (T0 + T1) // 2))   # scan_warps: at least two vectors per warp
        T, start, owner, _, _ = _weighted(T0, T1, W, w0, w1, RV, R)
        s = [start(w) for w in range(W + 1)]
        assert s[0] == 0 and s[W] == T
        assert all(s[w + 1] > s[w] for w in range(W)), ("empty warp", T0, T1, W, RV, R)
        probe = set(rng.integers(0, T, 2000).tolist()) | {x for x in s[:-1]} | {x - 1 for x in s[1:]}
        for v in probe:
            w = owner(int(v))
            assert s[w] <= v < s[w + 1], (T0, T1, W, v, w)
    # balance: each warp's cost is within one vector's cost of C / W
    T0, T1, W = 16 * 32 * 18992, 16 * 33 * 18992, 2432
    for R in (0, 4000):
        T, start, owner, _, C = _weighted(T0, T1, W, 10, 9, 18992, R)
        cost = lambda v: (10 * min(v, T0) + 9 * max(v - T0, 0)
                          + R * (-(-min(v, T0) // 18992) + -(-max(v - T0, 0) // 18992)))
        per = [cost(start(w + 1)) - cost(start(w)) for w in range(W)]
        assert max(per) - min(per) <= 2 * (10 + R) and sum(per) == C


def test_partition_cost_against_its_definition():
    """cost(v) in part_owner equals the plain sum of the vectors' costs."""
    rng = np.random.default_rng(5)
    for _ in range(30):
        RV = int(rng.integers(1, 40))
        rows0, rows1 = int(rng.integers(0, 5)), int(rng.integers(0, 5))
        if rows0 + rows1 == 0:
            continue
        R = int(rng.integers(0, 50))
        T0, T1 = rows0 * RV, rows1 * RV
        T, start, owner, cost, C = _weighted(T0, T1, 1, 10, 9, RV, R)
        assert cost(T) == C
        for w_ in (2, 3, 7):
            T, start, owner, cost, C = _weighted(T0, T1, w_, 10, 9, RV, R)
            for v in range(T):
                # the owner of v: the warp whose cost interval holds cost(v)
                w = owner(v)
                assert (w * C) // w_ <= cost(v) < ((w + 1) * C) // w_, (RV, R, v)


def _scan_warps(W_max, T, rows, per_row=16):
    """scan_warps of csrc/internal.h."""
    w = min(W_max, T // 2, rows * per_row)
    return max(w, 1)


def test_pipelined_pass_partitions():
    """The pipelined round streams on fourteen (or, after a small round,
    twelve) warps per CTA with drafter : target weights 21 : 18 and a
    row-start cost of 400 drafter vectors: every warp's range is non-empty
    and the owner of every vector agrees with the starts (the decide merges
    the partials of warps first_owner .. last_owner of each row)."""
    rng = np.random.default_rng(12)
    RV = 18992                                      # 151,936 bf16 entries per row
    cases = []
    for B, gamma, wpc in ((16, 32, 14), (24, 32, 14), (1, 32, 12), (5, 8, 12), (16, 64, 14)):
        rows0, rows1 = B * gamma, B * (gamma + 1)
        T = (rows0 + rows1) * RV
        W = _scan_warps(152 * wpc, T, rows0 + rows1)
        R = 400 * 21
        if RV < 32 or 18 * RV + R < 16 * (R + 2 * 21):   # set_divisors keeps no row-start cost
            R = 0
        cases.append((rows0 * RV, rows1 * RV, W, RV, R))
    cases.append((1 * 8 * 2000, 1 * 9 * 2000, _scan_warps(152 * 12, 17 * 2000, 17), 2000, 0))
    for T0, T1, W, rv, R in cases:
        T, start, owner, _, C = _weighted(T0, T1, W, 21, 18, rv, R)
        s = [start(w) for w in range(W + 1)]
        assert s[0] == 0 and s[W] == T
        assert all(s[w + 1] > s[w] for w in range(W)), ("empty warp", T0, T1, W, rv, R)
        probe = set(rng.integers(0, T, 3000).tolist()) | set(s[:-1]) | {x - 1 for x in s[1:]}
        for v in probe:
            w = owner(int(v))
            assert s[w] <= v < s[w + 1], (T0, T1, W, v, w)
