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


def _weighted(T0, T1, W, w0, w1):
    """The cost-balanced partition of the streaming kernel (part_start /
    part_owner in csrc/internal.h), emulated with the same magic divisions."""
    T, C = T0 + T1, w0 * T0 + w1 * T1
    fW, fC, f0, f1 = make_fastdiv(W), make_fastdiv(C), make_fastdiv(w0), make_fastdiv(w1)

    def start(w):
        c = fast_div(w * C, fW)
        return fast_div(c + w0 - 1, f0) if c <= w0 * T0 else T0 + fast_div(c - w0 * T0 + w1 - 1, f1)

    def owner(v):
        cost = w0 * v if v < T0 else w0 * T0 + w1 * (v - T0)
        return fast_div((cost + 1) * W - 1, fC)
    return T, start, owner


def test_cost_weighted_partition():
    rng = np.random.default_rng(2)
    cases = [(16 * 32 * 18992, 16 * 33 * 18992, 2432, 10, 9),   # the 16 x 32 block workload, drafter rows first
             (16 * 33 * 18992, 16 * 32 * 18992, 2432, 9, 10),   # target rows first
             (5 * 1001, 0, 37, 1, 1), (3, 4, 3, 10, 9), (8, 9, 8, 10, 9)]
    for _ in range(20):
        T0, T1 = int(rng.integers(1, 50000)), int(rng.integers(1, 50000))
        cases.append((T0, T1, int(rng.integers(1, (T0 + T1) // 2 + 1)), 10, 9))
    for T0, T1, W, w0, w1 in cases:
        if (w0, w1) != (1, 1):
            W = max(1, min(W, (T0 + T1) // 2))   # scan_warps: at least two vectors per warp
        T, start, owner = _weighted(T0, T1, W, w0, w1)
        s = [start(w) for w in range(W + 1)]
        assert s[0] == 0 and s[W] == T
        assert all(s[w + 1] > s[w] for w in range(W)), "empty warp"
        probe = set(rng.integers(0, T, 2000).tolist()) | {x for x in s[:-1]} | {x - 1 for x in s[1:]}
        for v in probe:
            w = owner(int(v))
            assert s[w] <= v < s[w + 1], (T0, T1, W, v, w)
    # balance: each warp's cost is within one vector's cost of C / W
    T0, T1, W = 16 * 32 * 18992, 16 * 33 * 18992, 2432
    T, start, owner = _weighted(T0, T1, W, 10, 9)
    cost = lambda v: 10 * min(v, T0) + 9 * max(v - T0, 0)
    per = [cost(start(w + 1)) - cost(start(w)) for w in range(W)]
    C = cost(T)
    assert max(per) - min(per) <= 2 * 10 and abs(sum(per) - C) == 0
