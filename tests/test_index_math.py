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
