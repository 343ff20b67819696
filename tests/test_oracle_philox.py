"""Pins for the oracle's Philox4x32-10 and its uniform mapping."""
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def _kat_rows():
    rows = []
    for line in open(GOLDEN):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        f = [int(x, 16) for x in line.split()]
        rows.append((f[0:4], f[4:6], f[6:10]))
    return rows


def test_known_answer_vectors(orc):
    rows = _kat_rows()
    assert len(rows) == 3
    for ctr, key, want in rows:
        got = orc.philox4x32_10(ctr, key)
        assert [int(x) for x in got] == want


def test_uniform_is_odd_multiple_of_2_pow_minus_24(orc):
    u = orc.uniform_many(1234, np.arange(1, 20001), 7, 3, 0)
    k = u * 2.0 ** 24
    assert np.all(k == np.round(k))
    assert np.all(np.mod(k, 2) == 1)
    assert np.all((u > 0) & (u < 1))
    # exactly representable in fp32
    assert np.all(u.astype(np.float32).astype(np.float64) == u)


def test_uniform_matches_word0_mapping(orc):
    # u = ((word0 >> 8) | 1) * 2^-24 for counter (j, b, round_lo, purpose | round_hi << 8), key = seed
    seed, j, b, rnd, purpose = (0x0123456789ABCDEF, 5, 9, (7 << 32) | 11, 2)
    out = orc.philox4x32_10([j, b, rnd & 0xFFFFFFFF, purpose | ((rnd >> 32) << 8)],
                            [seed & 0xFFFFFFFF, seed >> 32])
    want = (((int(out[0]) >> 8) | 1) * 2.0 ** -24)
    assert orc.uniform(seed, j, b, rnd, purpose) == want


def test_uniform_statistics(orc):
    scipy_stats = pytest.importorskip("scipy.stats")
    n = 200_000
    u = orc.uniform_many(99, np.arange(n) % 4096, np.arange(n) // 4096, 5, 0)
    assert abs(u.mean() - 0.5) < 5 * np.sqrt(1 / 12 / n)
    assert abs(u.var() - 1 / 12) < 0.003
    assert scipy_stats.kstest(u, "uniform").pvalue > 1e-4


def test_streams_are_distinct(orc):
    n = 4096
    base = orc.uniform_many(3, np.arange(n), 0, 0, 0)
    for j, b, r, p in [(np.arange(n), 1, 0, 0), (np.arange(n), 0, 1, 0), (np.arange(n), 0, 0, 1)]:
        other = orc.uniform_many(3, j, b, r, p)
        assert np.mean(other == base) < 0.01
    other_seed = orc.uniform_many(4, np.arange(n), 0, 0, 0)
    assert np.mean(other_seed == base) < 0.01
