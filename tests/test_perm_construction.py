"""The parallel construction of the permutation diagnostic's shuffle, as a
plain-Python model of its steps, against Fisher-Yates applied swap by swap
(the definition the oracle follows): for any partner sequence k_a <= a,
bucketing the steps by partner, taking each bucket in index order and
following the "first step above" chains gives the same permutation, whatever
the order of the bucket scatter and of the in-place pointer jumping."""
import random


def _serial(orig, k):
    s = list(orig)
    for a in range(len(s) - 1, 0, -1):
        s[a], s[k[a]] = s[k[a]], s[a]
    return s


def _parallel(orig, k, rng):
    n = len(orig)
    if n <= 1:
        return list(orig)
    end = [0] * n
    for a in range(1, n):
        end[k[a]] += 1
    run = 0
    for t in range(n):           # exclusive prefix: bucket starts
        end[t], run = run, run + end[t]
    bkt = [0] * (n - 1)
    steps = list(range(1, n))
    rng.shuffle(steps)           # the scatter's atomics: any order
    for a in steps:              # starts advance to ends
        bkt[end[k[a]]] = a
        end[k[a]] += 1
    nxt, ptr = [-1] * n, [0] * n
    for t in range(n):
        b0, b1 = (end[t - 1] if t else 0), end[t]
        bkt[b0:b1] = sorted(bkt[b0:b1])
        above = t
        for u in range(b0, b1):
            v = bkt[u]
            nxt[v] = bkt[u + 1] if u + 1 < b1 else -1
            if above == t and v > t:
                above = v
        ptr[t] = above
    span = 1
    while span < n:              # in-place pointer jumping, any interleaving
        order = list(range(n))
        rng.shuffle(order)
        for t in order:
            ptr[t] = ptr[ptr[t]]
        span <<= 1
    return [orig[ptr[0]]] + [orig[ptr[nxt[a]]] if nxt[a] >= 0 else orig[k[a]] for a in range(1, n)]


def test_parallel_construction_equals_serial_fisher_yates():
    rng = random.Random(7)
    for _ in range(600):
        n = rng.choice([1, 2, 3, 4, 5, 8, 17, 64, 65, 200])
        orig = rng.sample(range(10 * n + 5), n)
        if rng.random() < 0.25:    # many steps aimed at few slots
            k = [0] + [rng.choice([0, a, a // 2, min(a, 1)]) for a in range(1, n)]
        else:
            k = [0] + [rng.randint(0, a) for a in range(1, n)]
        assert _parallel(orig, k, rng) == _serial(orig, k), (n, k)
