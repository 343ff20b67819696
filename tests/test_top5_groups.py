"""The selection behind the streaming kernel's extended features, as a
plain-Python model of its steps, against the brute-force five largest entries
of a row piece: each lane keeps its five largest tile maxima (a tile maximum
enters only if it beats the lane's fifth, as in the kernel); the warp merges
the lanes' lists into the five largest (lane, tile) groups; the five largest
entries of those groups are the piece's five largest, with multiplicity --
also with heavy ties, which quantised (bf16-like) logits produce."""
import random

LANES, VPL, EPV = 32, 8, 8   # lanes of a warp, vectors per lane per tile, entries per vector


def _piece(rng, tiles, levels):
    # piece[t][lane] = the 64 entries of that lane's 8 vectors in tile t
    return [[[rng.choice(levels) for _ in range(VPL * EPV)] for _ in range(LANES)] for _ in range(tiles)]


def _kernel_model(piece):
    lists = [[] for _ in range(LANES)]            # per lane: [(max, tile)] descending, at most 5
    for t, tile in enumerate(piece):
        for lane in range(LANES):
            m = max(tile[lane])
            lst = lists[lane]
            if len(lst) == 5 and m <= lst[4][0]:   # the kernel's early return
                continue
            k = 0
            while k < len(lst) and lst[k][0] >= m:   # strictly greater moves down (ties keep order)
                k += 1
            lst.insert(k, (m, t))
            del lst[5:]
    groups = []                                   # five rounds: the first lane holding the largest head
    for _ in range(5):
        heads = [(lists[l][0][0] if lists[l] else float("-inf"), l) for l in range(LANES)]
        best = max(h for h, _ in heads)
        owner = min(l for h, l in heads if h == best)
        if lists[owner]:
            groups.append((owner, lists[owner].pop(0)[1]))
    cand = [e for lane, t in groups for e in piece[t][lane]]
    return sorted(cand, reverse=True)[:5]


def test_top5_from_five_groups_matches_brute_force():
    rng = random.Random(3)
    for trial in range(300):
        tiles = rng.choice([1, 2, 3, 7, 16])
        if trial % 3 == 0:
            levels = [x / 8 for x in range(-16, 24)]          # coarse: many ties
        elif trial % 3 == 1:
            levels = [0.0, 1.0, 2.0]                          # extreme ties
        else:
            levels = [rng.gauss(0, 1) for _ in range(4000)]   # nearly distinct
        piece = _piece(rng, tiles, levels)
        everything = sorted((e for tile in piece for lane in tile for e in lane), reverse=True)[:5]
        assert _kernel_model(piece) == everything, (trial, tiles)
