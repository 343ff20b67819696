"""Planted mistakes in the oracle: each test compiles a copy of the oracle's C
source with one plausible error and checks that the pin meant to catch it
fails, then that the unmodified oracle still passes.  This shows that the
pins are sharp enough to see the mistakes they guard against.

* softmax not normalised (exp(z - m) instead of exp(z - LSE)) -> check_row_probs
* the floor check dropped (rows below -2^23 treated as distributions) -> check_floor
* Sattolo's variant of the shuffle (partner drawn from [0, i)) -> check_fisher_yates
"""
import pytest

from oracle_pins import check_fisher_yates, check_floor, check_row_probs

MUTANTS = {
    "unnormalised_softmax": (
        [("for (int64_t v = 0; v < V; ++v) p[v] = exp(orc_clamp(orc_load(logits, dtype, offset + v)) - lse);",
          "for (int64_t v = 0; v < V; ++v) p[v] = exp(orc_clamp(orc_load(logits, dtype, offset + v)) - m);")],
        check_row_probs),
    "no_floor_check": (
        [("        if (!(m > orc_floor)) bad = 1;\n        int64_t tok",
          "        if (m == -INFINITY) bad = 1;\n        int64_t tok")],
        check_floor),
    "sattolo_shuffle": (
        [("        int k = (int)(((uint64_t)out[0] * (uint64_t)(i + 1)) >> 32);\n        int32_t tmp = perm[i];",
          "        int k = (int)(((uint64_t)out[0] * (uint64_t)(i)) >> 32);\n        int32_t tmp = perm[i];")],
        lambda orc: check_fisher_yates(orc, n_draws=2400)),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(orc, tmp_path, name):
    replacements, check = MUTANTS[name]
    path = orc.build_variant(replacements, str(tmp_path))
    with orc.using_library(path):
        with pytest.raises(AssertionError):
            check(orc)
    check(orc)   # the real oracle is restored and passes
