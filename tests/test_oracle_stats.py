"""Pins for the oracle's per-row softmax statistics (Sec. 4.2 raw confidence)
and its rank definition (App. A.6 top-k membership)."""
import math

import numpy as np
import pytest
import torch


def _bf16_bits(x: np.ndarray) -> np.ndarray:
    return torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def _bf16_vals(bits: np.ndarray) -> np.ndarray:
    return torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).double().numpy()


@pytest.mark.parametrize("V", [1, 7, 1000, 32000])
@pytest.mark.parametrize("c", [0.0, -3.25, 17.5])
def test_all_equal_row_closed_form(orc, V, c):
    z = np.full((1, V), c, dtype=np.float32)
    st = orc.row_stats(z, tokens=[V - 1])
    assert st.maxprob[0] == pytest.approx(1.0 / V, rel=1e-13)
    assert st.entropy[0] == pytest.approx(math.log(V), rel=1e-12, abs=1e-13)
    assert st.lse[0] == pytest.approx(c + math.log(V), rel=1e-13, abs=1e-13)
    assert st.q[0] == pytest.approx(1.0 / V, rel=1e-13)
    assert st.argmax[0] == 0


@pytest.mark.parametrize("k,V,a,c", [(1, 1000, 5.0, 0.0), (3, 50, 2.0, -1.0), (10, 32000, 12.5, 0.25)])
def test_two_level_row_closed_form(orc, k, V, a, c):
    # k entries at logit a (at indices 5..5+k-1), V-k entries at c
    z = np.full((1, V), c, dtype=np.float32)
    z[0, 5:5 + k] = a
    Z = k * math.exp(a) + (V - k) * math.exp(c)
    p_hi, p_lo = math.exp(a) / Z, math.exp(c) / Z
    H = -(k * p_hi * math.log(p_hi) + (V - k) * p_lo * math.log(p_lo))
    st = orc.row_stats(z, tokens=[5 + k - 1])
    assert st.maxprob[0] == pytest.approx(p_hi, rel=1e-12)
    assert st.q[0] == pytest.approx(p_hi, rel=1e-12)
    assert st.entropy[0] == pytest.approx(H, rel=1e-11)
    assert st.lse[0] == pytest.approx(math.log(Z), rel=1e-13)
    assert st.argmax[0] == 5          # lowest index among the tied maxima
    st2 = orc.row_stats(z, tokens=[0])
    assert st2.q[0] == pytest.approx(p_lo, rel=1e-12)
    assert st2.logq[0] == pytest.approx(c - math.log(Z), rel=1e-13)


def test_planted_margin_is_sigmoid(orc):
    # a token planted m nats above the log-sum-exp of the rest has p = sigmoid(m)
    rng = np.random.default_rng(0)
    z = rng.normal(size=(1, 5000)).astype(np.float32)
    rest = np.delete(z[0].astype(np.float64), 17)
    lse_rest = np.log(np.exp(rest - rest.max()).sum()) + rest.max()
    z[0, 17] = np.float32(lse_rest + 8.0)
    m = float(z[0, 17]) - lse_rest          # margin after fp32 rounding
    st = orc.row_stats(z, tokens=[17])
    assert st.q[0] == pytest.approx(1.0 / (1.0 + math.exp(-m)), rel=1e-12)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_random_rows_vs_library_fp64(orc, dtype):
    rng = np.random.default_rng(1)
    R, V = 6, 3001
    x = (rng.normal(size=(R, V)) * rng.uniform(0.3, 4.0, size=(R, 1))).astype(np.float32)
    if dtype == "bf16":
        z = _bf16_bits(x)
        zf = _bf16_vals(z)
    else:
        z = x
        zf = x.astype(np.float64)
    tok = rng.integers(0, V, size=R)
    st = orc.row_stats(z, tokens=tok)
    t = torch.from_numpy(zf)
    lse = torch.logsumexp(t, dim=-1).numpy()
    p = torch.softmax(t, dim=-1)
    H = torch.special.entr(p).sum(-1).numpy()
    np.testing.assert_allclose(st.lse, lse, rtol=1e-13)
    np.testing.assert_allclose(st.entropy, H, rtol=1e-10)
    np.testing.assert_allclose(st.maxprob, p.max(-1).values.numpy(), rtol=1e-12)
    np.testing.assert_allclose(st.q, p.numpy()[np.arange(R), tok], rtol=1e-12)
    np.testing.assert_array_equal(st.argmax, torch.argmax(t, dim=-1).numpy())


def test_bf16_conversion_is_exact(orc):
    bits = np.arange(0, 65536, dtype=np.uint32).astype(np.uint16)
    vals = _bf16_vals(bits)
    finite = np.isfinite(vals)
    # one-element rows: the maximum of a single finite value is the value itself;
    # rows at or below the -2^23 logit floor have no distribution
    z = bits[finite].reshape(-1, 1)
    st = orc.row_stats(z)
    above = vals[finite] > -2.0 ** 23
    np.testing.assert_array_equal(st.m[above], vals[finite][above])
    assert np.all(np.isnan(st.m[~above])) and (~above).sum() > 0


def test_nonfinite_and_out_of_range(orc):
    z = np.zeros((4, 10), dtype=np.float32)
    z[0, 3] = np.nan
    z[1, 2] = np.inf
    z[2, :] = -np.inf
    st = orc.row_stats(z, tokens=[0, 0, 0, 10])
    assert np.all(np.isnan(st.q)) and np.all(st.argmax == -1)
    # -inf entries in an otherwise finite row are masked tokens, not an error
    z2 = np.zeros((1, 10), dtype=np.float32)
    z2[0, :4] = -np.inf
    st2 = orc.row_stats(z2, tokens=[5])
    assert st2.q[0] == pytest.approx(1 / 6)
    assert st2.entropy[0] == pytest.approx(math.log(6))
    assert st2.argmax[0] == 4


def test_rank_vs_library_sort(orc):
    rng = np.random.default_rng(2)
    for trial in range(20):
        V = int(rng.integers(1, 400))
        # bf16 rows at low precision have many ties
        x = (rng.normal(size=V) * 0.3).astype(np.float32)
        z = _bf16_bits(x)
        zf = _bf16_vals(z)
        order = np.lexsort((np.arange(V), -zf))    # sort by (-z, index)
        pos = np.empty(V, dtype=np.int64)
        pos[order] = np.arange(V)
        for t in rng.integers(0, V, size=5):
            assert orc.rank(z, int(t)) == pos[t]


# ---------------------------------------------------------------------------
# Extended features (App. A.7: probability margin, top-5 probability mass)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("V", [1, 3, 5, 6, 1000])
def test_features_all_equal_row(orc, V):
    z = np.full((1, V), 2.5, np.float32)
    mg, t5 = orc.row_features(z)
    assert mg[0] == pytest.approx(1.0 if V == 1 else 0.0, abs=1e-15)
    assert t5[0] == pytest.approx(min(5, V) / V, rel=1e-13)


@pytest.mark.parametrize("k,V,a", [(1, 100, 3.0), (2, 100, 3.0), (7, 5000, 1.25), (3, 10, -2.0)])
def test_features_two_level_row(orc, k, V, a):
    """k entries at level a, V - k at 0: p_hi = e^a / (k e^a + V - k)."""
    z = np.zeros((1, V), np.float32)
    z[0, np.random.default_rng(k).choice(V, k, replace=False)] = a
    mg, t5 = orc.row_features(z)
    Z = k * math.exp(a) + (V - k)
    hi, lo = math.exp(a) / Z, 1.0 / Z
    top = sorted([hi] * k + [lo] * (V - k), reverse=True)
    assert mg[0] == pytest.approx(top[0] - top[1], rel=1e-12, abs=1e-15)
    assert t5[0] == pytest.approx(sum(top[:5]), rel=1e-12)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_features_vs_library_sort(orc, dtype):
    rng = np.random.default_rng(3)
    R, V = 8, 4003
    x = (rng.normal(size=(R, V)) * rng.uniform(0.3, 6.0, size=(R, 1))).astype(np.float32)
    x[2, :40] = x[2].max()            # a tied maximum (margin 0)
    z, zf = (_bf16_bits(x), _bf16_vals(_bf16_bits(x))) if dtype == "bf16" else (x, x.astype(np.float64))
    mg, t5 = orc.row_features(z)
    p = torch.softmax(torch.from_numpy(zf), dim=-1)
    srt = torch.sort(p, dim=-1, descending=True).values.numpy()
    np.testing.assert_allclose(mg, srt[:, 0] - srt[:, 1], rtol=1e-11, atol=1e-15)
    np.testing.assert_allclose(t5, srt[:, :5].sum(-1), rtol=1e-12)
    assert mg[2] == 0.0


def test_features_nonfinite_and_masked(orc):
    z = np.zeros((4, 50), np.float32)
    z[0, 3] = np.nan
    z[1, :] = -np.inf
    z[2, 10:] = -np.inf                # ten finite entries: top-5 mass 0.5
    z[3, 7] = np.inf
    mg, t5 = orc.row_features(z)
    assert np.isnan(mg[[0, 1, 3]]).all() and np.isnan(t5[[0, 1, 3]]).all()
    assert mg[2] == 0.0 and t5[2] == pytest.approx(0.5, rel=1e-14)
