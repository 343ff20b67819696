"""Pins of the oracle's stand-in survival scorer sigmoid(w2 . GELU(W1 h + b1) + b2)
(the decode-loop workload's scorer, App. A.7 form): textbook values of the
standard normal CDF (GELU(z) = z Phi(z) in its erf form), exact sigmoid
points, the odd identity GELU(z) - GELU(-z) = z, a library fp64
Linear / GELU / sigmoid chain, and invariance under permuting hidden units."""
import math

import numpy as np
import pytest
import torch

PHI_1 = 0.8413447460685429   # Phi(1), standard normal CDF (textbook table value)
PHI_2 = 0.9772498680518208   # Phi(2)


def bf16_bits(x):
    t = torch.as_tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def bf16_vals(bits):
    return torch.from_numpy(np.asarray(bits, dtype=np.uint16).view(np.int16)).view(torch.bfloat16).double().numpy()


def logit(s):
    return np.log(s) - np.log1p(-s)


def test_sigmoid_points(orc):
    h = bf16_bits(np.zeros((2, 8)))
    W1 = bf16_bits(np.zeros((3, 8)))
    w2 = bf16_bits(np.zeros(3))
    b1 = np.zeros(3, np.float32)
    np.testing.assert_array_equal(orc.survival_mlp(h, W1, b1, w2, 0.0), [0.5, 0.5])
    np.testing.assert_allclose(orc.survival_mlp(h, W1, b1, w2, math.log(3.0)), [0.75, 0.75], rtol=0, atol=1e-15)


@pytest.mark.parametrize("z,phi", [(1.0, PHI_1), (2.0, PHI_2)])
def test_gelu_is_erf_form(orc, z, phi):
    # W1 = 0, one hidden unit with bias z, w2 = 1: the pre-sigmoid value is GELU(z) = z Phi(z)
    h = bf16_bits(np.zeros((1, 16)))
    W1 = bf16_bits(np.zeros((1, 16)))
    s = orc.survival_mlp(h, W1, np.array([z], np.float32), bf16_bits([1.0]), 0.0)
    np.testing.assert_allclose(logit(s), [z * phi], rtol=0, atol=1e-12)   # the tanh form is off by 1.5e-4 at z=1


def test_gelu_odd_identity(orc):
    # hidden units (z, -z) with w2 = (1, -1): GELU(z) - GELU(-z) = z for every z
    zs = np.array([-3.0, -0.75, 0.0, 0.5, 2.25, 6.0], np.float32)
    for z in zs:
        h = bf16_bits(np.zeros((1, 8)))
        W1 = bf16_bits(np.zeros((2, 8)))
        s = orc.survival_mlp(h, W1, np.array([z, -z], np.float32), bf16_bits([1.0, -1.0]), 0.125)
        np.testing.assert_allclose(logit(s), [0.125 + float(z)], rtol=0, atol=1e-12)


def test_matches_library_chain(orc):
    rng = np.random.default_rng(5)
    M, K, N = 37, 96, 24
    h = bf16_bits(rng.standard_normal((M, K)))
    W1 = bf16_bits(rng.uniform(-1, 1, (N, K)) / math.sqrt(K))
    w2 = bf16_bits(rng.uniform(-1, 1, N) / 4)
    b1 = rng.uniform(-0.5, 0.5, N).astype(np.float32)
    b2 = 0.3
    lin = torch.nn.functional.linear(torch.from_numpy(bf16_vals(h)), torch.from_numpy(bf16_vals(W1)),
                                     torch.from_numpy(b1.astype(np.float64)))
    g = torch.nn.functional.gelu(lin, approximate="none")
    want = torch.sigmoid(g @ torch.from_numpy(bf16_vals(w2)) + b2).numpy()
    np.testing.assert_allclose(orc.survival_mlp(h, W1, b1, w2, b2), want, rtol=1e-13, atol=0)


def test_hidden_unit_permutation_invariance(orc):
    rng = np.random.default_rng(6)
    M, K, N = 9, 64, 16
    h = bf16_bits(rng.standard_normal((M, K)))
    W1 = bf16_bits(rng.uniform(-1, 1, (N, K)) / 8)
    w2 = bf16_bits(rng.uniform(-1, 1, N))
    b1 = rng.uniform(-1, 1, N).astype(np.float32)
    perm = rng.permutation(N)
    a = orc.survival_mlp(h, W1, b1, w2, -0.2)
    b = orc.survival_mlp(h, W1[perm], b1[perm], w2[perm], -0.2)
    np.testing.assert_allclose(a, b, rtol=1e-14, atol=0)
    # and the rows are independent: scoring a subset gives the same values
    np.testing.assert_array_equal(orc.survival_mlp(h[3:5], W1, b1, w2, -0.2), a[3:5])


# ---------------------------------------------------------------------------
# The learned scorer's shape (App. A.7): K -> N -> N -> N -> 1, GELU, every
# activation in fp64
# ---------------------------------------------------------------------------

def _b(a):
    return torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def _gelu(z):
    return 0.5 * z * (1.0 + math.erf(z / math.sqrt(2.0)))


def _rbf16(v):
    return float(torch.tensor(float(v), dtype=torch.float32).to(torch.bfloat16).float())


def _zeros(N, K):
    return np.zeros((N, K), np.float32), np.zeros(N, np.float32)


def test_deep_zero_weights_closed_form(orc):
    N, K = 8, 16
    W, b = _zeros(N, K)
    b3 = np.linspace(-1.5, 2.0, N).astype(np.float32)
    w4 = np.linspace(0.5, -0.5, N).astype(np.float32)
    x = _b(np.random.default_rng(0).normal(size=(3, K)))
    s = orc.scorer_deep(x, _b(W), b, _b(np.zeros((N, N))), b, _b(np.zeros((N, N))), b3, _b(w4), 0.25)
    w4r = np.asarray(torch.from_numpy(w4).to(torch.bfloat16).float())
    t = 0.25 + sum(float(w4r[n]) * _gelu(float(b3[n])) for n in range(N))
    np.testing.assert_allclose(s, 1.0 / (1.0 + math.exp(-t)), rtol=1e-14)


def test_deep_single_path_closed_form(orc):
    """One weight per layer: s = sigmoid(e GELU(d GELU(c GELU(a x_j + beta)))),
    every other unit sees GELU(0) = 0; the activations are not rounded."""
    N, K, j, i, pu, q = 6, 10, 3, 2, 4, 1
    a, beta, c, d, e = 1.25, 0.3, -0.75, 1.5, 2.0
    W1, z = _zeros(N, K)
    W1[i, j] = a
    b1 = z.copy()
    b1[i] = beta
    W2 = np.zeros((N, N), np.float32)
    W2[pu, i] = c
    W3 = np.zeros((N, N), np.float32)
    W3[q, pu] = d
    w4 = np.zeros(N, np.float32)
    w4[q] = e
    x = np.zeros((2, K), np.float32)
    x[0, j], x[1, j] = 0.6875, -2.5
    s = orc.scorer_deep(_b(x), _b(W1), b1, _b(W2), z, _b(W3), z, _b(w4), 0.0)
    for m in range(2):
        t = e * _gelu(d * _gelu(c * _gelu(a * float(x[m, j]) + float(np.float32(beta)))))
        assert s[m] == pytest.approx(1.0 / (1.0 + math.exp(-t)), rel=1e-14)
        rounded = e * _gelu(d * _rbf16(_gelu(c * _rbf16(_gelu(a * float(x[m, j]) + float(np.float32(beta)))))))
        assert abs(s[m] - 1.0 / (1.0 + math.exp(-rounded))) > 1e-9   # no activation is rounded


def test_deep_matches_library_chain(orc):
    """Special case that reduces to library routines: fp64 torch Linear / gelu
    (erf form) / sigmoid on the same bf16 weights and inputs."""
    rng = np.random.default_rng(11)
    M, K, N = 9, 48, 24
    x = _b(rng.normal(size=(M, K)))
    W1, W2, W3 = (rng.uniform(-1, 1, s) / math.sqrt(s[1]) for s in ((N, K), (N, N), (N, N)))
    b1, b2, b3 = (rng.uniform(-0.3, 0.3, N).astype(np.float32) for _ in range(3))
    w4 = rng.uniform(-1, 1, N) / math.sqrt(N)
    s = orc.scorer_deep(x, _b(W1), b1, _b(W2), b2, _b(W3), b3, _b(w4), 0.125)
    v = lambda a: torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16).double()   # noqa: E731
    F = torch.nn.functional
    a1 = F.gelu(F.linear(torch.from_numpy(bf16_vals(x)), v(W1), torch.from_numpy(b1).double()))
    a2 = F.gelu(F.linear(a1, v(W2), torch.from_numpy(b2).double()))
    a3 = F.gelu(F.linear(a2, v(W3), torch.from_numpy(b3).double()))
    want = torch.sigmoid(a3 @ v(w4) + 0.125).numpy()
    np.testing.assert_allclose(s, want, rtol=1e-12, atol=1e-15)


def test_deep_hidden_unit_permutation_invariance(orc):
    rng = np.random.default_rng(7)
    N, K, M = 16, 40, 5
    x = _b(rng.normal(size=(M, K)))
    W1, W2, W3 = (rng.normal(size=s) * 0.3 for s in ((N, K), (N, N), (N, N)))
    b1, b2, b3 = (rng.normal(size=N).astype(np.float32) * 0.2 for _ in range(3))
    w4 = rng.normal(size=N) * 0.2
    s0 = orc.scorer_deep(x, _b(W1), b1, _b(W2), b2, _b(W3), b3, _b(w4), -0.1)
    p1, p2, p3 = rng.permutation(N), rng.permutation(N), rng.permutation(N)
    s1 = orc.scorer_deep(x, _b(W1[p1]), b1[p1], _b(W2[p2][:, p1]), b2[p2], _b(W3[p3][:, p2]), b3[p3], _b(w4[p3]), -0.1)
    np.testing.assert_allclose(s1, s0, rtol=1e-12)
