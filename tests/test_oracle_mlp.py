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
