"""Pins for the oracle's linear layers (Sec. III-D.2 draft pass, Sec. III-D.3
verify pass): y = x W^T (+ b) in fp64.

* exact rational arithmetic (fractions) on a small case;
* numpy's float64 matmul (a library routine) on random shapes that are not
  square, so a transposed operand or swapped index cannot pass;
* one-hot activations select one weight column exactly;
* the SiLU gate against scipy's logistic function.
"""
from fractions import Fraction

import numpy as np
import pytest
import scipy.special

import oracle


def test_linear_exact_rationals():
    rng = np.random.default_rng(11)
    M, N, K = 2, 3, 128
    x = rng.standard_normal((M, K)).astype(np.float16).astype(np.float64)
    w = (rng.standard_normal((N, K)) * 0.02).astype(np.float16).astype(np.float64)
    b = rng.standard_normal(N).astype(np.float16).astype(np.float64)
    y = oracle.linear(x, w, b)
    for m in range(M):
        for n in range(N):
            exact = sum(Fraction(x[m, k]) * Fraction(w[n, k]) for k in range(K)) + Fraction(b[n])
            assert abs(Fraction(y[m, n]) - exact) <= abs(exact) * Fraction(1, 2 ** 44) + Fraction(1, 2 ** 80)


@pytest.mark.parametrize("M,N,K", [(1, 7, 256), (5, 33, 128), (9, 4, 640), (3, 1, 1)])
def test_linear_matches_numpy(M, N, K):
    rng = np.random.default_rng(M * 1000 + N)
    x = rng.standard_normal((M, K))
    w = rng.standard_normal((N, K))
    b = rng.standard_normal(N)
    y = oracle.linear(x, w, b)
    assert y.shape == (M, N)
    np.testing.assert_allclose(y, x @ w.T + b, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(oracle.linear(x, w), x @ w.T, rtol=1e-12, atol=1e-12)


def test_linear_one_hot_selects_column_exactly():
    rng = np.random.default_rng(12)
    N, K = 17, 384
    w = (rng.standard_normal((N, K)) * 0.02).astype(np.float16).astype(np.float64)
    for k in (0, 1, 200, K - 1):
        x = np.zeros((1, K))
        x[0, k] = 1.0
        assert np.array_equal(oracle.linear(x, w)[0], w[:, k])


def test_silu_gate_matches_scipy():
    g = np.linspace(-20, 20, 4001)
    u = np.cos(g)
    h = oracle.silu_gate(g, u)
    np.testing.assert_allclose(h, g * scipy.special.expit(g) * u, rtol=1e-14, atol=1e-300)
    assert oracle.silu_gate(np.array([0.0]), np.array([5.0]))[0] == 0.0
