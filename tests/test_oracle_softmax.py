"""Pins of the oracle's probabilities-from-logits definition (softmax with
temperature, exp_neg = Cody-Waite + degree-7 Taylor in fp32 operations,
fixed-point normaliser) against mathematics the oracle does not use:
libm's double-precision exp, fp64 softmax, exact special cases and
invariances.  The accept rule it feeds is pinned in test_oracle_accept*."""
import math

import numpy as np
import pytest

import oracle

F32_TINY = np.float32(2.0 ** -126)


def test_exp_neg_against_double_exp():
    rng = np.random.default_rng(0)
    x = np.concatenate([
        -rng.uniform(0, 104, 400_000).astype(np.float32),
        -np.float32(2.0) ** -rng.uniform(1, 30, 50_000).astype(np.float32),  # near zero
        np.float32([0.0, -0.0, -np.log(2) / 2, -88.0, -87.3, -100.0, -103.9]),
    ]).astype(np.float32)
    got = oracle.exp_neg(x).astype(np.float64)
    ref = np.exp(x.astype(np.float64))
    normal = ref >= float(F32_TINY)
    # normal range: within 2 units in the last place of fp32
    ulp = np.spacing(ref[normal].astype(np.float32)).astype(np.float64)
    assert np.max(np.abs(got[normal] - ref[normal]) / ulp) <= 2.0
    # subnormal range: within one subnormal step (2^-149) of the true value
    assert np.max(np.abs(got[~normal] - ref[~normal])) <= 2.0 ** -149


def test_exp_neg_special_values():
    e = oracle.exp_neg(np.float32([0.0, -0.0, -104.0, -200.0, -np.inf, np.nan]))
    assert e[0] == 1.0 and e[1] == 1.0
    assert np.all(e[2:] == 0.0)


def _softmax64(z, T):
    z = z.astype(np.float64) / T
    w = np.exp(z - z.max())
    return w / w.sum()


def _rel_bound(z, T):
    # x = (z - max) * (1/T) is formed in fp32: two roundings of relative size
    # 2^-24 put an absolute error of about |x| 2^-23 into x, hence a relative
    # error |x| 2^-23 into e^x; exp_neg adds <= 2 ulp, the normaliser and the
    # division a few 2^-24 more
    x = (z.astype(np.float64).max() - z.astype(np.float64)) / T
    return 6e-7 + 1.2e-7 * x


@pytest.mark.parametrize("V,T,scale", [(1000, 1.0, 2.0), (151936, 1.0, 2.0), (5000, 0.7, 3.0),
                                       (4096, 2.0, 8.0)])
def test_softmax_matches_fp64(V, T, scale):
    z = np.random.default_rng(V).normal(0, scale, V).astype(np.float16)
    p = oracle.softmax_row(z, T).astype(np.float64)
    ref = _softmax64(z, T)
    big = ref > 1e-30
    assert np.all(np.abs(p[big] - ref[big]) <= _rel_bound(z, T)[big] * ref[big])
    assert abs(p.sum() - 1.0) < 1e-5


def test_softmax_equal_logits_is_uniform_exactly():
    for V in (1, 3, 1000, 151936):
        p = oracle.softmax_row(np.full(V, 1.5, np.float16))
        assert np.all(p == np.float32(1.0) / np.float32(V))


def test_softmax_one_hot():
    z = np.full(300, -60.0, np.float16)
    z[17] = 60.0
    p = oracle.softmax_row(z)
    assert p[17] == 1.0 and np.count_nonzero(p) == 1


def test_softmax_shift_invariance_bitwise():
    # z and z + c give the same differences z - max exactly, so the same bits
    z = np.random.default_rng(3).integers(-40, 40, 2000).astype(np.float16)
    a = oracle.softmax_row(z)
    b = oracle.softmax_row((z.astype(np.float32) + 16.0).astype(np.float16))
    assert np.array_equal(a.view(np.uint32), b.view(np.uint32))


def test_softmax_temperature_is_logit_scaling():
    z = np.random.default_rng(5).normal(0, 2, 3000).astype(np.float16)
    for T in (0.5, 2.0, 4.0):
        p = oracle.softmax_row(z, T).astype(np.float64)
        ref = _softmax64(z, T)
        big = ref > 1e-30
        assert np.all(np.abs(p[big] - ref[big]) <= _rel_bound(z, T)[big] * ref[big])


def test_softmax_rejects_bad_arguments():
    with pytest.raises(ValueError):
        oracle.softmax_row(np.zeros(10, np.float16), 0.0)
    with pytest.raises(ValueError):
        oracle.softmax_row(np.zeros(10, np.float16), float("inf"))
    z = np.zeros(10, np.float16)
    z[3] = np.float16(np.inf)
    with pytest.raises(ValueError):
        oracle.softmax_row(z, 1.0)


def test_accept_logits_is_accept_on_softmax_rows():
    # composition: the logits entry point equals oq_accept on the rows it
    # derives (draft logits laid out [K, B, V])
    rng = np.random.default_rng(11)
    B, K, V, T = 3, 4, 777, 0.9
    zp = rng.normal(0, 2, (B, K + 1, V)).astype(np.float16)
    zq = rng.normal(0, 2, (K, B, V)).astype(np.float16)
    draft = rng.integers(0, V, (B, K)).astype(np.int32)
    u = rng.random((B, K + 1)).astype(np.float32)
    p = np.stack([[oracle.softmax_row(zp[b, i], T) for i in range(K + 1)] for b in range(B)])
    q = np.stack([[oracle.softmax_row(zq[i, b], T) for i in range(K)] for b in range(B)])
    for mode in (oracle.ACCEPT_SAMPLE, oracle.ACCEPT_GREEDY):
        st1, n1, t1 = oracle.accept_logits(zp, zq, draft, u, T, mode)
        st2, n2, t2 = oracle.accept(p, q, draft, u, mode)
        assert st1 == st2 and np.array_equal(n1, n2) and np.array_equal(t1, t2)


def test_sample_logits_distribution():
    # the sampled token frequencies follow fp64 softmax (chi-square bound)
    rng = np.random.default_rng(2)
    V = 12
    z = rng.normal(0, 1.5, V).astype(np.float16)
    n = 40_000
    st, toks = oracle.sample_logits(np.tile(z, (n, 1)), rng.random(n).astype(np.float32))
    assert st == oracle.OK
    counts = np.bincount(toks, minlength=V)
    expect = _softmax64(z, 1.0) * n
    chi2 = float(((counts - expect) ** 2 / expect).sum())
    assert chi2 < 40.0  # 11 degrees of freedom: p ~ 4e-5 for a correct sampler
