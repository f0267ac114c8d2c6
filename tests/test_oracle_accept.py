"""Pins for the oracle's accept / correct / resample step.

Sec. III-A.3 gives the token rule (keep the draft token if the parent agrees,
otherwise the parent's own prediction); Sec. III-D.4 says the result is
guaranteed correct; Sec. I says the method adheres to standard speculative
decoding.  The oracle implements the greedy rule literally and, by default,
the lossless speculative-sampling rule.  These tests pin it by:

* exhaustive enumeration over the full 2^24 uniform grid at V = 8, K = 2:
  the emitted first token is distributed exactly as the target p_1, and the
  first two emitted tokens exactly as p_1 x p_2 (and as p_1(a) p_2(b | a) for
  prefix-dependent tables);
* closed forms: P(accept) = sum_v min(p, q) at every position;
* K = 0 equals a textbook searchsorted on the integer CDF;
* exact integer arithmetic for the fixed-point helpers (Python big ints);
* special cases: p == q accepts everything, a one-hot target forces its
  token, greedy output equals the parent's argmax predictions;
* a Monte-Carlo run of the batched call for the composition.
"""
import math
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2609_21704_gb300 import synth

SAMPLE, GREEDY = oracle.ACCEPT_SAMPLE, oracle.ACCEPT_GREEDY
GRID = 24
ALMOST_ONE = np.float32(1.0 - 2.0 ** -24)


# ---------------------------------------------------------------- helpers

def _dyadic_dist(rng, V, bits=12, zero_some=False):
    """A probability vector with entries k / 2^bits summing to exactly 1 (so
    fp32 holds it exactly and p - q is exact)."""
    total = 1 << bits
    cuts = np.sort(rng.choice(np.arange(1, total), size=V - 1, replace=False))
    k = np.diff(np.concatenate([[0], cuts, [total]])).astype(np.float64)
    if zero_some:
        j = rng.integers(0, V)
        k[(j + 1) % V] += k[j]
        k[j] = 0
    return (k / total).astype(np.float32)


def _grid_prob(count):
    return count / float(1 << GRID)


# ---------------------------------------------------------------- fixed point

@pytest.mark.parametrize("r", [0.0, 1.0, 2.0 ** -44, 2.0 ** -45, 0.3, 1 / 3, 0.999999940395, 1e-20])
def test_fix44_is_exact_floor(r):
    r32 = np.float32(r)
    assert oracle.fix44(r32) == math.floor(Fraction(float(r32)) * 2 ** 44)


def test_scale_floor_is_exact_big_int():
    rng = np.random.default_rng(5)
    for _ in range(2000):
        u = np.float32(rng.integers(0, 1 << 24) * 2.0 ** -24) if rng.random() < 0.5 \
            else np.float32(rng.random())
        S = int(rng.integers(0, 1 << 63)) * 2 + int(rng.integers(0, 2))
        assert oracle.scale_floor(u, S) == math.floor(Fraction(float(u)) * S)
    assert oracle.scale_floor(np.float32(1e-40), (1 << 64) - 1) == math.floor(Fraction(float(np.float32(1e-40))) * ((1 << 64) - 1))


# ---------------------------------------------------------------- K = 0

def test_k0_equals_searchsorted_on_integer_cdf():
    rng = np.random.default_rng(6)
    B, V = 64, 1000
    p, _, _, u = synth.spec_block(21, B, 0, V)
    p[3, 0, :] = 0
    p[3, 0, 17] = 0.25           # single-token mass
    p[4, 0, ::2] = 0             # zero-mass tokens are never chosen
    st, n, tok = oracle.accept(p, None, np.zeros((B, 0), np.int32), u, SAMPLE)
    st2, tok2 = oracle.sample(p[:, 0, :], u[:, 0])
    assert st == oracle.OK and st2 == oracle.OK
    assert np.array_equal(tok[:, 0], tok2) and (n == 0).all()
    for b in range(B):
        R = [math.floor(Fraction(float(x)) * 2 ** 44) for x in p[b, 0]]
        C = np.cumsum(np.array(R, dtype=object))
        T = math.floor(Fraction(float(u[b, 0])) * int(C[-1]))
        want = int(np.searchsorted(np.array([int(c) for c in C], dtype=np.uint64),
                                   np.uint64(T), side="right"))
        assert tok[b, 0] == want
        assert p[b, 0, want] > 0
    assert tok[3, 0] == 17


# ---------------------------------------------------------------- special cases

def test_identical_draft_and_target_accepts_everything():
    B, K, V = 32, 6, 500
    p, _, draft, u = synth.spec_block(22, B, K, V)
    q = p[:, :K, :].copy()
    # draft tokens with positive mass under q
    st, n, tok = oracle.accept(p, q, draft, u, SAMPLE)
    assert st == oracle.OK
    assert (n == K).all()
    assert np.array_equal(tok[:, :K], draft)


def test_one_hot_target_forces_token():
    B, K, V = 16, 3, 64
    p, q, draft, u = synth.spec_block(23, B, K, V, draft_noise=None)
    p[:] = 0
    p[:, :, 9] = 1.0
    draft[:] = 10                  # never the target token
    st, n, tok = oracle.accept(p, q, draft, u, SAMPLE)
    assert (n == 0).all() and (tok[:, 0] == 9).all() and (tok[:, 1:] == -1).all()


def test_zero_draft_prob_with_positive_target_accepts():
    p = np.zeros((1, 2, 4), np.float32)
    q = np.zeros((1, 1, 4), np.float32)
    p[0, 0] = [0.25, 0.25, 0.25, 0.25]
    p[0, 1] = [1, 0, 0, 0]
    q[0, 0] = [0, 0.5, 0.5, 0]
    st, n, tok = oracle.accept(p, q, np.array([[3]], np.int32),
                               np.array([[0.9, 0.1]], np.float32), SAMPLE)
    assert n[0] == 1 and tok[0].tolist() == [3, 0]


def test_invalid_draft_token_and_uniform_flag_the_sequence():
    p, q, draft, u = synth.spec_block(24, 3, 2, 16)
    draft[1, 1] = 16
    u[2, 2] = 1.0
    st, n, tok = oracle.accept(p, q, draft, u, SAMPLE)
    assert st == oracle.BAD_SEQ
    assert n[0] >= 0 and n[1] == -1 and n[2] == -1
    assert (tok[1] == -1).all() and (tok[2] == -1).all()


def test_greedy_follows_the_token_rule_literally():
    # Hand-worked: V = 4, K = 3.  Parent argmax per position: 2, 0, 3, 1.
    p = np.array([[[0.1, 0.2, 0.6, 0.1],
                   [0.5, 0.2, 0.2, 0.1],
                   [0.1, 0.1, 0.1, 0.7],
                   [0.1, 0.6, 0.2, 0.1]]], np.float32)
    u = np.zeros((1, 4), np.float32)
    cases = {  # draft -> (n, tokens)
        (2, 0, 3): (3, [2, 0, 3, 1]),   # parent agrees everywhere, bonus token 1
        (2, 0, 1): (2, [2, 0, 3, -1]),  # disagrees at the third: parent's 3 instead
        (1, 0, 3): (0, [2, -1, -1, -1]),
        (2, 3, 3): (1, [2, 0, -1, -1]),
    }
    for d, (n_want, t_want) in cases.items():
        st, n, tok = oracle.accept(p, None, np.array([d], np.int32), u, GREEDY)
        assert st == oracle.OK and n[0] == n_want and tok[0].tolist() == t_want


def test_greedy_ties_take_lowest_index_and_match_argmax_property():
    rng = np.random.default_rng(8)
    B, K, V = 200, 4, 6
    p = rng.integers(0, 3, size=(B, K + 1, V)).astype(np.float32)  # many ties
    p[:, :, 0] += 0.0
    am = p.argmax(axis=2)  # numpy: first (lowest) index among maxima
    draft = np.where(rng.random((B, K)) < 0.7, am[:, :K], rng.integers(0, V, (B, K))).astype(np.int32)
    st, n, tok = oracle.accept(p, None, draft, np.zeros((B, K + 1), np.float32), GREEDY)
    for b in range(B):
        mism = np.nonzero(draft[b] != am[b, :K])[0]
        n_want = int(mism[0]) if len(mism) else K
        assert n[b] == n_want
        assert tok[b, : n_want + 1].tolist() == am[b, : n_want + 1].tolist()
        assert (tok[b, n_want + 1:] == -1).all()


# ---------------------------------------------------------------- exhaustive enumeration

def _sweep(p, q, draft, ufix, pos, grid=GRID):
    h = oracle.enum_sweep(p, q, np.asarray(draft, np.int32), np.asarray(ufix, np.float32), pos,
                          grid_bits=grid)
    K = p.shape[0] - 1
    V = p.shape[1]
    assert h[-1] == 0, "no invalid outcomes expected"
    return h[:-1].reshape(K + 1, V).astype(np.float64) / float(1 << grid)


def _first_token_law(p, q, V, grid=GRID):
    """Distribution of the first emitted token, from sweeps of the actual
    oq_accept over every grid value of the uniforms it depends on."""
    A1 = np.zeros(V)
    for x1 in range(V):
        h = _sweep(p, q, [x1, 0], [0, 0, 0.5], 0, grid)
        A1[x1] = h[1:].sum()                   # outcomes with n >= 1
    x1r = int(np.argmax(q[0] - p[0, :]))
    assert q[0, x1r] > p[0, x1r]
    hr = _sweep(p, q, [x1r, 0], [ALMOST_ONE, 0, 0], 2, grid)
    assert hr[1:].sum() == 0                    # always rejected at position 1
    R1 = hr[0]
    law = np.array([q[0, a] * A1[a] for a in range(V)]) + (q[0] * (1 - A1)).sum() * R1
    return law, A1, R1


@pytest.mark.parametrize("seed", [0, 1])
def test_enumeration_first_token_is_target_distributed(seed):
    rng = np.random.default_rng(100 + seed)
    V, K = 8, 2
    p = np.stack([_dyadic_dist(rng, V, zero_some=(seed == 1)) for _ in range(K + 1)])
    q = np.stack([_dyadic_dist(rng, V) for _ in range(K)])
    law, A1, _ = _first_token_law(p, q, V)
    tol = V * 2.0 ** -24 + 2.0 ** -40
    assert np.max(np.abs(law - p[0])) <= tol
    # closed form of the acceptance probability: sum_v min(p, q)
    assert abs((q[0] * A1).sum() - np.minimum(p[0], q[0]).sum()) <= V * 2.0 ** -24


def test_enumeration_first_two_tokens_prefix_independent():
    rng = np.random.default_rng(200)
    V, K = 8, 2
    p = np.stack([_dyadic_dist(rng, V) for _ in range(K + 1)])
    q = np.stack([_dyadic_dist(rng, V) for _ in range(K)])
    law1, A1, R1 = _first_token_law(p, q, V)
    # position 2, given the first draft token was accepted (u_1 = 0 accepts
    # any x_1 with positive target mass)
    x1a = int(np.argmax(p[0]))
    A2 = np.zeros(V)
    for x2 in range(V):
        h = _sweep(p, q, [x1a, x2], [0, 0, 0.5], 1)
        assert h[0].sum() == 0
        A2[x2] = h[2].sum()
    x2r = int(np.argmax(q[1] - p[1]))
    hr = _sweep(p, q, [x1a, x2r], [0, ALMOST_ONE, 0], 2)
    assert hr[1].sum() == 1.0
    R2 = hr[1]
    hb = _sweep(p, q, [x1a, int(np.argmax(p[1]))], [0, 0, 0], 2)
    assert hb[2].sum() == 1.0
    bonus = hb[2]
    second_given_accept = q[1] * A2 + (q[1] * (1 - A2)).sum() * R2
    joint = np.outer(q[0] * A1, second_given_accept) \
        + (q[0] * (1 - A1)).sum() * np.outer(R1, p[1])  # next cycle starts with p_2
    tol = 2 * V * 2.0 ** -24 + 2.0 ** -40
    assert np.max(np.abs(joint - np.outer(p[0], p[1]))) <= tol
    # the bonus position samples p_3 itself
    assert np.max(np.abs(bonus - p[2])) <= V * 2.0 ** -24 + 2.0 ** -40
    assert abs((q[1] * A2).sum() - np.minimum(p[1], q[1]).sum()) <= V * 2.0 ** -24


def test_enumeration_first_two_tokens_prefix_dependent():
    """Tables at position 2 depend on the token emitted at position 1."""
    rng = np.random.default_rng(300)
    V, grid = 8, 20
    p1, q1 = _dyadic_dist(rng, V), _dyadic_dist(rng, V)
    p2 = np.stack([_dyadic_dist(rng, V) for _ in range(V)])   # p2[a] = p_2(. | a)
    q2 = np.stack([_dyadic_dist(rng, V) for _ in range(V)])
    p3 = _dyadic_dist(rng, V)

    def tables(a):
        return np.stack([p1, p2[a], p3]), np.stack([q1, q2[a]])

    joint = np.zeros((V, V))
    # rejection at position 1: the residual law does not depend on the
    # position-2 tables; the next cycle emits from p_2(. | t1)
    pa, qa = tables(0)
    A1 = np.zeros(V)
    for x1 in range(V):
        pp, qq = tables(x1)
        A1[x1] = _sweep(pp, qq, [x1, 0], [0, 0, 0.5], 0, grid)[1:].sum()
    x1r = int(np.argmax(q1 - p1))
    pp, qq = tables(x1r)
    R1 = _sweep(pp, qq, [x1r, 0], [ALMOST_ONE, 0, 0], 2, grid)[0]
    joint += (q1 * (1 - A1)).sum() * R1[:, None] * p2
    for a in range(V):
        if q1[a] * A1[a] == 0:
            continue
        pp, qq = tables(a)
        A2 = np.array([_sweep(pp, qq, [a, x2], [0, 0, 0.5], 1, grid)[2].sum() for x2 in range(V)])
        x2r = int(np.argmax(q2[a] - p2[a]))
        R2 = _sweep(pp, qq, [a, x2r], [0, ALMOST_ONE, 0], 2, grid)[1]
        joint[a] += q1[a] * A1[a] * (q2[a] * A2 + (q2[a] * (1 - A2)).sum() * R2)
    want = p1[:, None] * p2
    assert np.max(np.abs(joint - want)) <= 2 * V * 2.0 ** -grid + 2.0 ** -40


def test_monte_carlo_batched_composition():
    """The batched call, with independent uniforms for every decision,
    reproduces the target law of the first emitted token (chi-square)."""
    rng = np.random.default_rng(400)
    V, K, B = 8, 2, 200_000
    p1 = np.stack([_dyadic_dist(rng, V) for _ in range(K + 1)])
    q1 = np.stack([_dyadic_dist(rng, V) for _ in range(K)])
    p = np.broadcast_to(p1, (B, K + 1, V)).copy()
    q = np.broadcast_to(q1, (B, K, V)).copy()
    draft = np.stack([rng.choice(V, size=B, p=q1[i].astype(np.float64)) for i in range(K)], 1)
    u = synth.uniforms(77, (B, K + 1))
    st, n, tok = oracle.accept(p, q, draft.astype(np.int32), u, SAMPLE)
    assert st == oracle.OK
    counts = np.bincount(tok[:, 0], minlength=V)
    expected = p1[0].astype(np.float64) * B
    mask = expected > 0
    chi2 = (((counts - expected) ** 2)[mask] / expected[mask]).sum()
    assert chi2 < 30.0            # 7 degrees of freedom: p ~ 1e-4 at 30
    assert counts[~mask].sum() == 0
    beta = np.minimum(p1[:K], q1).sum(axis=1)
    mean_n = beta[0] + beta[0] * beta[1]
    assert abs(n.mean() - mean_n) < 5 * math.sqrt(2.0 / B)


def test_exact_tie_rejects():
    # u * q(x) == p(x) exactly: the test is a strict "<", so the draft is
    # rejected; the residual max(0, p - q) then puts all mass on token 1.
    p = np.array([[[0.25, 0.75], [0.5, 0.5]]], np.float32)
    q = np.array([[[0.5, 0.5]]], np.float32)
    st, n, tok = oracle.accept(p, q, np.array([[0]], np.int32),
                               np.array([[0.5, 0.3]], np.float32), SAMPLE)
    assert n[0] == 0 and tok[0].tolist() == [1, -1]
    st, n, tok = oracle.accept(p, q, np.array([[0]], np.int32),
                               np.array([[0.4999999701976776, 0.3]], np.float32), SAMPLE)
    assert n[0] == 1 and tok[0, 0] == 0


def test_inverse_cdf_boundaries_by_hand():
    # p = [1/4, 1/4, 1/2]: R = [2^42, 2^42, 2^43], S = 2^44.  A uniform that
    # lands exactly on a cumulative boundary belongs to the next token:
    # u = 1/4 -> T = 2^42 = R_0, so the token is 1 (the smallest v with
    # R_0 + ... + R_v > T).
    p = np.array([[0.25, 0.25, 0.5]], np.float32)
    for u, want in ((0.0, 0), (0.25 - 2.0 ** -24, 0), (0.25, 1), (0.5, 2), (1 - 2.0 ** -24, 2)):
        st, tok = oracle.sample(p, np.array([u], np.float32))
        assert tok[0] == want, (u, tok[0])
    # u = 0 never selects a leading zero-mass token.
    p0 = np.array([[0.0, 0.0, 0.5, 0.5]], np.float32)
    assert oracle.sample(p0, np.array([0.0], np.float32))[1][0] == 2
