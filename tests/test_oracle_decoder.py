"""Pins of the oracle's decoder pieces (RMSNorm, RoPE, grouped-query
attention over a cache) by invariants and special cases the definitions
imply, not by restating them: scale invariance and unit mean square of
RMSNorm; norm preservation, additivity of rotations, identity at position
0 and the relative-position property of RoPE; single-key, identical-key,
one-hot-score, permutation, causal-prefix and GQA-sharing properties of
attention."""
import numpy as np

import oracle


def test_rmsnorm_scale_invariance_and_unit_rms():
    rng = np.random.default_rng(0)
    x = rng.normal(0, 3, (5, 64))
    g = np.ones(64)
    y = oracle.rmsnorm(x, g, eps=0.0)
    assert np.allclose(np.sqrt((y ** 2).mean(axis=1)), 1.0, rtol=0, atol=1e-12)
    assert np.allclose(oracle.rmsnorm(7.5 * x, g, eps=0.0), y, rtol=1e-13, atol=0)
    gamma = rng.normal(size=64)
    assert np.allclose(oracle.rmsnorm(x, gamma, eps=0.0), y * gamma, rtol=1e-13, atol=1e-15)


def test_rmsnorm_eps_limit():
    # a zero row stays zero; a tiny row is damped by eps
    y = oracle.rmsnorm(np.zeros((1, 8)), np.ones(8), eps=1e-6)
    assert np.all(y == 0.0)
    y = oracle.rmsnorm(np.full((1, 8), 1e-6), np.ones(8), eps=1e-6)
    assert np.allclose(y, 1e-6 / np.sqrt(1e-12 + 1e-6))


def test_rope_identity_norms_and_additivity():
    rng = np.random.default_rng(1)
    D, H = 128, 3
    x = rng.normal(size=(1, H * D))
    assert np.allclose(oracle.rope(x, [0], H, D), x, rtol=0, atol=0)
    for pos in (1, 17, 1000, 30000):
        r = oracle.rope(x, [pos], H, D).reshape(H, 2, D // 2)
        x3 = x.reshape(H, 2, D // 2)
        # each (d, d + D/2) pair keeps its length
        assert np.allclose(np.hypot(r[:, 0], r[:, 1]), np.hypot(x3[:, 0], x3[:, 1]), rtol=1e-12)
    # rotating by a then by b equals rotating by a + b
    a, b = 123, 4567
    two = oracle.rope(oracle.rope(x, [a], H, D), [b], H, D)
    assert np.allclose(two, oracle.rope(x, [a + b], H, D), rtol=1e-9, atol=1e-9)


def test_rope_relative_position():
    # q(m) . k(n) depends only on m - n
    rng = np.random.default_rng(2)
    D = 128
    q = rng.normal(size=(1, D))
    k = rng.normal(size=(1, D))
    dots = [float((oracle.rope(q, [m], 1, D) @ oracle.rope(k, [m - 5], 1, D).T)[0, 0]) for m in (5, 40, 999)]
    assert np.allclose(dots, dots[0], rtol=1e-9)
    assert not np.isclose(dots[0], float((q @ k.T)[0, 0]))  # the rotation does act


def _qkv(seed, T, L, Hq, Hkv, D):
    rng = np.random.default_rng(seed)
    return rng.normal(size=(T, Hq, D)), rng.normal(size=(L, Hkv, D)), rng.normal(size=(L, Hkv, D))


def test_attention_single_key_returns_its_value():
    q, k, v = _qkv(3, 2, 1, 4, 2, 16)
    out = oracle.attention(q, k, v, [0, 0])
    assert np.allclose(out[:, :2], v[0, 0], rtol=1e-14)
    assert np.allclose(out[:, 2:], v[0, 1], rtol=1e-14)


def test_attention_identical_keys_average_values():
    q, k, v = _qkv(4, 1, 7, 2, 1, 8)
    k[:] = k[0]
    out = oracle.attention(q, k, v, [6])
    assert np.allclose(out[0, 0], v[:, 0].mean(axis=0), rtol=1e-12)


def test_attention_one_hot_scores_pick_a_value():
    D = 16
    q = np.zeros((1, 1, D))
    q[0, 0, 3] = 400.0          # score 400 / 4 = 100 for the matching key
    k = np.zeros((4, 1, D))
    k[2, 0, 3] = 1.0
    v = np.random.default_rng(5).normal(size=(4, 1, D))
    assert np.allclose(oracle.attention(q, k, v, [3])[0, 0], v[2, 0], rtol=1e-12, atol=1e-30)


def test_attention_key_permutation_invariance():
    q, k, v = _qkv(6, 1, 9, 4, 2, 32)
    perm = np.random.default_rng(7).permutation(9)
    a = oracle.attention(q, k, v, [8])
    b = oracle.attention(q, k[perm], v[perm], [8])
    assert np.allclose(a, b, rtol=1e-12)


def test_attention_causal_prefix():
    # a query at position p ignores keys after p: appending more keys, or
    # changing them, leaves its output unchanged
    q, k, v = _qkv(8, 3, 12, 4, 2, 32)
    pos = [4, 7, 11]
    out = oracle.attention(q, k, v, pos)
    k2, v2 = k.copy(), v.copy()
    k2[8:] += 10.0
    v2[8:] -= 3.0
    out2 = oracle.attention(q, k2, v2, pos)
    assert np.allclose(out[:2], out2[:2], rtol=1e-14) and not np.allclose(out[2], out2[2])
    short = oracle.attention(q[:1], k[:5], v[:5], [4])
    assert np.allclose(short[0], out[0], rtol=1e-14)


def test_attention_grouped_heads_share_keys():
    # with Hq = 2 Hkv, query heads 2h and 2h+1 equal single-head attention on kv head h
    q, k, v = _qkv(9, 2, 6, 4, 2, 16)
    out = oracle.attention(q, k, v, [5, 3])
    for h in range(4):
        ref = oracle.attention(q[:, h:h + 1], k[:, h // 2:h // 2 + 1], v[:, h // 2:h // 2 + 1], [5, 3])
        assert np.allclose(out[:, h], ref[:, 0], rtol=1e-14)
