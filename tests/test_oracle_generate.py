"""Pins of the oracle's generation pieces (Sec. III-D): the bookkeeping
between cycles, and the cache-free decoder that the GPU generation is
compared with.

The bookkeeping is pinned by running the whole speculative cycle on toy
models whose next token is a hash of everything they have seen: each model
keeps a toy cache (the token fed at every position) and answers from it, so
a wrong position or a missing re-feed shows up twice, as a cache read that
differs from the true sequence and as a continuation that differs from
direct greedy decoding (which speculative decoding must reproduce exactly).
"""
import zlib

import numpy as np
import pytest

import oracle as O
from paper_2609_21704_gb300 import synth


# ---- bookkeeping -------------------------------------------------------------------

def _h(seq, salt=0):
    return zlib.crc32(np.asarray(seq, np.int64).tobytes() + bytes([salt]))


def _target(seq, V):
    return _h(seq) % V


def _draft(seq, V, agree):
    t = _target(seq, V)
    return t if _h(seq, 7) % 100 < agree else (t + 1) % V


class _ToyModel:
    """A model with a cache: feeding token t at position p stores it; the
    output at p is a function of the cached positions 0..p."""

    def __init__(self, cap, fn):
        self.C = [-1] * cap
        self.fn = fn
        self.reads = []

    def forward(self, toks, pos0, truth):
        out = []
        for t, tok in enumerate(toks):
            p = pos0 + t
            self.C[p] = int(tok)
            seen = self.C[:p + 1]
            self.reads.append(seen == list(truth[:p + 1]))
            out.append(self.fn(seen))
        return out


def _speculative(prompt, K, cycles, cap, V, agree):
    P = len(prompt)
    hist = np.zeros((1, cap), np.int32)
    hist[0, :P] = prompt
    length = np.array([P], np.int32)
    tgt = _ToyModel(cap, lambda s: _target(s, V))
    drf = _ToyModel(cap, lambda s: _draft(s, V, agree))
    drf.forward(prompt, 0, list(prompt))
    first = tgt.forward(prompt, 0, list(prompt))[-1]
    hist, length, pos, last2, bad = O.spec_commit(None, np.array([[first]]), hist, length, K)
    assert not bad.any()
    ns = []
    for _ in range(cycles):
        L = int(length[0])
        committed = list(hist[0, :L])
        samples = []
        out = drf.forward(last2[0], int(pos[0, 0]), committed)[-1]
        samples.append(out)
        for k in range(1, K):
            out = drf.forward([samples[-1]], int(pos[k, 0]), committed + samples)[-1]
            samples.append(out)
        verify, draft = O.spec_drafts(np.array(samples, np.int32).reshape(K, 1), last2)
        assert verify[0, 0] == committed[-1] and list(draft[0]) == samples
        p = tgt.forward(verify[0], int(pos[K, 0]), committed + samples)
        n = 0
        while n < K and draft[0, n] == p[n]:
            n += 1
        tokens = np.full((1, K + 1), -1, np.int32)
        tokens[0, :n] = draft[0, :n]
        tokens[0, n] = p[n]
        ns.append(n)
        hist, length, pos, last2, bad = O.spec_commit(np.array([n]), tokens, hist, length, K)
        assert not bad.any()
    return list(hist[0, :length[0]]), ns, tgt.reads, drf.reads


def _direct(prompt, n_new, V):
    seq = list(prompt)
    for _ in range(n_new):
        seq.append(_target(seq, V))
    return seq


@pytest.mark.parametrize("K", [1, 2, 4, 7])
def test_speculative_cycle_is_lossless_and_reads_the_right_cache_entries(K):
    V, cap, cycles = 37, 400, 40
    prompt = [3, 1, 4, 1, 5]
    seq, ns, tr, dr = _speculative(prompt, K, cycles, cap, V, agree=75)
    assert seq == _direct(prompt, len(seq) - len(prompt), V)
    assert all(tr) and all(dr)              # every cache read saw the true sequence
    assert len(seq) == len(prompt) + 1 + sum(n + 1 for n in ns)
    assert K in ns and min(ns) < K          # both all-accepted and rejected cycles ran


def test_dropping_the_refeed_of_the_second_last_token_breaks_the_draft_cache():
    # the plausible mistake (feed only the last token, T = 1 at L - 1) leaves
    # a hole in the draft cache after a cycle that accepted every draft
    V, K, cap = 37, 3, 200
    prompt = [2, 7, 1, 8]
    hist = np.zeros((1, cap), np.int32)
    hist[0, :4] = prompt
    length = np.array([4], np.int32)
    drf = _ToyModel(cap, lambda s: _target(s, V))     # agrees always: n = K every cycle
    tgt = _ToyModel(cap, lambda s: _target(s, V))
    drf.forward(prompt, 0, prompt)
    first = tgt.forward(prompt, 0, prompt)[-1]
    hist, length, pos, last2, _ = O.spec_commit(None, np.array([[first]]), hist, length, K)
    for _ in range(3):
        committed = list(hist[0, :length[0]])
        samples = [drf.forward([last2[0, 1]], int(pos[0, 0]) + 1, committed)[-1]]
        for k in range(1, K):
            samples.append(drf.forward([samples[-1]], int(pos[k, 0]), committed + samples)[-1])
        p = tgt.forward([committed[-1]] + samples, int(pos[K, 0]), committed + samples)
        tokens = np.array([samples + [p[K]]], np.int32)
        hist, length, pos, last2, _ = O.spec_commit(np.array([K]), tokens, hist, length, K)
    assert not all(drf.reads)


def test_commit_positions_and_last_tokens_by_hand():
    hist = np.zeros((2, 16), np.int32)
    hist[0, :5] = [10, 11, 12, 13, 14]
    hist[1, :3] = [20, 21, 22]
    tokens = np.array([[30, 31, 32, -1], [40, -1, -1, -1]], np.int32)
    h, L, pos, last2, bad = O.spec_commit(np.array([2, 0]), tokens, hist, np.array([5, 3]), 3)
    assert list(h[0, :8]) == [10, 11, 12, 13, 14, 30, 31, 32]
    assert list(h[1, :4]) == [20, 21, 22, 40]
    assert list(L) == [8, 4]
    assert pos.tolist() == [[6, 2], [8, 4], [9, 5], [7, 3]]
    assert last2.tolist() == [[31, 32], [22, 40]]
    assert not bad.any()
    # K = 0 (direct decoding): one row, the position of the last token
    _, L0, pos0, _, _ = O.spec_commit(None, np.array([[9], [9]]), hist, np.array([5, 3]), 0)
    assert list(L0) == [6, 4] and pos0.tolist() == [[5, 3]]


def test_commit_edge_cases():
    hist = np.zeros((3, 6), np.int32)
    hist[:, :4] = [[1, 2, 3, 4], [5, 6, 7, 8], [9, 9, 9, 9]]
    tokens = np.array([[7, 7, 7], [1, 2, 3], [4, 4, 4]], np.int32)
    h, L, _, last2, bad = O.spec_commit(np.array([-1, 2, 5]), tokens, hist, np.array([4, 4, 4]), 2)
    assert L[0] == 4 and list(h[0, :4]) == [1, 2, 3, 4] and not bad[0]      # n < 0: nothing
    assert L[1] == 6 and list(h[1]) == [5, 6, 7, 8, 1, 2] and bad[1]         # full history
    assert L[2] == 4 and bad[2]                                             # n >= ldt
    assert last2[1].tolist() == [1, 2]
    _, L1, _, last1, bad1 = O.spec_commit(np.array([-1]), np.array([[0]]), np.zeros((1, 4), np.int32),
                                          np.array([1]), 1)
    assert bad1[0] and last1[0].tolist() == [-1, 0]                         # L < 2


def test_drafts_layout():
    v, d = O.spec_drafts(np.array([[5, 6], [7, 8], [9, 10]]), np.array([[1, 2], [3, 4]]))
    assert v.tolist() == [[2, 5, 7, 9], [4, 6, 8, 10]]
    assert d.tolist() == [[5, 7, 9], [6, 8, 10]]


# ---- the cache-free decoder ---------------------------------------------------------

def _params(L=1, H=256, Hq=2, Hkv=1, inter=384, V=300, seed=1, zero_o=False, zero_down=False):
    D = 128
    rng = np.random.default_rng(seed)
    w = lambda n, k: (rng.standard_normal((n, k)) * 0.05).astype(np.float16).astype(np.float64)
    layers = []
    for _ in range(L):
        qkv, o, gu, dn = w((Hq + 2 * Hkv) * D, H), w(H, Hq * D), w(2 * inter, H), w(H, inter)
        if zero_o:
            o[:] = 0
        if zero_down:
            dn[:] = 0
        layers.append((qkv, o, gu, dn))
    gam = [(1 + 0.1 * rng.standard_normal(H)).astype(np.float64) for _ in range(2 * L + 1)]
    return dict(layers=layers, lm_head=w(V, H), gamma=gam, q_heads=Hq, kv_heads=Hkv, head_dim=D,
                intermediate=inter, eps=1e-6, theta=1e6)


def _norm(x, g, eps=1e-6):
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * g


def test_decoder_without_layers_is_the_tied_embedding_bilinear_form():
    p = _params(L=0)
    tok = [5, 17, 299, 0]
    E = p["lm_head"]
    want = _norm(E[tok], p["gamma"][-1]) @ E.T
    np.testing.assert_allclose(O.decoder_logits(p, tok), want, rtol=1e-12, atol=1e-12)


def test_zero_output_projections_leave_the_residual_stream_alone():
    p = _params(L=2, zero_o=True, zero_down=True)
    q = _params(L=0)
    q["lm_head"], q["gamma"] = p["lm_head"], [p["gamma"][-1]]
    tok = [4, 8, 15, 16, 23]
    np.testing.assert_allclose(O.decoder_logits(p, tok), O.decoder_logits(q, tok), rtol=1e-12, atol=1e-12)


def test_one_token_attention_returns_its_value_rows():
    # n = 1: softmax over one key is 1 and RoPE at position 0 is the
    # identity, so the attention block adds v(h) W_o^T (v = the last Hkv*D
    # columns of qkv, repeated over the Hq/Hkv query heads of its group)
    p = _params(L=1, zero_down=True)
    E = p["lm_head"]
    qkv, o, _, _ = p["layers"][0]
    t = 42
    x = E[[t]]
    h = _norm(x, p["gamma"][0])
    v = (h @ qkv.T)[:, 3 * 128:]                       # Hq = 2, Hkv = 1
    a = np.concatenate([v, v], axis=1)                  # both query heads read kv head 0
    x1 = x + a @ o.T
    want = _norm(x1, p["gamma"][-1]) @ E.T
    np.testing.assert_allclose(O.decoder_logits(p, [t]), want, rtol=1e-10, atol=1e-12)


def test_grouped_heads_equal_duplicated_kv_heads():
    # Hq = 2 over one kv head equals Hq = 2 over two identical kv heads
    p = _params(L=1, Hq=2, Hkv=1, seed=3)
    q = dict(p)
    qkv, o, gu, dn = p["layers"][0]
    D = 128
    qw, kw, vw = qkv[:2 * D], qkv[2 * D:3 * D], qkv[3 * D:]
    q["layers"] = [(np.concatenate([qw, kw, kw, vw, vw]), o, gu, dn)]
    q["kv_heads"] = 2
    tok = [1, 2, 3, 5, 8, 13]
    np.testing.assert_allclose(O.decoder_logits(p, tok), O.decoder_logits(q, tok), rtol=1e-11, atol=1e-12)


def test_decoder_is_causal_and_rows_select_positions():
    p = _params(L=2, seed=5)
    a = [7, 3, 9, 1, 200, 45]
    b = a[:3] + [100, 2, 299]
    za, zb = O.decoder_logits(p, a), O.decoder_logits(p, b)
    np.testing.assert_allclose(za[:3], zb[:3], rtol=1e-12, atol=1e-13)
    assert np.abs(za[3:] - zb[3:]).max() > 1e-3
    np.testing.assert_allclose(O.decoder_logits(p, a, rows=[5, 2]), za[[5, 2]], rtol=0, atol=0)


def test_greedy_generation_extends_by_argmax():
    p = _params(L=1, seed=7)
    prompt = [11, 22, 33]
    toks, gaps = O.generate_greedy(p, prompt, 4)
    seq = prompt + toks
    z = O.decoder_logits(p, seq)
    for i, t in enumerate(toks):
        row = z[len(prompt) - 1 + i]
        assert t == int(np.argmax(row))
        assert gaps[i] == pytest.approx(np.sort(row)[-1] - np.sort(row)[-2], abs=1e-12)


def test_synthetic_prompts_are_seeded_and_in_range():
    a = synth.prompt_tokens(3, 2, 40, 1000)
    assert a.shape == (2, 40) and a.dtype == np.int32
    assert a.min() >= 0 and a.max() < 1000
    np.testing.assert_array_equal(a, synth.prompt_tokens(3, 2, 40, 1000))
    assert not np.array_equal(a, synth.prompt_tokens(4, 2, 40, 1000))
