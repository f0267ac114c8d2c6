"""GPU parity: probabilities from logits (sq_softmax) bit for bit, and the
accept / sample step on logits (sq_accept_logits, sq_sample_logits) against
the oracle: identical n_accepted and tokens in both modes, over K = 0..16,
ragged vocabularies, several temperatures, correlated and independent
draft logits; workspace reuse; a non-finite logit invalidates only its own
sequence and sets SQ_DEV_NONFINITE_LOGIT."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_21704_gb300 as sq

from gpu_util import dev

pytestmark = pytest.mark.gpu


def _logits(seed, B, K, V, draft_noise):
    rng = np.random.default_rng(seed)
    zp = rng.normal(0, 2.0, (B, K + 1, V)).astype(np.float16)
    if draft_noise is None:
        zq = rng.normal(0, 2.0, (K, B, V)).astype(np.float16)
    else:
        base = np.transpose(zp[:, :K, :], (1, 0, 2)).astype(np.float32)
        zq = (base + rng.normal(0, draft_noise, (K, B, V))).astype(np.float16)
    # draft tokens: the draft's argmax-ish picks (so some get accepted)
    draft = np.argmax(np.transpose(zq, (1, 0, 2)), axis=2).astype(np.int32) if K else \
        np.zeros((B, 0), np.int32)
    flip = rng.random((B, K)) < 0.3
    draft = np.where(flip, rng.integers(0, V, (B, K)), draft).astype(np.int32)
    u = rng.random((B, K + 1)).astype(np.float32)
    return zp, zq, draft, u


def _t(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev())


@pytest.mark.parametrize("R,V,T", [(5, 151936, 1.0), (3, 152064, 0.7), (33, 9001, 2.3), (1, 1, 1.0)])
def test_softmax_bit_exact(R, V, T):
    z = np.random.default_rng(R * V).normal(0, 3.0, (R, V)).astype(np.float16)
    ws = torch.zeros(sq.sq_softmax_workspace_bytes(R, V), dtype=torch.uint8, device=dev())
    p = torch.empty(R, V, dtype=torch.float32, device=dev())
    sq.sq_softmax(_t(z), T, p, ws)
    assert sq.sq_check() == 0
    got = p.cpu().numpy()
    for r in range(R):
        ref = oracle.softmax_row(z[r], T)
        assert np.array_equal(got[r].view(np.uint32), ref.view(np.uint32)), f"row {r}"


def test_softmax_nonfinite_row():
    z = np.random.default_rng(1).normal(0, 1, (3, 5000)).astype(np.float16)
    z[1, 4321] = np.float16(np.inf)
    ws = torch.zeros(sq.sq_softmax_workspace_bytes(3, 5000), dtype=torch.uint8, device=dev())
    p = torch.empty(3, 5000, dtype=torch.float32, device=dev())
    sq.sq_softmax(_t(z), 1.0, p, ws)
    assert sq.sq_check() & sq.SQ_DEV_NONFINITE_LOGIT
    got = p.cpu().numpy()
    assert np.all(np.isnan(got[1]))
    for r in (0, 2):
        assert np.array_equal(got[r].view(np.uint32), oracle.softmax_row(z[r]).view(np.uint32))


CASES = [
    # B, K, V, T, draft noise (None: independent draft logits), mode
    (1, 4, 151936, 1.0, 0.5, sq.SQ_ACCEPT_SAMPLE),
    (1, 4, 151936, 0.7, 0.5, sq.SQ_ACCEPT_SAMPLE),
    (3, 2, 5000, 1.3, None, sq.SQ_ACCEPT_SAMPLE),
    (8, 5, 152064, 1.0, 0.5, sq.SQ_ACCEPT_SAMPLE),
    (4, 16, 3000, 1.0, 0.3, sq.SQ_ACCEPT_SAMPLE),
    (16, 8, 9001, 0.9, 0.2, sq.SQ_ACCEPT_SAMPLE),
    (2, 8, 32000, 1.0, 0.5, sq.SQ_ACCEPT_GREEDY),
    (5, 3, 4097, 2.0, None, sq.SQ_ACCEPT_GREEDY),
    (6, 0, 20000, 1.0, None, sq.SQ_ACCEPT_SAMPLE),
]


@pytest.mark.parametrize("B,K,V,T,noise,mode", CASES)
def test_accept_logits_matches_oracle(B, K, V, T, noise, mode):
    zp, zq, draft, u = _logits(B * 1000 + K * 10 + V, B, K, V, noise)
    ws = torch.zeros(sq.sq_accept_logits_workspace_bytes(B, K, V), dtype=torch.uint8, device=dev())
    n = torch.empty(B, dtype=torch.int32, device=dev())
    tok = torch.empty(B, K + 1, dtype=torch.int32, device=dev())
    args = (_t(zp), _t(zq) if K else None, _t(draft), _t(u), T, mode, n, tok, ws)
    sq.sq_accept_logits(*args)
    assert sq.sq_check() == 0
    st, on, otok = oracle.accept_logits(zp, zq if K else None, draft, u, T,
                                        oracle.ACCEPT_SAMPLE if mode == sq.SQ_ACCEPT_SAMPLE
                                        else oracle.ACCEPT_GREEDY)
    assert np.array_equal(n.cpu().numpy(), on)
    assert np.array_equal(tok.cpu().numpy(), otok)
    # the same workspace again (its counters were left at zero)
    n2, tok2 = n.clone(), tok.clone()
    n.fill_(-7)
    sq.sq_accept_logits(*args)
    assert sq.sq_check() == 0
    assert torch.equal(n, n2) and torch.equal(tok, tok2)


def test_accept_logits_outcome_spread():
    # with correlated draft logits every outcome class shows up across the batch
    B, K, V = 64, 4, 2000
    zp, zq, draft, u = _logits(77, B, K, V, 0.5)
    ws = torch.zeros(sq.sq_accept_logits_workspace_bytes(B, K, V), dtype=torch.uint8, device=dev())
    n = torch.empty(B, dtype=torch.int32, device=dev())
    tok = torch.empty(B, K + 1, dtype=torch.int32, device=dev())
    sq.sq_accept_logits(_t(zp), _t(zq), _t(draft), _t(u), 1.0, sq.SQ_ACCEPT_SAMPLE, n, tok, ws)
    assert sq.sq_check() == 0
    _, on, otok = oracle.accept_logits(zp, zq, draft, u, 1.0)
    assert np.array_equal(n.cpu().numpy(), on) and np.array_equal(tok.cpu().numpy(), otok)
    assert len(set(on.tolist())) >= 3


@pytest.mark.parametrize("B,V,T", [(1, 151936, 1.0), (7, 12345, 0.6)])
def test_sample_logits_matches_oracle(B, V, T):
    rng = np.random.default_rng(B + V)
    z = rng.normal(0, 2.0, (B, V)).astype(np.float16)
    u = rng.random(B).astype(np.float32)
    ws = torch.zeros(sq.sq_accept_logits_workspace_bytes(B, 0, V), dtype=torch.uint8, device=dev())
    tok = torch.empty(B, 1, dtype=torch.int32, device=dev())
    sq.sq_sample_logits(_t(z), _t(u), T, tok, ws)
    assert sq.sq_check() == 0
    _, otok = oracle.sample_logits(z, u, T)
    assert np.array_equal(tok.cpu().numpy()[:, 0], otok)


def test_nonfinite_logit_invalidates_its_sequence_only():
    B, K, V = 2, 3, 6000
    zp, zq, draft, u = _logits(5, B, K, V, 0.5)
    zq[1, 0, 17] = np.float16(np.nan)  # draft step 1, sequence 0
    ws = torch.zeros(sq.sq_accept_logits_workspace_bytes(B, K, V), dtype=torch.uint8, device=dev())
    n = torch.empty(B, dtype=torch.int32, device=dev())
    tok = torch.empty(B, K + 1, dtype=torch.int32, device=dev())
    sq.sq_accept_logits(_t(zp), _t(zq), _t(draft), _t(u), 1.0, sq.SQ_ACCEPT_SAMPLE, n, tok, ws)
    assert sq.sq_check() & sq.SQ_DEV_NONFINITE_LOGIT
    nn, tt = n.cpu().numpy(), tok.cpu().numpy()
    assert nn[0] == -1 and np.all(tt[0] == -1)
    _, on, otok = oracle.accept_logits(zp[1:], zq[:, 1:], draft[1:], u[1:], 1.0)
    assert nn[1] == on[0] and np.array_equal(tt[1], otok[0])
