"""GPU parity: sq_accept / sq_sample (Sec. III-A.3 token rule, Sec. III-D.4
acceptance and correction) against the oracle, bit-exact on identical fp32
p, q, draft tokens and uniforms, plus the exhaustive V=8, K=2 sweep run on
the GPU and compared count for count with the oracle's."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_21704_gb300 as sq
from paper_2609_21704_gb300 import synth

from gpu_util import dev

pytestmark = pytest.mark.gpu


def _t(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev())


def _gpu_accept(p, q, draft, u, mode=sq.SQ_ACCEPT_SAMPLE):
    B, K1, V = p.shape
    ws = torch.zeros(sq.sq_accept_workspace_bytes(B, K1 - 1, V), dtype=torch.uint8, device=dev())
    n = torch.full((B,), -7, dtype=torch.int32, device=dev())
    tok = torch.full((B, K1), -7, dtype=torch.int32, device=dev())
    sq.sq_accept(_t(p), None if q is None else _t(q), _t(draft), _t(u), mode, n, tok, ws)
    bits = sq.sq_check()
    return n.cpu().numpy(), tok.cpu().numpy(), bits, ws


def _assert_same(p, q, draft, u, mode=sq.SQ_ACCEPT_SAMPLE):
    n, tok, bits, ws = _gpu_accept(p, q, draft, u, mode)
    st, on, otok = oracle.accept(p, q, draft, u, mode)
    assert np.array_equal(n, on), (n, on)
    assert np.array_equal(tok, otok)
    B = p.shape[0]
    ctr = ws[: 4 * B].view(torch.int32)
    assert int(ctr.abs().sum()) == 0, "ticket counters must return to zero"
    return n, tok, bits, st


@pytest.mark.parametrize("B,K,V,noise", [
    (1, 4, 32000, None),          # 0.5B MLP workload: independent draft logits
    (1, 2, 152064, 0.5), (1, 4, 152064, 0.5), (1, 8, 152064, 0.5),  # 7B, target + N(0, 0.5)
    (8, 5, 152064, 0.5),          # 7B batch 8 x (K+1)=6
    (4, 4, 151936, 0.5),          # 1.5B vocabulary
    (16, 8, 5000, None), (3, 1, 2049, 0.5), (2, 3, 2048, None), (5, 16, 777, 0.5),
])
def test_accept_sampling_bitexact(B, K, V, noise):
    p, q, draft, u = synth.spec_block(B * 100 + K * 10 + V % 97, B, K, V, draft_noise=noise)
    n, tok, bits, st = _assert_same(p, q, draft, u)
    assert bits == 0 and st == oracle.OK


@pytest.mark.parametrize("B,K,V", [(1, 4, 32000), (8, 5, 152064), (4, 0, 1000), (3, 16, 2100)])
def test_accept_greedy_bitexact(B, K, V):
    p, q, draft, u = synth.spec_block(B + K + V, B, K, V, draft_noise=0.5)
    am = p.argmax(axis=2)
    draft[:, : K // 2] = am[:, : K // 2]   # force some agreement
    _assert_same(p, None, draft, u, sq.SQ_ACCEPT_GREEDY)


def test_k0_sampling_and_sq_sample():
    B, V = 12, 152064
    p, _, _, u = synth.spec_block(41, B, 0, V)
    _assert_same(p, None, np.zeros((B, 0), np.int32), u)
    ws = torch.zeros(sq.sq_accept_workspace_bytes(B, 0, V), dtype=torch.uint8, device=dev())
    tok = torch.empty(B, dtype=torch.int32, device=dev())
    sq.sq_sample(_t(p[:, 0, :]), _t(u[:, 0]), tok, ws)
    st, otok = oracle.sample(p[:, 0, :], u[:, 0])
    assert np.array_equal(tok.cpu().numpy(), otok)


def test_edge_cases_bitexact():
    B, K, V = 8, 3, 4100
    p, q, draft, u = synth.spec_block(42, B, K, V, draft_noise=None)
    q[0] = p[0, :K]                    # identical draft: all accepted
    draft[0] = p[0, :K].argmax(axis=1)
    p[1, :, :] = 0
    p[1, :, 4099] = 1.0                # one-hot target at the last token
    draft[2, 1] = V                    # draft token out of range
    u[3, K] = 1.0                      # correction uniform out of range
    p[4, 0, :] = q[4, 0, :] * np.float32(0.5)  # p <= q everywhere: rejected draft,
    u[4, 0] = np.float32(0.9)                  # residual without mass -> fallback to p
    p[5, 0, :] = 0                     # row 0 empty: zero target mass for every draft
    p[5, 0, 7] = 2.0 ** -40            # below the 2^-44 grid after subtraction
    u[6, :] = 0.0                      # u = 0 everywhere
    n, tok, bits, st = _assert_same(p, q, draft, u)
    assert n[2] == -1 and n[3] == -1 and (tok[2] == -1).all()
    assert bits & sq.SQ_DEV_BAD_DRAFT_TOKEN and bits & sq.SQ_DEV_BAD_UNIFORM


def test_row_without_mass_is_flagged():
    p = np.zeros((1, 1, 64), np.float32)
    u = np.array([[0.5]], np.float32)
    n, tok, bits, st = _assert_same(p, None, np.zeros((1, 0), np.int32), u)
    assert n[0] == -1 and bits & sq.SQ_DEV_NO_MASS


def _dyadic(rng, V, bits=12):
    cuts = np.sort(rng.choice(np.arange(1, 1 << bits), size=V - 1, replace=False))
    k = np.diff(np.concatenate([[0], cuts, [1 << bits]]))
    return (k / float(1 << bits)).astype(np.float32)


@pytest.mark.parametrize("pos", [0, 1, 2])
def test_enumeration_sweep_matches_oracle_count_for_count(pos):
    """Every grid value of one uniform (2^20 points), as a batch of 2^20
    sequences on the GPU; the histogram of (n, token) equals the oracle's."""
    rng = np.random.default_rng(500 + pos)
    V, K, bits = 8, 2, 20
    P = np.stack([_dyadic(rng, V) for _ in range(K + 1)])
    Q = np.stack([_dyadic(rng, V) for _ in range(K)])
    draft1 = np.array([int(np.argmax(Q[0] - P[0])), int(np.argmax(P[1]))], np.int32)
    ufix = np.array([0.3, 0.6, 0.5], np.float32)
    if pos > 0:
        ufix[0] = 0.0  # accept the first draft so later positions are reached
    B = 1 << bits
    p = np.broadcast_to(P, (B, K + 1, V))
    q = np.broadcast_to(Q, (B, K, V))
    draft = np.broadcast_to(draft1, (B, K))
    u = np.broadcast_to(ufix, (B, K + 1)).copy()
    u[:, pos] = (np.arange(B, dtype=np.float64) * 2.0 ** -bits).astype(np.float32)
    n, tok, bits_dev, ws = _gpu_accept(p, q, draft, u)
    hist = np.zeros((K + 1) * V + 1, np.uint64)
    ok = n >= 0
    np.add.at(hist, n[ok] * V + tok[ok, :][np.arange(ok.sum()), n[ok]], 1)
    hist[-1] = (~ok).sum()
    ref = oracle.enum_sweep(P, Q, draft1, ufix, pos, grid_bits=bits)
    assert np.array_equal(hist, ref)
