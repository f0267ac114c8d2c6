"""GPU parity of the decoder pieces around the linear stack (RMSNorm, RoPE +
KV-cache append, grouped-query decode attention, cache rollback) against
the fp64 oracle: relative L2 <= 1e-3 and max-abs <= 2e-2 for the fp16
outputs, exact for positions and lengths.  Contexts cross 64-key chunk
boundaries; query groups cover the 1.5B (12/2 heads) and 7B (28/4) layouts
at the draft (T = 1) and verify (T = K + 1) sizes."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_21704_gb300 as sq

from gpu_util import assert_close, dev

pytestmark = pytest.mark.gpu
D = 128
THETA = 1e6


def _t(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev())


def test_rmsnorm_matches_oracle():
    rng = np.random.default_rng(0)
    x = rng.normal(0, 3, (5, 1536)).astype(np.float16)
    g = rng.normal(1, 0.1, 1536).astype(np.float16)
    y = torch.empty(5, 1536, dtype=torch.float16, device=dev())
    sq.sq_rmsnorm(_t(x), _t(g), 1e-6, y)
    assert sq.sq_check() == 0
    ref = oracle.rmsnorm(x.astype(np.float64), g.astype(np.float64), 1e-6)
    assert_close(y.float().cpu().numpy().astype(np.float64), ref, "rmsnorm")


def _fill_prefix(rng, B, Hkv, max_ctx, pos0):
    kc = np.zeros((B, Hkv, max_ctx, D), np.float16)
    vc = np.zeros((B, Hkv, max_ctx, D), np.float16)
    for b in range(B):
        kc[b, :, : pos0[b]] = rng.normal(0, 1, (Hkv, pos0[b], D)).astype(np.float16)
        vc[b, :, : pos0[b]] = rng.normal(0, 1, (Hkv, pos0[b], D)).astype(np.float16)
    return kc, vc


@pytest.mark.parametrize("B,T,Hq,Hkv,pos0,max_ctx", [
    (2, 5, 12, 2, [37, 300], 512),
    (1, 1, 12, 2, [1023], 1024),
    (3, 9, 28, 4, [64, 127, 700], 1024),
    (1, 17, 12, 2, [0], 64),            # 102 queries per group
    (1, 1, 12, 2, [3000], 4096),        # 94 chunks merged by the combine
    (2, 3, 12, 2, [5, 0], 128),         # one chunk in use; an empty prefix
    (1, 32, 4, 2, [100], 256),          # T at its limit
])
def test_append_and_attention_match_oracle(B, T, Hq, Hkv, pos0, max_ctx):
    rng = np.random.default_rng(B * 100 + T)
    width = (Hq + 2 * Hkv) * D
    qkv = rng.normal(0, 1, (B * T, width)).astype(np.float16)
    kc, vc = _fill_prefix(rng, B, Hkv, max_ctx, pos0)
    kc_t, vc_t = _t(kc), _t(vc)
    p0 = _t(np.array(pos0, np.int32))
    sq.sq_kv_append(_t(qkv), B, T, Hq, Hkv, p0, THETA, kc_t, vc_t)
    out = torch.empty(B * T, Hq * D, dtype=torch.float16, device=dev())
    ws = torch.empty(sq.sq_attention_workspace_bytes(B, T, Hq, Hkv, max_ctx), dtype=torch.uint8,
                     device=dev())
    sq.sq_attention(_t(qkv), B, T, Hq, Hkv, p0, THETA, kc_t, vc_t, out, ws)
    assert sq.sq_check() == 0
    kc_g, vc_g = kc_t.cpu().numpy(), vc_t.cpu().numpy()
    got = out.float().cpu().numpy().astype(np.float64)
    for b in range(B):
        rows = qkv[b * T:(b + 1) * T].astype(np.float64)
        pos = np.arange(pos0[b], pos0[b] + T)
        k_new = oracle.rope(rows[:, Hq * D:(Hq + Hkv) * D], pos, Hkv, D, THETA).reshape(T, Hkv, D)
        v_new = rows[:, (Hq + Hkv) * D:].reshape(T, Hkv, D)
        # the cache now holds the rotated keys (fp16) and the values (bit copies)
        assert_close(kc_g[b, :, pos0[b]:pos0[b] + T].transpose(1, 0, 2).astype(np.float64), k_new,
                     f"k append b={b}")
        assert np.array_equal(vc_g[b, :, pos0[b]:pos0[b] + T].transpose(1, 0, 2),
                              v_new.astype(np.float16))
        L = pos0[b] + T
        k_all = kc_g[b, :, :L].transpose(1, 0, 2).astype(np.float64)
        v_all = vc_g[b, :, :L].transpose(1, 0, 2).astype(np.float64)
        q = oracle.rope(rows[:, :Hq * D], pos, Hq, D, THETA).reshape(T, Hq, D)
        ref = oracle.attention(q, k_all, v_all, pos).reshape(T, Hq * D)
        assert_close(got[b * T:(b + 1) * T], ref, f"attention b={b}")


def test_rollback_lengths():
    base = _t(np.array([10, 20, 30, 40], np.int32))
    n = _t(np.array([0, 3, -1, 8], np.int32))
    length = torch.empty(4, dtype=torch.int32, device=dev())
    sq.sq_kv_rollback(base, n, 5, length)
    assert sq.sq_check() == 0
    assert length.cpu().tolist() == [11, 24, 30, 45]


def test_append_outside_the_cache_sets_status():
    B, T, Hq, Hkv, max_ctx = 1, 3, 12, 2, 64
    qkv = torch.zeros(B * T, (Hq + 2 * Hkv) * D, dtype=torch.float16, device=dev())
    kc = torch.zeros(B, Hkv, max_ctx, D, dtype=torch.float16, device=dev())
    vc = torch.zeros_like(kc)
    sq.sq_kv_append(qkv, B, T, Hq, Hkv, _t(np.array([62], np.int32)), THETA, kc, vc)
    assert sq.sq_check() & sq.SQ_DEV_BAD_POSITION


def test_embed_gathers_rows_exactly():
    rng = np.random.default_rng(11)
    V, H = 1000, 1536
    table = rng.normal(0, 1, (V, H)).astype(np.float16)
    ids = np.array([0, 999, 17, 17, 500], np.int32)
    out = torch.empty(len(ids), H, dtype=torch.float16, device=dev())
    sq.sq_embed(_t(ids), _t(table), out)
    assert sq.sq_check() == 0
    assert np.array_equal(out.cpu().numpy().view(np.uint16), table[ids].view(np.uint16))
    bad = _t(np.array([5, 1000], np.int32))
    out2 = torch.empty(2, H, dtype=torch.float16, device=dev())
    sq.sq_embed(bad, _t(table), out2)
    assert sq.sq_check() & sq.SQ_DEV_BAD_TOKEN_ID
    assert np.array_equal(out2[0].cpu().numpy().view(np.uint16), table[5].view(np.uint16))
    assert bool((out2[1] == 0).all())


@pytest.mark.parametrize("B,T,Hq,Hkv,pos0,max_ctx", [
    (2, 5, 12, 2, [37, 300], 512),      # new tokens straddle a 32-key chunk boundary in b = 0
    (1, 1, 12, 2, [1023], 1024),        # last position of the cache
    (3, 9, 28, 4, [64, 127, 700], 1024),
    (1, 17, 12, 2, [0], 64),            # empty prefix, two chunks of new tokens
    (4, 2, 40, 8, [30, 31, 32, 33], 96),
])
def test_fused_append_equals_append_then_attention(B, T, Hq, Hkv, pos0, max_ctx):
    rng = np.random.default_rng(B * 1000 + T)
    width = (Hq + 2 * Hkv) * D
    qkv = _t(rng.normal(0, 1, (B * T, width)).astype(np.float16))
    kc, vc = _fill_prefix(rng, B, Hkv, max_ctx, pos0)
    p0 = _t(np.array(pos0, np.int32))
    ws = torch.empty(sq.sq_attention_workspace_bytes(B, T, Hq, Hkv, max_ctx), dtype=torch.uint8,
                     device=dev())
    k1, v1 = _t(kc), _t(vc)
    out1 = torch.empty(B * T, Hq * D, dtype=torch.float16, device=dev())
    sq.sq_kv_append(qkv, B, T, Hq, Hkv, p0, THETA, k1, v1)
    sq.sq_attention(qkv, B, T, Hq, Hkv, p0, THETA, k1, v1, out1, ws)
    k2, v2 = _t(kc), _t(vc)
    out2 = torch.empty(B * T, Hq * D, dtype=torch.float16, device=dev())
    sq.sq_attention_append(qkv, B, T, Hq, Hkv, p0, THETA, k2, v2, out2, ws)
    assert sq.sq_check() == 0
    assert torch.equal(k1.view(torch.int16), k2.view(torch.int16))
    assert torch.equal(v1.view(torch.int16), v2.view(torch.int16))
    assert torch.equal(out1.view(torch.int16), out2.view(torch.int16))


def test_fused_append_outside_the_cache_sets_status_and_writes_nothing():
    B, T, Hq, Hkv, max_ctx = 1, 3, 12, 2, 64
    qkv = torch.ones(B * T, (Hq + 2 * Hkv) * D, dtype=torch.float16, device=dev())
    kc = torch.zeros(B, Hkv, max_ctx, D, dtype=torch.float16, device=dev())
    vc = torch.zeros_like(kc)
    out = torch.empty(B * T, Hq * D, dtype=torch.float16, device=dev())
    ws = torch.empty(sq.sq_attention_workspace_bytes(B, T, Hq, Hkv, max_ctx), dtype=torch.uint8,
                     device=dev())
    sq.sq_attention_append(qkv, B, T, Hq, Hkv, _t(np.array([62], np.int32)), THETA, kc, vc, out, ws)
    assert sq.sq_check() & sq.SQ_DEV_BAD_POSITION
    assert not bool(kc.any()) and not bool(vc.any())
    assert not bool(out.any())
