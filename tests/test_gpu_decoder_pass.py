"""GPU: one layer of the decoder pass (stack.decoder_pass) against the same
layer composed from oracle pieces in fp64 (RMSNorm, the variant's linears
over the oracle-dequantised weights, RoPE, cache, grouped-query attention,
residual adds), for the INT4 draft (T = 1) and the FP16 verify (T = 5)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_21704_gb300 import stack as stk
from paper_2609_21704_gb300.shapes import QWEN25_1P5B

from gpu_util import assert_close, bits16, dev

pytestmark = pytest.mark.gpu


def _w64(proj, variant):
    w16 = bits16(proj.w16)
    if variant == "fp16":
        return w16.view(np.float16).astype(np.float64)
    c, s = oracle.quantize_int4(w16)
    return oracle.dequant_int4(c, s, proj.k_in)


def _r16(a):  # round to fp16 like the GPU's intermediate buffers
    return a.astype(np.float16).astype(np.float64)


@pytest.mark.parametrize("variant,T", [("int4", 1), ("fp16", 5)])
def test_one_layer_matches_oracle_composition(variant, T):
    sh = QWEN25_1P5B
    S = stk.LinearStack(sh, dev(), seed=8, variants=("int4",), layers=1, with_lm_head=False)
    B, ctx, max_ctx = 1, 70, 128
    st = stk.DecoderState(S, B, T, max_ctx, ctx, seed=9)
    rng = np.random.default_rng(10)
    for c in (st.k[0], st.v[0]):
        pre = rng.normal(0, 1, (B, sh.kv_heads, ctx, 128)).astype(np.float16)
        c[:, :, :ctx] = torch.from_numpy(pre).to(dev())
    x0 = st.x.float().cpu().numpy().astype(np.float64)
    k_pre = st.k[0][0, :, :ctx].float().cpu().numpy().astype(np.float64)
    v_pre = st.v[0][0, :, :ctx].float().cpu().numpy().astype(np.float64)
    g1 = st.gamma[0].float().cpu().numpy().astype(np.float64)
    g2 = st.gamma[1].float().cpu().numpy().astype(np.float64)
    stk.decoder_pass(S, variant, st)
    torch.cuda.synchronize()

    qkv_p, o_p, gu_p, down_p = S.layers[0]
    Hq, Hkv, D, I = sh.q_heads, sh.kv_heads, 128, sh.intermediate
    pos = np.arange(ctx, ctx + T)
    h = _r16(oracle.rmsnorm(x0, g1, stk.RMS_EPS))
    qkv = _r16(oracle.linear(h, _w64(qkv_p, variant)))
    q = oracle.rope(qkv[:, :Hq * D], pos, Hq, D, stk.ROPE_THETA).reshape(T, Hq, D)
    k_new = _r16(oracle.rope(qkv[:, Hq * D:(Hq + Hkv) * D], pos, Hkv, D, stk.ROPE_THETA))
    v_new = qkv[:, (Hq + Hkv) * D:]
    k_all = np.concatenate([k_pre.transpose(1, 0, 2), k_new.reshape(T, Hkv, D)])
    v_all = np.concatenate([v_pre.transpose(1, 0, 2), v_new.reshape(T, Hkv, D)])
    attn = _r16(oracle.attention(q, k_all, v_all, pos).reshape(T, Hq * D))
    x1 = _r16(x0 + oracle.linear(attn, _w64(o_p, variant)))
    h2 = _r16(oracle.rmsnorm(x1, g2, stk.RMS_EPS))
    full = oracle.linear(h2, _w64(gu_p, variant))
    gact = _r16(oracle.silu_gate(full[:, :I], full[:, I:]))
    x2 = x1 + oracle.linear(gact, _w64(down_p, variant))
    assert_close(st.x.float().cpu().numpy().astype(np.float64), x2, f"{variant} layer output")


@pytest.mark.parametrize("variant,T,last_only", [("int4", 1, False), ("int4", 2, True), ("fp16", 5, False),
                                                 ("fp8", 3, True)])
def test_fused_pass_equals_unfused(variant, T, last_only):
    # sq_linear_norm and sq_attention_append are bit-identical to the calls
    # they replace, so two layers plus the lm_head must agree exactly
    sh = QWEN25_1P5B
    S = stk.LinearStack(sh, dev(), seed=3, variants=("int4", "fp8"), layers=2)
    B, max_ctx = 2, 256
    rng = np.random.default_rng(12)
    states = [stk.DecoderState(S, B, T, max_ctx, 0, seed=4) for _ in range(2)]
    pre = [rng.normal(0, 1, (B, sh.kv_heads, 100, 128)).astype(np.float16) for _ in range(4)]
    for st in states:
        st.pos0.copy_(torch.tensor([100, 37], dtype=torch.int32))
        for li in range(2):
            st.k[li][:, :, :100] = torch.from_numpy(pre[2 * li]).to(dev())
            st.v[li][:, :, :100] = torch.from_numpy(pre[2 * li + 1]).to(dev())
    rows = B if last_only else B * T
    out = [torch.empty(rows, sh.vocab, dtype=torch.float16, device=dev()) for _ in range(2)]
    stk.decoder_pass(S, variant, states[0], logits=out[0], last_only=last_only, fuse_norm=True,
                     fuse_append=True)
    stk.decoder_pass(S, variant, states[1], logits=out[1], last_only=last_only, fused=False)
    torch.cuda.synchronize()
    a, b = states
    assert torch.equal(out[0].view(torch.int16), out[1].view(torch.int16))
    assert torch.equal(a.x.view(torch.int16), b.x.view(torch.int16))
    for li in range(2):
        assert torch.equal(a.k[li].view(torch.int16), b.k[li].view(torch.int16))
        assert torch.equal(a.v[li].view(torch.int16), b.v[li].view(torch.int16))
