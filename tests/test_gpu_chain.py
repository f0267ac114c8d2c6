"""GPU: sq_linear_chain (Sec. III-D.2/3 passes as one call) gives exactly
the results of the same calls made one by one with sq_linear_ex, on draft
(INT4, FP8) and verify (FP16) passes that mix the CUDA-core and tensor-core
engines; a bad op anywhere in the chain launches nothing.  The fp64 oracle
checks one layer of the chained pass as well."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_21704_gb300 as sq
from paper_2609_21704_gb300 import stack as stk
from paper_2609_21704_gb300.shapes import QWEN25_1P5B, QWEN25_7B

from gpu_util import assert_close, bits16, dev, dev_to_f64

pytestmark = pytest.mark.gpu


def _outputs(b):
    return [b.qkv.clone(), b.o.clone(), b.h.clone(), b.d.clone(), b.logits.clone()]


@pytest.mark.parametrize("shape,variant,M", [
    (QWEN25_1P5B, "int4", 1), (QWEN25_1P5B, "fp8", 1), (QWEN25_1P5B, "fp16", 5),
    (QWEN25_1P5B, "fp16", 9), (QWEN25_7B, "int4", 1), (QWEN25_7B, "fp16", 5)])
def test_chain_equals_separate_calls(shape, variant, M):
    variants = () if variant == "fp16" else (variant,)
    st = stk.LinearStack(shape, dev(), seed=3, variants=variants, layers=2)
    b = stk.PassBuffers(st, M, seed=4)
    stk.run_pass_unchained(st, variant, b)
    torch.cuda.synchronize()
    ref = _outputs(b)
    for t in (b.qkv, b.o, b.h, b.d, b.logits):
        t.fill_(7.0)
    stk.run_pass(st, variant, b)
    assert sq.sq_check() == 0
    for a, r in zip(_outputs(b), ref):
        assert torch.equal(a, r)


def test_chain_layer_matches_oracle():
    st = stk.LinearStack(QWEN25_1P5B, dev(), seed=5, variants=("int4",), layers=1, with_lm_head=False)
    b = stk.PassBuffers(st, 1, seed=6)
    stk.run_pass(st, "int4", b)
    assert sq.sq_check() == 0
    qkv, o, gu, down = st.layers[0]

    def ref(proj, x16):
        c, s = oracle.quantize_int4(bits16(proj.w16))
        w64 = oracle.dequant_int4(c, s, proj.k_in)
        return oracle.linear(bits16(x16).view(np.float16).astype(np.float64), w64)

    assert_close(dev_to_f64(b.qkv), ref(qkv, b.x), "qkv")
    assert_close(dev_to_f64(b.o), ref(o, b.attn), "o (reads qkv's output)")
    full = ref(gu, b.x)
    I = QWEN25_1P5B.intermediate
    assert_close(dev_to_f64(b.h), oracle.silu_gate(full[:, :I], full[:, I:]), "gate_up")
    assert_close(dev_to_f64(b.d), ref(down, b.h), "down (reads gate_up's output)")


def test_chain_bad_op_launches_nothing():
    st = stk.LinearStack(QWEN25_1P5B, dev(), seed=7, variants=("int4",), layers=1)
    b = stk.PassBuffers(st, 1, seed=8)
    ops = stk.pass_ops(st, "int4", b)
    wk, x, w, s, bias, res, epi, y = ops[2]
    ops[2] = (wk, x, w, None, bias, res, epi, y)  # INT4 without scales
    for t in (b.qkv, b.h, b.d, b.logits):
        t.fill_(3.0)
    torch.cuda.synchronize()
    with pytest.raises(sq.SQError, match="op 2"):
        sq.sq_linear_chain(ops)
    torch.cuda.synchronize()
    for t in (b.qkv, b.h, b.d, b.logits):
        assert bool((t == 3.0).all())
    sq.sq_linear_chain([])  # empty chain: nothing to do
