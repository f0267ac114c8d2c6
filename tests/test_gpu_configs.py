"""GPU parity at the five workload shapes, one test per workload.

Every projection of one decoder layer plus lm_head runs at its full size
through the same C calls the step uses, with the variants derived on the
GPU by sq_quantize; 48 output columns per projection (first, last and 46
seeded others) are recomputed by the fp64 oracle from the same fp16 parent
rows, quantised by the oracle itself.  Each workload's accept setting runs
at full vocabulary and is compared bit for bit.

  0.5B MLP : INT4 draft M=1, FP16 verify M=5, accept V=32000 (independent draft)
  1.5B     : INT4 and FP8 draft M=1, FP16 verify M=5, accept V=151936
  7B       : INT4 draft M=1, FP16 verify M=3/5/9 (K=2/4/8), accept K=2/4/8
  7B b8    : FP8 draft M=8, FP16 verify M=48 (tensor cores), accept B=8, K=5
  14B      : INT4/FP8/FP16 resident; draft M=1 and 16, verify M=5 and 144
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_21704_gb300 as sq
from paper_2609_21704_gb300 import synth
from paper_2609_21704_gb300.shapes import QWEN25_0P5B_MLP, QWEN25_14B, QWEN25_1P5B, QWEN25_7B

from gpu_util import assert_close, bits16, dev, dev_to_f64

pytestmark = pytest.mark.gpu

WK = {"int4": sq.SQ_W_INT4, "fp8": sq.SQ_W_FP8, "fp16": sq.SQ_W_FP16}


class Layer:
    """One projection, fp16 parent on the device plus derived variants."""

    def __init__(self, name, n, k, seed, variants):
        self.name, self.n, self.k = name, n, k
        self.epi = sq.SQ_EPI_SILU_GATE if name == "gate_up" else sq.SQ_EPI_NONE
        self.w16 = synth.weights_fp16_device(seed, n, k, dev())
        self.q = {}
        for v in variants:
            kind = sq.SQ_INT4_G128 if v == "int4" else sq.SQ_FP8_E4M3_ROW
            cb, sbytes = sq.sq_quantized_bytes(kind, n, k)
            codes = torch.empty(n, cb // n, dtype=torch.uint8, device=dev())
            scales = (torch.empty(n, k // 128, dtype=torch.float16, device=dev()) if v == "int4"
                      else torch.empty(n, dtype=torch.float32, device=dev()))
            sq.sq_quantize(self.w16, kind, codes, scales)
            self.q[v] = (codes, scales)

    def run(self, variant, M, seed):
        x = synth.activations_fp16_device(seed, M, self.k, dev())
        out_cols = self.n // 2 if self.epi == sq.SQ_EPI_SILU_GATE else self.n
        y = torch.empty(M, out_cols, dtype=torch.float16, device=dev())
        w, s = (self.w16, None) if variant == "fp16" else self.q[variant]
        sq.sq_linear_ex(WK[variant], x, w, s, None, None, self.epi, y)
        return x, y

    def check(self, variant, M, seed):
        x, y = self.run(variant, M, seed)
        assert sq.sq_check() == 0
        out_cols = y.shape[1]
        cols = np.unique(np.concatenate([[0, out_cols - 1],
                                         np.random.default_rng(seed).integers(0, out_cols, 46)]))
        rows = cols if self.epi != sq.SQ_EPI_SILU_GATE else np.concatenate([cols, cols + out_cols])
        w_rows = bits16(self.w16[torch.from_numpy(rows).to(dev())]).view(np.float16)
        if variant == "int4":
            c, s = oracle.quantize_int4(w_rows.view(np.uint16))
            w64 = oracle.dequant_int4(c, s, self.k)
        elif variant == "fp8":
            c, s = oracle.quantize_fp8(w_rows.view(np.uint16))
            w64 = oracle.dequant_fp8(c, s)
        else:
            w64 = w_rows.astype(np.float64)
        ref = oracle.linear(bits16(x).view(np.float16).astype(np.float64), w64)
        if self.epi == sq.SQ_EPI_SILU_GATE:
            ref = oracle.silu_gate(ref[:, : len(cols)], ref[:, len(cols):])
        assert_close(dev_to_f64(y)[:, cols], ref, f"{self.name} {variant} M={M}")


def _layers(shape, variants, with_lm=True, seed=0):
    projs = shape.projections() + ([shape.lm_head()] if with_lm else [])
    return [Layer(n, N, K, seed + i, variants) for i, (n, N, K) in enumerate(projs)]


def _accept(B, K, V, noise, seed):
    p, q, d, u = synth.spec_block(seed, B, K, V, draft_noise=noise)
    ws = torch.zeros(sq.sq_accept_workspace_bytes(B, K, V), dtype=torch.uint8, device=dev())
    n = torch.empty(B, dtype=torch.int32, device=dev())
    tok = torch.empty(B, K + 1, dtype=torch.int32, device=dev())
    sq.sq_accept(*(torch.from_numpy(a).to(dev()) for a in (p, q, d, u)), sq.SQ_ACCEPT_SAMPLE, n, tok, ws)
    assert sq.sq_check() == 0
    _, on, otok = oracle.accept(p, q, d, u, oracle.ACCEPT_SAMPLE)
    assert np.array_equal(n.cpu().numpy(), on) and np.array_equal(tok.cpu().numpy(), otok)


def test_workload_0p5b_mlp():
    layers = _layers(QWEN25_0P5B_MLP, ("int4",), with_lm=False)
    for lyr in layers:
        if lyr.name in ("gate_up", "down"):  # the MLP block
            for step in range(4):
                lyr.check("int4", 1, 100 + step)
            lyr.check("fp16", 5, 110)
    _accept(1, 4, 32000, None, 120)


def test_workload_1p5b():
    for lyr in _layers(QWEN25_1P5B, ("int4", "fp8"), seed=10):
        lyr.check("int4", 1, 200)
        lyr.check("fp8", 1, 201)
        lyr.check("fp16", 5, 202)
    _accept(1, 4, 151936, 0.5, 203)


def test_workload_7b():
    for lyr in _layers(QWEN25_7B, ("int4",), seed=20):
        lyr.check("int4", 1, 300)
        for K in (2, 4, 8):
            lyr.check("fp16", K + 1, 301 + K)
    for K in (2, 4, 8):
        _accept(1, K, 152064, 0.5, 310 + K)


def test_workload_7b_batch8():
    for lyr in _layers(QWEN25_7B, ("fp8",), seed=30):
        lyr.check("fp8", 8, 400)
        lyr.check("fp16", 48, 401)
    _accept(8, 5, 152064, 0.5, 402)


def test_workload_14b():
    for lyr in _layers(QWEN25_14B, ("int4", "fp8"), seed=40):
        lyr.check("int4", 1, 500)
        lyr.check("int4", 16, 501)
        lyr.check("fp8", 16, 502)
        lyr.check("fp16", 5, 503)
        lyr.check("fp16", 144, 504)
    _accept(16, 8, 152064, 0.5, 505)
