"""GPU parity: the shared-memory ring engine (one activation row, Sec.
III-D.2 draft pass at batch 1, and direct decoding with the parent) against
the fp64 oracle over the same dequantised weights.

The cases are shapes sq_linear_path sends to the ring (engine 3), at one
activation row and at two to eight (INT4 and FP8): ragged
last tiles, row splits over several warps (few tiles) and whole-row jobs
(many tiles), partial last stages, the epilogues (bias, SiLU gate,
residual), calls chained on one stream that read the previous call's output
(the next call fills its ring while the previous one runs), repeats that
must be bit-identical (also under graph replay), and the full-size
14B-shaped matrices on sampled output columns.  Bar: relative L2 <= 1e-3
and max-abs <= 2e-2 per output."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_21704_gb300 as sq
from paper_2609_21704_gb300 import synth
from paper_2609_21704_gb300.shapes import QWEN25_14B

from gpu_util import assert_close, bits16, dev, dev_to_f64, f16_to_dev

pytestmark = pytest.mark.gpu

WK = {"int4": sq.SQ_W_INT4, "fp8": sq.SQ_W_FP8, "fp16": sq.SQ_W_FP16}
SILU, NONE, RES = sq.SQ_EPI_SILU_GATE, sq.SQ_EPI_NONE, sq.SQ_EPI_RESIDUAL


def _codes(kind, w16_dev, rows, K):
    """Device codes / scales of a device fp16 weight (sq_quantize)."""
    if kind == "fp16":
        return w16_dev, None
    qk = sq.SQ_INT4_G128 if kind == "int4" else sq.SQ_FP8_E4M3_ROW
    cb, _ = sq.sq_quantized_bytes(qk, rows, K)
    codes = torch.empty(rows, cb // rows, dtype=torch.uint8, device=dev())
    if kind == "int4":
        scales = torch.empty(rows, K // 128, dtype=torch.float16, device=dev())
    else:
        scales = torch.empty(rows, dtype=torch.float32, device=dev())
    sq.sq_quantize(w16_dev, qk, codes, scales)
    return codes, scales


def _deq_rows(kind, w16_dev, idx, K):
    """fp64 dequantised weight rows idx, by the oracle from the fp16 parent."""
    w = bits16(w16_dev[torch.from_numpy(np.asarray(idx)).to(dev())])
    if kind == "int4":
        c, s = oracle.quantize_int4(w)
        return oracle.dequant_int4(c, s, K)
    if kind == "fp8":
        c, s = oracle.quantize_fp8(w)
        return oracle.dequant_fp8(c, s)
    return w.view(np.float16).astype(np.float64)


class _Op:
    """One linear call on the ring engine and its oracle on sampled columns."""

    def __init__(self, kind, seed, N, K, x, epi=NONE, bias=False, residual=None):
        rows = 2 * N if epi == SILU else N
        M = x.shape[0]
        assert sq.sq_linear_path(WK[kind], M, N, K, epi) == 3, (kind, M, N, K, epi)
        self.w16 = synth.weights_fp16_device(seed, rows, K, dev())
        self.wd, self.sd = _codes(kind, self.w16, rows, K)
        self.kind, self.N, self.K, self.epi, self.x = kind, N, K, epi, x
        self.bias = f16_to_dev(synth.weights_fp16(seed + 1, 1, rows, std=0.5)[0]) if bias else None
        self.residual = residual
        self.res64 = dev_to_f64(residual) if residual is not None else None
        self.y = torch.full((M, N), 9.0, dtype=torch.float16, device=dev())

    def run(self, stream=None):
        sq.sq_linear_ex(WK[self.kind], self.x, self.wd, self.sd, self.bias, self.residual, self.epi, self.y,
                        stream)

    def tup(self):
        return (WK[self.kind], self.x, self.wd, self.sd, self.bias, self.residual, self.epi, self.y)

    def check(self, what, ncols=512, seed=0):
        N = self.N
        cols = np.arange(N) if N <= ncols else np.sort(np.random.default_rng(seed).choice(N, ncols, replace=False))
        if N - 1 not in cols:
            cols = np.append(cols, N - 1)  # the ragged tail
        idx = np.concatenate([cols, cols + N]) if self.epi == SILU else cols
        full = oracle.linear(dev_to_f64(self.x), _deq_rows(self.kind, self.w16, idx, self.K))
        if self.bias is not None:
            full = full + dev_to_f64(self.bias)[idx][None, :]
        if self.epi == SILU:
            full = oracle.silu_gate(full[:, : len(cols)], full[:, len(cols):])
        if self.epi == RES:
            full = full + self.res64[:, cols]
        assert_close(dev_to_f64(self.y)[:, cols], full, what)


CASES = [
    # kind, N, K, epi: FP16 lm_head-like rows (N >= 65536), ragged tails, K
    # from one unit to many, row splits
    ("fp16", 65536 + 33, 128, NONE), ("fp16", 65536 + 7, 896, RES), ("fp16", 70001, 1536, NONE),
    # FP16 fused gate/up of >= 16 Mi weights
    ("fp16", 9400 + 5, 896, SILU), ("fp16", 2048, 4096 + 128, SILU),
    # INT4 fused gate/up of >= 64 Mi weights (even group count)
    ("int4", 13824 + 9, 2560, SILU), ("int4", 2048 + 16, 16384, SILU),
    # FP8 lm_head-like (>= 400 Mi weights)
    ("fp8", 110003, 4096, NONE), ("fp8", 51203, 8192 + 128, RES),
]


# two to eight activation rows (INT4 and FP8 drafts at batch > 1): every
# row count's column layout, ragged tiles, the K split, the epilogues
CASES_M = [
    ("int4", 2, 7168 + 5, 5120, NONE), ("int4", 3, 1000, 2048, RES), ("int4", 4, 13824, 5120, SILU),
    ("int4", 5, 5120, 5120, NONE), ("int4", 8, 4133, 1536, SILU), ("int4", 8, 152064, 5120, NONE),
    ("int4", 4, 5120, 13824, RES), ("fp8", 8, 7168, 5120, NONE), ("fp8", 5, 300, 1024, SILU),
    ("fp8", 4, 37, 13824, RES),
    # INT4 warp counts when the staged rows leave less room: 12 warps at two
    # rows of K = 27648, 8 warps at eight rows of K = 8192
    ("int4", 2, 3000, 27648, SILU), ("int4", 8, 1000 + 3, 8192, RES),
]


@pytest.mark.parametrize("kind,M,N,K,epi", CASES_M)
def test_ring_rows_match_oracle(kind, M, N, K, epi):
    x = f16_to_dev(synth.activations_fp16(N % 1000 + K + M, M, K))
    res = f16_to_dev(synth.activations_fp16(N % 777 + M, M, N)) if epi == RES else None
    op = _Op(kind, N * 7 + K + M, N, K, x, epi=epi, bias=(N % 2 == 1), residual=res)
    op.run()
    assert sq.sq_check() == 0
    op.check(f"{kind} M={M} N={N} K={K} epi={epi}", ncols=768, seed=M)
    first = op.y.clone()
    op.run()
    assert torch.equal(first, op.y), "repeat not bit-identical"


@pytest.mark.parametrize("kind,N,K,epi", CASES)
def test_ring_matches_oracle(kind, N, K, epi):
    x = f16_to_dev(synth.activations_fp16(N % 1000 + K, 1, K))
    res = f16_to_dev(synth.activations_fp16(N % 777, 1, N)) if epi == RES else None
    op = _Op(kind, N * 7 + K, N, K, x, epi=epi, bias=(N % 2 == 1), residual=res)
    op.run()
    assert sq.sq_check() == 0
    op.check(f"{kind} N={N} K={K} epi={epi}")
    first = op.y.clone()
    op.run()
    assert torch.equal(first, op.y), "repeat not bit-identical"


def test_ring_chain_reads_previous_output():
    """FP16 calls back to back on one stream, each reading the one before:
    the next call's weight copies start while the previous call runs, its
    activations only after it completed.  Repeats are bit-identical, in a
    graph as well."""
    x = f16_to_dev(synth.activations_fp16(5, 1, 896))
    a = _Op("fp16", 11, 9472, 896, x, epi=SILU)
    b = _Op("fp16", 13, 1024, 9472, a.y, epi=SILU, bias=True)
    c = _Op("fp16", 15, 65536 + 100, 1024, b.y)
    ops = [a, b, c]
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        for o in ops:
            o.run(s)
    s.synchronize()
    assert sq.sq_check() == 0
    for i, o in enumerate(ops):
        o.check(f"op {i}")
    first = [o.y.clone() for o in ops]
    with torch.cuda.stream(s):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            sq.sq_linear_chain([o.tup() for o in ops], s)
        for _ in range(3):
            for o in ops:
                o.y.fill_(5.0)
            g.replay()
    s.synchronize()
    for f, o in zip(first, ops):
        assert torch.equal(f, o.y)


@pytest.mark.parametrize("kind,name", [("int4", "gate_up"), ("fp16", "gate_up"), ("fp16", "lm_head"),
                                       ("fp8", "lm_head")])
def test_ring_full_size_14b_sampled(kind, name):
    """The 14B-shaped matrices the ring takes, at full size: sampled output
    columns against the oracle."""
    sh = QWEN25_14B
    K = sh.hidden
    N, epi = (sh.intermediate, SILU) if name == "gate_up" else (sh.vocab, NONE)
    x = synth.activations_fp16_device(72, 1, K, dev())
    op = _Op(kind, 71, N, K, x, epi=epi)
    op.run()
    assert sq.sq_check() == 0
    op.check(f"14B {kind} {name}", ncols=384, seed=3)
