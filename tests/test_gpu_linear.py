"""GPU parity: the draft and verify linear layers (Sec. III-D.2 / III-D.3)
against the fp64 oracle over the same dequantised weights.

Bar: relative L2 <= 1e-3 and max-abs <= 2e-2 over each output tensor.
Small cases run whole; full-size projections are checked on sampled
output columns that the oracle computes one by one."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_21704_gb300 as sq
from paper_2609_21704_gb300 import synth
from paper_2609_21704_gb300.shapes import QWEN25_1P5B, QWEN25_7B

from gpu_util import assert_close, bits16, dev, dev_to_f64, f16_to_dev

pytestmark = pytest.mark.gpu

KINDS = ("int4", "fp8", "fp16")
WK = {"int4": sq.SQ_W_INT4, "fp8": sq.SQ_W_FP8, "fp16": sq.SQ_W_FP16}


def _variant(kind, w):
    """(device weight, device scales, fp64 dequantised weight) from oracle codes."""
    N, K = w.shape
    if kind == "int4":
        c, s = oracle.quantize_int4(w.view(np.uint16))
        return (torch.from_numpy(c).to(dev()), f16_to_dev(s.view(np.float16)),
                oracle.dequant_int4(c, s, K))
    if kind == "fp8":
        c, s = oracle.quantize_fp8(w.view(np.uint16))
        return torch.from_numpy(c).to(dev()), torch.from_numpy(s).to(dev()), oracle.dequant_fp8(c, s)
    return f16_to_dev(w), None, w.astype(np.float64)


def _run(kind, x, wd, sd, N_out, bias=None, residual=None, epi=sq.SQ_EPI_NONE, y=None):
    M = x.shape[0]
    if y is None:
        y = torch.empty(M, N_out, dtype=torch.float16, device=dev())
    sq.sq_linear_ex(WK[kind], x, wd, sd, bias, residual, epi, y)
    return y


@pytest.mark.parametrize("kind", KINDS)
@pytest.mark.parametrize("M", [1, 2, 3, 5, 8, 9, 16])
@pytest.mark.parametrize("N,K", [(33, 128), (384, 896), (1000, 1536), (96, 4864)])
def test_linear_matches_oracle(kind, M, N, K):
    w = synth.weights_fp16(N * 31 + K, N, K)
    x = synth.activations_fp16(M * 7 + K, M, K)
    wd, sd, w64 = _variant(kind, w)
    y = _run(kind, f16_to_dev(x), wd, sd, N)
    assert_close(dev_to_f64(y), oracle.linear(x.astype(np.float64), w64), f"{kind} M={M} N={N} K={K}")


@pytest.mark.parametrize("kind", KINDS)
def test_named_entry_points_match_generic(kind):
    N, K, M = 200, 896, 5
    w = synth.weights_fp16(1, N, K)
    x = f16_to_dev(synth.activations_fp16(2, M, K))
    wd, sd, _ = _variant(kind, w)
    y1 = torch.empty(M, N, dtype=torch.float16, device=dev())
    if kind == "int4":
        sq.sq_linear_w4a16(x, wd, sd, None, y1)
    elif kind == "fp8":
        sq.sq_linear_fp8(x, wd, sd, None, y1)
    else:
        sq.sq_verify(x, wd, None, y1)
    y2 = _run(kind, x, wd, sd, N)
    assert torch.equal(y1, y2)


@pytest.mark.parametrize("kind", KINDS)
def test_bias_and_residual_in_place(kind):
    N, K, M = 300, 1536, 4
    w = synth.weights_fp16(3, N, K)
    x = synth.activations_fp16(4, M, K)
    b = synth.fp16_normal(5, (N,), 1.0)
    r = synth.fp16_normal(6, (M, N), 1.0)
    wd, sd, w64 = _variant(kind, w)
    y = f16_to_dev(r)  # residual and output share the buffer
    _run(kind, f16_to_dev(x), wd, sd, N, bias=f16_to_dev(b), residual=y, epi=sq.SQ_EPI_RESIDUAL, y=y)
    ref = oracle.linear(x.astype(np.float64), w64, b.astype(np.float64)) + r.astype(np.float64)
    assert_close(dev_to_f64(y), ref, kind)


@pytest.mark.parametrize("kind", KINDS)
@pytest.mark.parametrize("M", [1, 5])
def test_silu_gate_epilogue(kind, M):
    I, K = 640, 896
    w = synth.weights_fp16(7, 2 * I, K)
    x = synth.activations_fp16(8, M, K)
    b = synth.fp16_normal(9, (2 * I,), 0.5)
    wd, sd, w64 = _variant(kind, w)
    y = _run(kind, f16_to_dev(x), wd, sd, I, bias=f16_to_dev(b), epi=sq.SQ_EPI_SILU_GATE)
    full = oracle.linear(x.astype(np.float64), w64, b.astype(np.float64))
    assert_close(dev_to_f64(y), oracle.silu_gate(full[:, :I], full[:, I:]), kind)


@pytest.mark.parametrize("kind", KINDS)
@pytest.mark.parametrize("M", [17, 48])
def test_more_than_sixteen_rows(kind, M):
    N, K = 256, 1536
    w = synth.weights_fp16(10, N, K)
    x = synth.activations_fp16(11, M, K)
    wd, sd, w64 = _variant(kind, w)
    y = _run(kind, f16_to_dev(x), wd, sd, N)
    assert_close(dev_to_f64(y), oracle.linear(x.astype(np.float64), w64), kind)


def test_repeatable_bit_for_bit():
    N, K, M = 4096, 3584, 5
    w = synth.weights_fp16(12, N, K)
    x = f16_to_dev(synth.activations_fp16(13, M, K))
    for kind in KINDS:
        wd, sd, _ = _variant(kind, w)
        assert torch.equal(_run(kind, x, wd, sd, N), _run(kind, x, wd, sd, N))


def test_one_hot_activation_selects_a_column():
    N, K = 512, 1536
    w = synth.weights_fp16(14, N, K)
    x = np.zeros((2, K), np.float16)
    x[0, 5] = 1
    x[1, K - 1] = 1
    for kind in KINDS:
        wd, sd, w64 = _variant(kind, w)
        y = dev_to_f64(_run(kind, f16_to_dev(x), wd, sd, N))
        ref = np.stack([w64[:, 5], w64[:, K - 1]])
        # the column itself, rounded as the kernel rounds: fp32 product
        # (exact for INT4 and FP16), then fp16
        assert np.array_equal(y, ref.astype(np.float32).astype(np.float16).astype(np.float64))


def _sampled_full_size(kind, shape, M, epi=sq.SQ_EPI_NONE, seed=0):
    name, Nw, K = shape
    N_out = Nw // 2 if epi == sq.SQ_EPI_SILU_GATE else Nw
    wt = synth.weights_fp16_device(seed + 1, Nw, K, dev())
    xt = synth.activations_fp16_device(seed + 2, M, K, dev())
    if kind == "fp16":
        wd, sd = wt, None
    else:
        qk = sq.SQ_INT4_G128 if kind == "int4" else sq.SQ_FP8_E4M3_ROW
        cb, sb = sq.sq_quantized_bytes(qk, Nw, K)
        wd = torch.empty(cb, dtype=torch.uint8, device=dev())
        sd = torch.empty(sb // (2 if kind == "int4" else 4),
                         dtype=torch.float16 if kind == "int4" else torch.float32, device=dev())
        sq.sq_quantize(wt, qk, wd, sd)
        wd = wd.view(Nw, -1)
        sd = sd.view(Nw, -1) if kind == "int4" else sd
    y = _run(kind, xt, wd, sd, N_out, epi=epi)
    cols = np.unique(np.concatenate([[0, N_out - 1], np.random.default_rng(Nw).integers(0, N_out, 62)]))
    rows = cols if epi != sq.SQ_EPI_SILU_GATE else np.concatenate([cols, cols + N_out])
    ridx = torch.from_numpy(rows).to(dev())
    w_rows = bits16(wt[ridx]).view(np.float16)
    if kind == "int4":
        c, s = oracle.quantize_int4(w_rows.view(np.uint16))
        w64 = oracle.dequant_int4(c, s, K)
    elif kind == "fp8":
        c, s = oracle.quantize_fp8(w_rows.view(np.uint16))
        w64 = oracle.dequant_fp8(c, s)
    else:
        w64 = w_rows.astype(np.float64)
    x64 = bits16(xt).view(np.float16).astype(np.float64)
    ref = oracle.linear(x64, w64)
    if epi == sq.SQ_EPI_SILU_GATE:
        ref = oracle.silu_gate(ref[:, : len(cols)], ref[:, len(cols):])
    got = dev_to_f64(y)[:, cols]
    assert_close(got, ref, f"{kind} {name} M={M}")


@pytest.mark.parametrize("kind,M", [("int4", 1), ("fp8", 1), ("fp16", 5), ("fp8", 5)])
def test_full_size_lm_head_1p5b(kind, M):
    _sampled_full_size(kind, QWEN25_1P5B.lm_head(), M)


@pytest.mark.parametrize("kind,M", [("int4", 1), ("fp16", 9), ("fp8", 8)])
def test_full_size_down_proj_7b(kind, M):
    _sampled_full_size(kind, QWEN25_7B.projections()[3], M, seed=3)


@pytest.mark.parametrize("kind,M", [("int4", 1), ("fp16", 5)])
def test_full_size_gate_up_silu_7b(kind, M):
    _sampled_full_size(kind, QWEN25_7B.projections()[2], M, epi=sq.SQ_EPI_SILU_GATE, seed=5)


# ---- INT4 single-row calls with many 16-row tiles (the fused gate/up, the
# lm_head) take the tensor cores' register path (mma.sync): every output
# column of whole matrices, ragged tile counts, odd group counts, split K.
@pytest.mark.parametrize("N,K,epi", [
    (8960, 1536, sq.SQ_EPI_SILU_GATE),   # the 1.5B fused gate/up, whole
    (4869, 896, sq.SQ_EPI_NONE),         # ragged last tile, 7 groups split 4 ways
    (5003, 8960, sq.SQ_EPI_RESIDUAL),    # 70 groups, bias and residual
    (40000, 256, sq.SQ_EPI_NONE),        # two groups, no split
])
def test_int4_single_row_tensor_path(N, K, epi):
    Nw = 2 * N if epi == sq.SQ_EPI_SILU_GATE else N
    assert sq.sq_linear_path(sq.SQ_W_INT4, 1, N, K, epi) == 2
    w = synth.weights_fp16(Nw + 3 * K, Nw, K)
    x = synth.activations_fp16(N + 7, 1, K)
    b = synth.fp16_normal(Nw + 1, (Nw,), 1.0)
    wd, sd, w64 = _variant("int4", w)
    ref = oracle.linear(x.astype(np.float64), w64, b.astype(np.float64))
    if epi == sq.SQ_EPI_RESIDUAL:
        r = synth.fp16_normal(K + 1, (1, N), 1.0)
        y = f16_to_dev(r)
        _run("int4", f16_to_dev(x), wd, sd, N, bias=f16_to_dev(b), residual=y, epi=epi, y=y)
        ref = ref + r.astype(np.float64)
    else:
        y = _run("int4", f16_to_dev(x), wd, sd, N, bias=f16_to_dev(b), epi=epi)
        if epi == sq.SQ_EPI_SILU_GATE:
            ref = oracle.silu_gate(ref[:, :N], ref[:, N:])
    assert_close(dev_to_f64(y), ref, f"int4 tensor path N={N} K={K} epi={epi}")
    y2 = _run("int4", f16_to_dev(x), wd, sd, N, bias=f16_to_dev(b), epi=epi) if epi != sq.SQ_EPI_RESIDUAL else None
    if y2 is not None:
        assert torch.equal(y, y2), "not repeatable bit for bit"
    assert sq.sq_check() == 0
